// plan.cuh -- workspace layout and the device-side planner shared by the kernels.
#pragma once

#include "common.cuh"

namespace wisp {

// One unit of attention work: KV tokens [t0, t1) of request r for KV head h, query rows
// [row0, row0 + rows) of the (Hq/Hkv) * (k_r + 1) rows of that head (row = j * (Hq/Hkv) + hh for
// query position j and head hh of the group).  The row set of a (request, head) is cut into
// nrg groups when it is larger than the kernel's row limit.
struct alignas(16) WorkItem {  // 48 bytes: written and read as three 16-byte vectors
  int32_t r, h, t0, t1;
  int32_t poff;   // offset (floats) of this item's split partials, -1 if the item covers the whole sequence
  int32_t rows;   // query rows of the item
  int32_t q0;     // first query row of request r
  int32_t ctx;    // c_r
  int32_t row0;   // first query row of the item within its (request, head)
  int32_t rg;     // row group of the item
  int32_t nrg;    // row groups of its (request, head): 1 or 2
  int32_t pad;
};
static_assert(sizeof(WorkItem) == 48, "work item layout");

struct PlanHeader {
  int32_t n_items;
  int32_t chunk_len;
  int32_t partial_floats;
  int32_t next_item;   // work counter of the persistent attention kernel (zeroed by the planner)
  int32_t attn_ctas;   // CTAs of the tensor-core attention that take items (the others exit at once)
  int32_t pad[3];
};

constexpr int kItemsPerSM = 2;     // work items per SM when (request, head) pairs are fewer than SMs
                                   // (measured best of 1, 2, 3 on the long-context workload)
constexpr int kMinChunk = 256;     // never split a sequence below this many tokens
constexpr int kChunkAlign = 128;   // chunk starts are multiples of the KV tile

constexpr int kTabCacheSlots = 32;  // exp tables of the draw kept in global memory per launch

// Global counters of one acceptance launch (zeroed by the planner).
struct AccCounters {
  int32_t n_items;       // statistics items (slices x rows of valid requests)
  int32_t n_valid;       // requests the planner accepted
  int32_t pad0[30];
  // draw queue: requests pushed, and draw tickets taken (ticket = queue entry * draw slices +
  // slice), each on its own 128-byte line
  int32_t q_reserve;
  int32_t pad1[31];
  int32_t q_head;
  int32_t pad4[31];
  int32_t n_claimed;     // requests whose L is known (queued) or that failed
  int32_t pad2[31];
  int32_t stats_next;    // next statistics item to claim (its own line)
  int32_t pad3[31];
  // the draw's exp tables shared through global memory, one per row maximum m (bf16 bits):
  // state 0 free, 1 being written, 2 ready (tab_m holds its m)
  int32_t tab_state[kTabCacheSlots];
  uint32_t tab_m[kTabCacheSlots];
};

// Byte offsets of every region inside the caller's workspace.
struct Layout {
  size_t status = 0;          // DeviceStatus (256 B)
  size_t q_row_start = 0;     // int32 [B+1]
  size_t draft_start = 0;     // int32 [B+1]
  size_t req_flag = 0;        // int32 [B]
  size_t plan_header = 0;     // PlanHeader
  size_t req_item_begin = 0;  // int32 [B]  first item of request r
  size_t req_chunks = 0;      // int32 [B]  chunks per KV head of request r
  size_t pair_done = 0;       // int32 [B * Hkv * 2] finished chunks per split (request, head, row group)
  size_t items = 0;           // WorkItem [max_items]
  size_t order = 0;           // int32 [max_items]  dispatch order of the items (largest first)
  size_t partials = 0;        // float [partial_cap]
  // acceptance pass (sampling rule)
  size_t acc_ctr = 0;         // AccCounters
  size_t row_order = 0;       // int2 [total_q_rows] (request, row index), level-major
  size_t row_cnt = 0;         // int32 [total_q_rows]
  size_t row_code = 0;        // int32 [total_q_rows]
  size_t row_rec = 0;         // RowRec [total_q_rows]
  size_t sparts = 0;          // SlicePart [total_q_rows, sslices]
  size_t req_state = 0;       // int32 [5, B]: lowest rejecting row, claim, L, finished draw slices, queue
  size_t dparts = 0;          // DrawPart [B, dslices]
  size_t tiles = 0;           // TileRec [B, ntiles]
  size_t tcache = 0;          // uint32 [kTabCacheSlots, 2 * kExpTabEntries]: the draw's exp tables
  // greedy variant
  size_t row_parts = 0;       // argmax partials [total_q_rows, slices]
  size_t total = 0;
  int64_t max_items = 0;
  int64_t partial_cap = 0;    // floats
  int target_items = 0;
};

struct PlanParams {
  int B, Hq, Hkv, D, max_blocks_per_seq, block_size;
  int total_q_rows, total_draft;  // total_draft < 0: not checked (attention-only call)
  int with_attention;          // 0: offsets and validation only
  int target_items;
  int max_rows_item;           // row groups of at most this many rows (rows per head <= 2 * this)
  int64_t max_items, partial_cap;
  const int32_t *draft_lens, *context_lens;
  const int64_t *request_ids;
  DeviceStatus *status;
  int32_t *q_row_start, *draft_start, *req_flag;
  PlanHeader *header;
  int32_t *req_item_begin, *req_chunks, *pair_done;
  WorkItem *items;
  int32_t *order;
  // acceptance pass: level-major dispatch order of the logit rows and the launch's state
  int with_accept;
  int split_sms;               // 1: the acceptance pass runs beside the attention (one step); the
                               // attention may then leave SMs to it from the start
  int accept_apart;            // 1: plan_accept_kernel lays out the acceptance part, not plan_kernel
  int V;                       // vocabulary of the acceptance pass
  int sslices;                 // statistics slices per row
  int2 *row_order;
  int32_t *row_cnt, *row_code;
  int32_t *req_rej, *req_claim, *req_dcnt, *queue;
  AccCounters *acc_ctr;
  int32_t *accepted_len, *next_token;  // -1 for the requests the planner refuses
};

__global__ void plan_kernel(const PlanParams p);
__global__ void plan_accept_kernel(const PlanParams p);

}  // namespace wisp
