// plan.cuh -- workspace layout and the device-side planner shared by the kernels.
#pragma once

#include "common.cuh"

namespace wisp {

// One unit of attention work: KV tokens [t0, t1) of request r for KV head h, query rows
// [row0, row0 + rows) of the (Hq/Hkv) * (k_r + 1) rows of that head (row = j * (Hq/Hkv) + hh for
// query position j and head hh of the group).  The row set of a (request, head) is cut into
// nrg groups when it is larger than the kernel's row limit.
struct WorkItem {
  int32_t r, h, t0, t1;
  int32_t poff;   // offset (floats) of this item's split partials, -1 if the item covers the whole sequence
  int32_t rows;   // query rows of the item
  int32_t q0;     // first query row of request r
  int32_t ctx;    // c_r
  int32_t row0;   // first query row of the item within its (request, head)
  int32_t rg;     // row group of the item
  int32_t nrg;    // row groups of its (request, head): 1 or 2
};

struct PlanHeader {
  int32_t n_items;
  int32_t chunk_len;
  int32_t partial_floats;
  int32_t next_item;   // work counter of the persistent attention kernel (zeroed by the planner)
  int32_t pad[4];
};

constexpr int kItemsPerSM = 2;     // work items per SM when (request, head) pairs are fewer than SMs
                                   // (measured best of 1, 2, 3 on the long-context workload)
constexpr int kMinChunk = 256;     // never split a sequence below this many tokens
constexpr int kChunkAlign = 128;   // chunk starts are multiples of the KV tile

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
  size_t row_parts = 0;       // RowPart [total_q_rows, slices] statistics of the logit rows
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
};

__global__ void plan_kernel(const PlanParams p);

}  // namespace wisp
