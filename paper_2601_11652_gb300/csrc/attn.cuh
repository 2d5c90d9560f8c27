// attn.cuh -- parameters of the attention kernels.
#pragma once

#include "plan.cuh"

namespace wisp {

struct AttnParams {
  int B, Hq, Hkv, D, max_blocks_per_seq, num_blocks;
  const int64_t *request_ids;
  const int32_t *block_tables;
  const void *q, *k_cache, *v_cache;
  void *out;
  DeviceStatus *status;
  const int32_t *req_flag, *req_item_begin, *req_chunks;
  const PlanHeader *header;
  PlanHeader *header_mut;  // same object: the work counter
  const WorkItem *items;
  const int32_t *order;  // dispatch order of the persistent kernel: item index per counter value
  float *partials;
  int32_t *pair_done;  // [B * Hkv] finished chunks of each split (request, head), zeroed by the planner
};

// Host launchers (defined next to their kernels).
cudaError_t attn_simt_setup();  // once per device: shared-memory attributes
cudaError_t attn_simt_launch(const AttnParams &p, bool bf16, int grid, cudaStream_t s);
cudaError_t attn_combine_launch(const AttnParams &p, bool bf16, cudaStream_t s);
// tcgen05 / TMA kernel for bf16 KV, D in {64, 128}; `grid` persistent CTAs
cudaError_t attn_tc_setup();
// pdl: programmatic dependent launch (the CTAs' set-up overlaps the previous kernel on `s`, which
// the kernel waits for before it reads the plan); off where another stream's kernel should get the
// SMs first
cudaError_t attn_tc_launch(const AttnParams &p, int grid, cudaStream_t s, bool pdl);

}  // namespace wisp
