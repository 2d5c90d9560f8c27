// accept.cuh -- parameters of the acceptance kernel.
#pragma once

#include "plan.cuh"

namespace wisp {

constexpr int kAcceptThreads = 256;  // 8 warps per CTA
constexpr int kMaxAcceptCluster = 8;
constexpr int kPreload = 256;        // decision inputs gathered up front for the first rows

struct AcceptParams {
  int B, V;
  int cluster;        // CTAs per request (1..8), = cluster size of the launch
  int vpc;            // 16-byte vectors of a row per CTA (multiple of 32)
  int vec_z, vec_q;   // 1 if logit rows / draft-prob rows are 16-byte aligned for vector loads
  int prefetch;       // 1: prefetch the next logit row into L2 while deciding the current one
  const int64_t *request_ids;
  const int32_t *draft_lens;
  const void *logits;
  const int32_t *draft_tokens;
  const float *draft_probs;
  const float *accept_u, *sample_u;
  int32_t *accepted_len, *next_token;
  const int32_t *q_row_start, *draft_start, *req_flag;
  DeviceStatus *status;
  Exp2Table tab;
};

cudaError_t accept_setup();  // once per device: shared-memory attributes
// rounds = ceil(vpc / kAcceptThreads): sizes the per-(round, warp) draw partials
cudaError_t accept_launch(const AcceptParams &p, bool bf16, cudaStream_t s);

}  // namespace wisp
