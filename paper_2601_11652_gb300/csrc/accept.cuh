// accept.cuh -- parameters of the acceptance kernel.
#pragma once

#include "plan.cuh"

namespace wisp {

struct AcceptParams {
  int B, V;
  int cluster;        // CTAs per request (1..8), = cluster size of the launch
  int vec_z, vec_q;   // 1 if logit rows / draft-prob rows are 16-byte aligned for vector loads
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

// Kernel shapes: SMALL serves rows of at most kSmallTiles 16-byte tiles with one CTA;
// LARGE serves up to 8 CTAs per request with kLargeTilesPerCta tiles each.
constexpr int kSmallTiles = 16;
constexpr int kLargeTilesPerCta = 256;
constexpr int kMaxAcceptCluster = 8;

cudaError_t accept_setup();  // once per device: shared-memory attributes
cudaError_t accept_launch(const AcceptParams &p, bool bf16, bool large, cudaStream_t s);

}  // namespace wisp
