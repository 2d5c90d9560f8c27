// accept.cuh -- parameters of the acceptance kernel.
#pragma once

#include "plan.cuh"

namespace wisp {

constexpr int kAcceptThreads = 256;  // 8 warps per CTA
constexpr int kMaxAcceptCluster = 8;
constexpr int kPreload = 256;        // decision inputs gathered up front for the first rows
// Per-CTA table of exp(u - m) for the bf16 values u with 2^-8 <= |u| < 2^6 (exponent fields
// kExpTabLo .. kExpTabLo + kExpTabBinades - 1, both signs), used by the draw.
constexpr int kExpTabLo = 119;
constexpr int kExpTabBinades = 14;
constexpr int kExpTabSize = 2 * kExpTabBinades * 128;
constexpr int kExpTabMinV = 16384;  // vocabularies smaller than this compute every exp directly

// Statistics of one vocabulary slice of one logit row (written by row_stats_kernel): running max,
// double-float sum of exp(z - m), the error terms of the certified bound, rescale count.
struct RowPart {
  float m, s_hi, s_lo, A, mfirst;
  int nres;
};
constexpr int kMaxSlices = 32;  // slices per row (one warp lane each when they are merged)

struct AcceptParams {
  int B, V;
  int cluster;        // CTAs per request (1..8), = cluster size of the launch
  int vpc;            // 16-byte vectors of a row per CTA (multiple of 32)
  int vec_z, vec_q;   // 1 if logit rows / draft-prob rows are 16-byte aligned for vector loads
  int slices;         // vocabulary slices per row of row_stats_kernel (1..kMaxSlices)
  int vps;            // 16-byte vectors per slice (multiple of 32)
  int64_t total_rows; // logit rows (grid of row_stats_kernel = total_rows * slices)
  RowPart *parts;     // [total_rows, slices]
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
// statistics of every logit row (needs only the logits)
cudaError_t accept_stats_launch(const AcceptParams &p, bool bf16, cudaStream_t s);
// per-request walk and draw (needs the statistics and the planner's offsets)
cudaError_t accept_walk_launch(const AcceptParams &p, bool bf16, cudaStream_t s);
// greedy (temperature 0) variant: argmax partials of every row, then the walk (two launches)
cudaError_t accept_greedy_launch(const AcceptParams &p, bool bf16, cudaStream_t s);

}  // namespace wisp
