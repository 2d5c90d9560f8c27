// accept.cuh -- parameters and workspace records of the acceptance pass (Eq. 1-3).
#pragma once

#include "plan.cuh"

namespace wisp {

constexpr int kAcceptThreads = 256;  // consumer threads of an acceptance CTA (8 warps; plus a producer and a keeper warp)
constexpr int kAcceptCtasPerSM = 2;  // resident CTAs per SM of the persistent acceptance kernel
constexpr int kStatsChunkVecs = 3;   // 16-byte vectors per consumer thread in one chunk of the statistics stream
constexpr int kAmbPerSlice = 8;      // residual elements per draw slice whose sign is left to the finisher
constexpr int kMaxSlices = 32;       // warp slices per row of the greedy variant

// Per-CTA table of exp(u - m) for the bf16 values u with 2^-16 <= |u| < 2^6 (exponent fields
// kExpTabLo .. kExpTabLo + kExpTabBinades - 1, both signs): 64-bit fixed-point values of the draw.
// kExpTabSize values; in the table each sign's kExpTabHalf values are followed by a zero entry,
// which every other bf16 value of that sign reads (kExpTabEntries entries, padded to 4).
constexpr int kExpTabLo = 111;
constexpr int kExpTabBinades = 22;
constexpr int kExpTabHalf = kExpTabBinades * 128;
constexpr int kExpTabSize = 2 * kExpTabHalf;
constexpr int kExpTabEntries = (2 * (kExpTabHalf + 1) + 3) / 4 * 4;
constexpr size_t kExpTabBytes = kExpTabEntries * 2 * sizeof(uint32_t);  // fixed point, two 32-bit words
// Fixed-point scale of the draw's weights: exp(z - m) in [0, 1] is held as round(2^56 exp(z - m)),
// so that a thread sums up to 2^7 of them in 64 bits and every sum is exact and order-free.
constexpr int kFixShift = 56;

// Statistics of one vocabulary slice of one logit row: max, double-float sum of exp(z - m), and
// the terms of the certified error bound: sum exp(z - m) (m - z), the smallest first maximum any
// thread started from, and the most rescales any thread's sum went through.
struct SlicePart {
  float m, s_hi, s_lo, A, mfirst;
  int nres;
  int pad[2];
};
// Merged statistics of a logit row: max, normaliser Z (double-float) and a certified bound dz on
// its relative error, |Z~ - Z| <= dz Z.
struct RowRec {
  float m, z_hi, z_lo, dz;
};
// Row codes (row_code[], written once by the CTA that finishes the row's statistics):
enum : int32_t {
  ROW_UNKNOWN = 0,
  ROW_ACCEPT = 1,     // the decision the row scores (draft token i + 1) accepted
  ROW_REJECT = 2,     // ... rejected: L = i
  ROW_BONUS = 3,      // i == k: the statistics of the bonus row are valid
  ROW_BAD_PROB = 4,   // no softmax, or q(y) negative / NaN at the decision
  ROW_BAD_TOKEN = 5,  // a draft token outside [0, V) (checked for the whole draft at row 0)
};

// A 96-bit unsigned sum (lo 64 bits, hi 32 bits) of fixed-point weights.
struct U96 {
  unsigned long long lo;
  unsigned int hi;
  unsigned int pad;
};

// Residual element whose sign max(0, p - q) could not be settled with the fp32 normaliser.
struct AmbElem {
  unsigned long long e;  // fixed-point exp(z - m)
  float q;
  int v;                 // token id
};

// Totals of one draw slice of row L: sum of exp(z - m) over all elements (fixed point); over the
// elements with p > q (certainly), the sum of exp(z - m) (fixed point) and of q (double-float);
// the undecided elements.
struct DrawPart {
  U96 e_all, e_p;
  float q_hi, q_lo;
  int n_amb;     // > kAmbPerSlice: overflowed (the finisher rescans the slice)
  int pad;
  AmbElem amb[kAmbPerSlice];
};

// Sums of one tile (tile_vecs consecutive vectors of row L) written by the draw: over all elements
// and over the elements with p > q (certainly) of exp(z - m) in units of 2^-56 (96-bit integers:
// low 64 bits, high 32 bits), and of q over the latter (double-float).  The crossing search
// locates the tile from them.
struct TileRec {
  unsigned long long a_lo, p_lo;
  unsigned int a_hi, p_hi;
  float q_hi, q_lo;
};

struct AcceptParams {
  int B, V;
  int vec_z, vec_q;   // 1 if logit rows / draft-prob rows are 16-byte aligned for vector loads
  int sslices;        // statistics slices per row
  int svps;           // 16-byte vectors per statistics slice
  int dslices;        // draw slices per row
  int vpd;            // 16-byte vectors per draw slice (a multiple of 8 tiles: one range of whole tiles per warp)
  int tile_vecs;      // 16-byte vectors per tile of the draw (a multiple of kAcceptThreads)
  int ntiles;         // tiles per row
  int64_t total_rows; // logit rows
  // greedy variant: one warp per (row, slice), argmax partials per (row, slice)
  int slices, vps;
  void *parts;
  // sampling rule
  const int2 *row_order;   // [total_rows] (request, row index) in level-major dispatch order
  int32_t *row_cnt;        // [total_rows] finished statistics slices
  int32_t *row_code;       // [total_rows] ROW_*
  RowRec *row_rec;         // [total_rows]
  SlicePart *sparts;       // [total_rows, slices]
  int32_t *req_rej;        // [B] lowest row index with a rejection so far
  int32_t *req_claim;      // [B] 1 once the request's L is known (or it failed)
  int32_t *req_L;          // [B]
  int32_t *req_dcnt;       // [B] finished draw slices
  int32_t *queue;          // [B] requests ready to draw (-1: not yet written)
  DrawPart *dparts;        // [B, dslices]
  TileRec *tiles;          // [B, ntiles]
  uint32_t *tcache;        // [kTabCacheSlots, 2 * kExpTabEntries] exp tables by row maximum (bf16 logits)
  AccCounters *ctr;
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

cudaError_t accept_setup();  // once per device: kernel attributes, the exp table of the draw
// the acceptance pass (one persistent kernel; needs the planner's offsets and dispatch order)
cudaError_t accept_launch(const AcceptParams &p, bool bf16, int sms, cudaStream_t s, bool pdl);
// greedy (temperature 0) variant: argmax partials of every row, then the walk (two launches)
cudaError_t accept_greedy_launch(const AcceptParams &p, bool bf16, cudaStream_t s);

}  // namespace wisp
