// accept.cu -- the in-order speculative acceptance pass over the vocabulary (Eq. 1-3).
//
// One persistent kernel, accept_kernel, with two kinds of work taken from device-side queues:
//
// Statistics items (row, slice), dispatched level-major (row index 0 of every request, then row
// index 1, ...), so that by the time row i of a request comes up its earlier decisions are usually
// known and rows past a rejection -- which the rule never reads -- are skipped.  A CTA streams its
// slice once as 16-byte vectors; every thread keeps a running max, a double-float sum of
// exp(z - m) (hardware 2^x) and the terms of a certified bound on the relative error of that sum.
// The CTA that finishes the last slice of a row merges the slices and takes the decision the row
// scores (Eq. 1, a = min(1, p(y)/q(y)), accept iff u <= a) in fp32 when u lies outside the
// certified interval of the ratio, else after recomputing the row's normaliser exactly.  It then
// checks whether the request's accepted length L is now known (Eq. 2: the first rejection, or k)
// and, if so, queues the request for its draw.
//
// Draw items (request, slice of row L) for the extra token (Eq. 3): the residual
// max(0, p_L - q_{L+1}) after a rejection, else p_L, by inverse CDF in ascending token order.  The
// weights exp(z - m) are exact 64-bit fixed-point numbers (a per-CTA table over the bf16 values,
// from the double exp), so every sum is exact and independent of its order.  One pass gives, per
// slice and per 64-vector tile, the sum over all elements (the exact normaliser) and, over the
// elements with p > q, the sums of exp(z - m) and of q; the residual mass of a slice is then
// E_P - Z Q_P once Z is known.  Elements whose sign the fp32 normaliser cannot settle are kept
// aside and weighed exactly.  The bookkeeping warp of the CTA that finishes the last slice of a
// request finds the slice and the tile holding the crossing of u * total, rescans that tile with
// exact weights and writes the token.
//
// Nothing waits on an unbounded condition: a CTA that finds no work sleeps briefly and gives up
// after about two seconds (recording WISP_DEV_TIMEOUT); the only other wait is for a queue entry
// whose slot was already reserved by a running CTA.
#include <cfloat>
#include <cmath>
#include <cstring>
#include <type_traits>

#include "accept.cuh"
#include "sm100_ptx.cuh"

namespace wisp {

// exp(u) for the bf16 values u of the draw's table (the host's double exp), written by
// accept_setup as a 64-bit mantissa M in [2^63, 2^64) whose low 8 bits (zero in a double's 53-bit
// significand) hold E + 128: exp(u) = M 2^(E - 63)
__device__ unsigned long long g_exp_m64[kExpTabSize];

namespace {

constexpr int NW = kAcceptThreads / 32;
constexpr int NT = kAcceptThreads;

template <typename LT>
struct LTraits;
template <>
struct LTraits<float> {
  static constexpr int E = 4;  // elements per 16-byte vector
  static constexpr uint32_t NEG_INF2 = 0xff800000u;
};
template <>
struct LTraits<uint16_t> {
  static constexpr int E = 8;
  static constexpr uint32_t NEG_INF2 = 0xff80ff80u;
};

template <typename LT>
__device__ __forceinline__ float vec_elem(const uint4 &w, int i);
template <>
__device__ __forceinline__ float vec_elem<float>(const uint4 &w, int i) {
  const uint32_t u = i == 0 ? w.x : i == 1 ? w.y : i == 2 ? w.z : w.w;
  return __uint_as_float(u);
}
template <>
__device__ __forceinline__ float vec_elem<uint16_t>(const uint4 &w, int i) {
  const uint32_t u = (i >> 1) == 0 ? w.x : (i >> 1) == 1 ? w.y : (i >> 1) == 2 ? w.z : w.w;
  return __uint_as_float((i & 1) ? (u & 0xffff0000u) : (u << 16));
}

__device__ __forceinline__ float load_scalar(const float *row, int64_t v) { return __ldg(row + v); }
__device__ __forceinline__ float load_scalar(const uint16_t *row, int64_t v) {
  return bf16_bits_to_float(__ldg(row + v));
}

// The E elements of vector vi of a row; elements at or past V read as -inf.
template <typename LT>
__device__ __forceinline__ uint4 load_vec(const LT *row, int64_t vi, int V, bool vec_ok) {
  constexpr int E = LTraits<LT>::E;
  const int64_t v0 = vi * E;
  if (vec_ok && v0 + E <= V) return __ldg(reinterpret_cast<const uint4 *>(row + v0));
  uint32_t w[4] = {0, 0, 0, 0};
#pragma unroll
  for (int i = 0; i < E; ++i) {
    const int64_t v = v0 + i;
    const float f = v < V ? load_scalar(row, v) : -INFINITY;
    if (E == 4) {
      w[i] = __float_as_uint(f);
    } else {
      const uint32_t b = __float_as_uint(f) >> 16;  // exact: the value is a bf16
      w[i >> 1] |= (i & 1) ? (b << 16) : b;
    }
  }
  return make_uint4(w[0], w[1], w[2], w[3]);
}

// Draft probabilities of elements v0 .. v0+E-1 (0 past V).
template <int E>
__device__ __forceinline__ void load_q(const float *qrow, int64_t v0, int V, bool vec_ok, float (&q)[E]) {
#pragma unroll
  for (int i = 0; i < E; i += 4) {
    if (vec_ok && v0 + i + 4 <= V) {
      const float4 t = __ldg(reinterpret_cast<const float4 *>(qrow + v0 + i));
      q[i] = t.x;
      q[i + 1] = t.y;
      q[i + 2] = t.z;
      q[i + 3] = t.w;
    } else {
#pragma unroll
      for (int j = 0; j < 4; ++j) q[i + j] = v0 + i + j < V ? __ldg(qrow + v0 + i + j) : 0.0f;
    }
  }
}

// Accesses to the launch's shared state (other CTAs write it; L1 is not coherent).
__device__ __forceinline__ int ld_vol(const int32_t *p) { return *(const volatile int32_t *)p; }
__device__ __forceinline__ void st_vol(int32_t *p, int v) { *(volatile int32_t *)p = v; }
__device__ __forceinline__ void fence_sc() { asm volatile("fence.sc.gpu;" ::: "memory"); }

// ---- the draw's exp table --------------------------------------------------------------------
__device__ __forceinline__ int exp_tab_index(uint32_t bits16) {
  const uint32_t d = ((bits16 >> 7) & 0xFFu) - (uint32_t)kExpTabLo;  // wraps below the range
  if (d >= (uint32_t)kExpTabBinades) return -1;
  return (int)((((bits16 >> 15) * kExpTabBinades + d) << 7) | (bits16 & 0x7Fu));
}
__device__ __forceinline__ uint32_t exp_tab_bits(int idx) {
  const uint32_t sign = (uint32_t)idx / (kExpTabBinades * 128), rem = (uint32_t)idx % (kExpTabBinades * 128);
  return (sign << 15) | (((rem >> 7) + kExpTabLo) << 7) | (rem & 0x7Fu);
}
// Entry of the per-CTA table for the bf16 value with bits b: its own for the table's values, else
// the zero entry after its sign's range; d >= kExpTabHalf tells the second case (-inf, whose weight
// is zero, or a value that needs the direct exp).
__device__ __forceinline__ uint32_t exp_tab_entry(uint32_t b, uint32_t &d) {
  d = (b & 0x7FFFu) - (uint32_t)(kExpTabLo << 7);
  return min(d, (uint32_t)kExpTabHalf) + (b >> 15) * (uint32_t)(kExpTabHalf + 1);
}
// The entry of the value with compact index idx (0 .. kExpTabSize - 1).
__device__ __forceinline__ int exp_tab_entry_of(int idx) { return idx + (idx >= kExpTabHalf ? 1 : 0); }

// round(2^56 x) for |x| <= 1 from the bits of x (integer operations only: 64-bit conversions run
// on the slow FP64 pipe); zero below 2^-126.
__device__ __forceinline__ long long f32_to_fix(float x) {
  const uint32_t b = __float_as_uint(x);
  const int e = (int)((b >> 23) & 0xFFu);
  if (e == 0) return 0;
  const unsigned long long mant = (unsigned long long)((b & 0x7FFFFFu) | 0x800000u);  // x = mant 2^(e - 150)
  const int sh = e - 150 + kFixShift;
  unsigned long long v;
  if (sh >= 0)
    v = mant << sh;
  else if (sh > -40)
    v = (mant + (1ull << (-sh - 1))) >> (-sh);
  else
    v = 0;
  return (b >> 31) ? -(long long)v : (long long)v;
}
// round(2^56 a) for a double-float a in [0, 1] (the two parts converted exactly up to the last
// half unit and added).
__device__ __forceinline__ unsigned long long ff_to_fix(ff a) {
  const long long r = f32_to_fix(a.hi) + f32_to_fix(a.lo);
  return r > 0 ? (unsigned long long)r : 0ull;
}

// A draw weight: round(2^56 exp(z - m)) and exp(z - m) rounded to float.
struct Wt {
  unsigned long long fix;
  float f;
};

// exp(z - m), z <= m, computed directly (double-float, Tang's method).
__device__ __noinline__ Wt exp_fix_direct(float z, float m, const float *th, const float *tl) {
  const ff x = ff_two_sum(z, -m);
  const ff e = ff_exp_nonpos(x.hi, x.lo, th, tl);
  return Wt{ff_to_fix(e), e.hi};
}

// s += q exactly as a double-float without renormalisation (Knuth's TwoSum; the low part collects
// the rounding errors).
__device__ __forceinline__ void ff_acc(ff &s, float q) {
  const float t = __fadd_rn(s.hi, q);
  const float bp = __fsub_rn(t, s.hi);
  const float ap = __fsub_rn(t, bp);
  s.lo = __fadd_rn(s.lo, __fadd_rn(__fsub_rn(s.hi, ap), __fsub_rn(q, bp)));
  s.hi = t;
}

// Two such sums at once in packed fp32x2 form: (hi.x, lo.x) += q.x and (hi.y, lo.y) += q.y, each
// lane rounding exactly as ff_acc (a fused multiply-add by -1 is the rounded difference).
__device__ __forceinline__ void ff_acc2(float2 &hi, float2 &lo, float2 q) {
  const float2 m1 = make_float2(-1.0f, -1.0f);
  const float2 t = __fadd2_rn(hi, q);
  const float2 bp = __ffma2_rn(hi, m1, t);   // t - hi
  const float2 ap = __ffma2_rn(bp, m1, t);   // t - bp
  const float2 e1 = __ffma2_rn(ap, m1, hi);  // hi - ap
  const float2 e2 = __ffma2_rn(bp, m1, q);   // q - bp
  lo = __fadd2_rn(lo, __fadd2_rn(e1, e2));
  hi = t;
}

__device__ __forceinline__ void u96_add(U96 &a, unsigned long long x) {
  const unsigned long long o = a.lo;
  a.lo += x;
  a.hi += (a.lo < o) ? 1u : 0u;
}
__device__ __forceinline__ void u96_add(U96 &a, const U96 &b) {
  u96_add(a, b.lo);
  a.hi += b.hi;
}
__device__ __forceinline__ double u96_to_double(const U96 &a) { return (double)a.hi * 0x1p64 + (double)a.lo; }
__device__ __forceinline__ U96 u96_zero() {
  U96 r;
  r.lo = 0;
  r.hi = 0;
  r.pad = 0;
  return r;
}
__device__ __forceinline__ U96 u96_shfl_xor(const U96 &a, int o) {
  U96 r;
  r.lo = __shfl_xor_sync(0xffffffffu, a.lo, o);
  r.hi = __shfl_xor_sync(0xffffffffu, a.hi, o);
  r.pad = 0;
  return r;
}
__device__ __forceinline__ U96 u96_warp_sum(U96 a) {
  for (int o = 16; o > 0; o >>= 1) u96_add(a, u96_shfl_xor(a, o));
  return a;
}

}  // namespace

namespace {

// ---- row statistics (Eq. 1 needs p = softmax of the row) ----------------------------------------
__device__ __forceinline__ uint32_t bmax2_nan(uint32_t a, uint32_t b) {
  uint32_t r;
  asm("max.NaN.bf16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
  return r;
}
__device__ __forceinline__ float fmax_nan(float a, float b) {
  float r;
  asm("max.NaN.f32 %0, %1, %2;" : "=f"(r) : "f"(a), "f"(b));
  return r;
}

// Per-thread streaming statistics of a row slice: running max m, double-float sum s of
// exp(z - m), A = sum exp(z - m) |z - m| (bounds the effect of rounding z - m and its product with
// log2 e), rescales so far, and the first finite max (bounds the size of all rescale arguments).
struct RowStats {
  float m;
  ff s;
  float A;
  int nres;
  float mfirst;
};

__device__ __forceinline__ void stats_init(RowStats &st) {
  st.m = -INFINITY;
  st.s = {0.0f, 0.0f};
  st.A = 0.0f;
  st.nres = 0;
  st.mfirst = INFINITY;
}

// Move the statistics to a larger reference max mnew (NaN propagates into m).
__device__ __forceinline__ void stats_rebase(RowStats &st, float mnew) {
  if (st.m == -INFINITY) {
    st.m = mnew;
    return;
  }
  if (mnew != mnew) {
    st.m = mnew;
    return;
  }
  if (!(mnew > st.m)) return;
  const float f = ex2_approx((st.m - mnew) * kLog2e);
  const float d = mnew - st.m;
  st.s = ff_mul_f(st.s, f);
  st.A = fmaf(st.A, f, d * st.s.hi);
  st.m = mnew;
  st.nres += 1;
}

// Max of the chunk's elements (NaN if any is NaN): bf16 pairs two at a time, then the two halves.
template <typename LT, int NV>
__device__ __forceinline__ float chunk_max(const uint4 (&w)[NV]) {
  if (std::is_same<LT, uint16_t>::value) {
    uint32_t a = bmax2_nan(w[0].x, w[0].y), b = bmax2_nan(w[0].z, w[0].w);
#pragma unroll
    for (int u = 1; u < NV; ++u) {
      a = bmax2_nan(a, bmax2_nan(w[u].x, w[u].y));
      b = bmax2_nan(b, bmax2_nan(w[u].z, w[u].w));
    }
    a = bmax2_nan(a, b);
    return fmax_nan(__uint_as_float(a << 16), __uint_as_float(a & 0xffff0000u));
  }
  float a = fmax_nan(__uint_as_float(w[0].x), __uint_as_float(w[0].y));
  float b = fmax_nan(__uint_as_float(w[0].z), __uint_as_float(w[0].w));
#pragma unroll
  for (int u = 1; u < NV; ++u) {
    a = fmax_nan(a, fmax_nan(__uint_as_float(w[u].x), __uint_as_float(w[u].y)));
    b = fmax_nan(b, fmax_nan(__uint_as_float(w[u].z), __uint_as_float(w[u].w)));
  }
  return fmax_nan(a, b);
}

// Min of the chunk's elements (NaN ignored: a NaN already makes the max NaN).
template <typename LT, int NV>
__device__ __forceinline__ float chunk_min(const uint4 (&w)[NV]) {
  if (std::is_same<LT, uint16_t>::value) {
    uint32_t a, b;
    asm("min.bf16x2 %0, %1, %2;" : "=r"(a) : "r"(w[0].x), "r"(w[0].y));
    asm("min.bf16x2 %0, %1, %2;" : "=r"(b) : "r"(w[0].z), "r"(w[0].w));
#pragma unroll
    for (int u = 1; u < NV; ++u) {
      uint32_t c, d;
      asm("min.bf16x2 %0, %1, %2;" : "=r"(c) : "r"(w[u].x), "r"(w[u].y));
      asm("min.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(w[u].z), "r"(w[u].w));
      asm("min.bf16x2 %0, %1, %2;" : "=r"(a) : "r"(a), "r"(c));
      asm("min.bf16x2 %0, %1, %2;" : "=r"(b) : "r"(b), "r"(d));
    }
    asm("min.bf16x2 %0, %1, %2;" : "=r"(a) : "r"(a), "r"(b));
    return fminf(__uint_as_float(a << 16), __uint_as_float(a & 0xffff0000u));
  }
  float a = fminf(__uint_as_float(w[0].x), __uint_as_float(w[0].y));
  float b = fminf(__uint_as_float(w[0].z), __uint_as_float(w[0].w));
#pragma unroll
  for (int u = 1; u < NV; ++u) {
    a = fminf(a, fminf(__uint_as_float(w[u].x), __uint_as_float(w[u].y)));
    b = fminf(b, fminf(__uint_as_float(w[u].z), __uint_as_float(w[u].w)));
  }
  return fminf(a, b);
}

// Add one chunk of vectors: its max first (one rescale at most per chunk), then
// exp(z - m) = 2^((z - m) log2 e) per element, a pairwise fp32 sum of the chunk (vector trees, then
// across the vectors) added to the double-float running sum, and the bound term A, here
// (chunk sum) * min(m - chunk min, 104) >= sum exp(z - m) |z - m| (below 104 every term is < 2^-150).
template <typename LT, int NV>
__device__ __forceinline__ void stats_add_chunk(RowStats &st, const uint4 (&w)[NV]) {
  constexpr int E = LTraits<LT>::E;
  const float cm = chunk_max<LT, NV>(w);
  if (cm == -INFINITY) return;  // nothing but padding (or -inf logits)
  if (st.m == -INFINITY) st.mfirst = cm;
  stats_rebase(st, cm);
  const float m = st.m;
  const float span = fminf(m - chunk_min<LT, NV>(w), 104.0f);
  if (std::is_same<LT, uint16_t>::value) {
    // bf16: the element pairs of each 32-bit word in packed fp32x2 arithmetic (z - m and the
    // product with log2 e round exactly as the scalar operations); the pairwise sum adds the pairs
    // of a vector, then the vectors, then the pair's two halves (depth 3 + 2 + 1 for 24 elements)
    const float2 nm = make_float2(-m, -m), l2 = make_float2(kLog2e, kLog2e);
    float2 vp[NV];
#pragma unroll
    for (int u = 0; u < NV; ++u) {
      const uint32_t wd[4] = {w[u].x, w[u].y, w[u].z, w[u].w};
      float2 e[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const float2 z = make_float2(__uint_as_float(wd[i] << 16), __uint_as_float(wd[i] & 0xffff0000u));
        const float2 x = __fmul2_rn(__fadd2_rn(z, nm), l2);
        e[i] = make_float2(ex2_approx(x.x), ex2_approx(x.y));
      }
      vp[u] = __fadd2_rn(__fadd2_rn(e[0], e[1]), __fadd2_rn(e[2], e[3]));
    }
#pragma unroll
    for (int h = 1; h < NV; h <<= 1) {
#pragma unroll
      for (int u = 0; u + h < NV; u += 2 * h) vp[u] = __fadd2_rn(vp[u], vp[u + h]);
    }
    const float cs = vp[0].x + vp[0].y;
    st.s = ff_add_f(st.s, cs);
    st.A = fmaf(cs, span, st.A);
    return;
  }
  float vs[NV];
#pragma unroll
  for (int u = 0; u < NV; ++u) {
    float e[E];
#pragma unroll
    for (int i = 0; i < E; ++i) {
      const float x = vec_elem<LT>(w[u], i) - m;
      e[i] = ex2_approx(x * kLog2e);
    }
#pragma unroll
    for (int h = 1; h < E; h <<= 1) {
#pragma unroll
      for (int i = 0; i < E; i += 2 * h) e[i] += e[i + h];
    }
    vs[u] = e[0];
  }
#pragma unroll
  for (int h = 1; h < NV; h <<= 1) {
#pragma unroll
    for (int u = 0; u + h < NV; u += 2 * h) vs[u] += vs[u + h];
  }
  st.s = ff_add_f(st.s, vs[0]);
  st.A = fmaf(vs[0], span, st.A);
}

// Warp-wide merge of per-lane statistics: max, rebase, tree sum (every lane ends with the result).
__device__ __forceinline__ RowStats warp_merge(RowStats st) {
  float gm = st.m, gf = st.mfirst;
  int gn = st.nres;
  for (int o = 16; o > 0; o >>= 1) {
    gm = fmax_nan(gm, __shfl_xor_sync(0xffffffffu, gm, o));
    gf = fminf(gf, __shfl_xor_sync(0xffffffffu, gf, o));
    gn = max(gn, __shfl_xor_sync(0xffffffffu, gn, o));
  }
  if (st.m > -INFINITY) stats_rebase(st, gm);
  ff gs = st.m > -INFINITY ? st.s : ff{0.0f, 0.0f};
  float ga = st.m > -INFINITY ? st.A : 0.0f;
  for (int o = 16; o > 0; o >>= 1) {
    gs = ff_add(gs, ff_shfl_xor(gs, o));
    ga += __shfl_xor_sync(0xffffffffu, ga, o);
  }
  RowStats r;
  r.m = gm;
  r.s = gs;
  r.A = ga;
  r.nres = gn + 1;  // the lane-to-warp rebase
  r.mfirst = gf;
  return r;
}

// Certified relative error of a row's normaliser Z~ (see RowStats): one 2^x error per element and
// per rescale on its way (thread, warp, CTA, row), three roundings in the argument of every element
// and every rescale, the pairwise fp32 sums; the double-float additions are covered by 1e-12.
__device__ __forceinline__ float z_bound(const RowStats &rs) {
  return 1.05f * ((float)(rs.nres + 2) * kEx2RelErr + 3.0f * 0x1p-24f * (rs.m - rs.mfirst) +
                  3.0f * 0x1p-24f * (rs.A / rs.s.hi) + 7.0f * 0x1p-24f) +
         1e-12f;
}

}  // namespace

namespace {

// ---- the persistent acceptance kernel: roles, items, shared state ----------------------------
// Warps 0..7 consume (compute from shared memory), warp 8 produces (picks the next item and keeps
// bulk copies of its rows in flight in a ring of stages), warp 9 keeps the books (slice records,
// atomics, the row decisions, L, the draw's crossing search).
enum : int { WORK_EXIT = 0, WORK_WAIT = 1, WORK_STATS = 2, WORK_DRAW = 3 };
enum : int { ROW_UNCERTAIN = 100 };  // transient: decided by the exact normaliser

constexpr int kConsumers = kAcceptThreads;    // consumer threads
constexpr int kCW = kConsumers / 32;          // consumer warps
constexpr int kProducerWarp = kCW;
constexpr int kCtaThreads = kConsumers + 64;
constexpr int kStages = 5;
constexpr int kStageBytes = 12288;
constexpr int kStatsChunk = kConsumers * kStatsChunkVecs;  // vectors per statistics chunk (12 KB)
constexpr int kDrawChunk = kConsumers;        // vectors per draw chunk: z 4 KB + q up to 8 KB
constexpr int kDrawTile = kDrawChunk / (kCW / 2);  // vectors per tile: one warp's share of a draw chunk
constexpr int kQOffset = 4096;                // the q part of a draw chunk within its stage
constexpr int kItemSlots = 4;
constexpr long long kWaitCycles = 4000000000LL;  // about two seconds: a wait that long is a failure
constexpr size_t kRingBytes = (size_t)kStages * kStageBytes;
static_assert(kDrawChunk * 16 <= kQOffset && kQOffset + kDrawChunk * 8 * 4 <= kStageBytes, "draw chunk layout");
static_assert(kStatsChunk * 16 <= kStageBytes, "statistics chunk layout");

// One unit of work, written by the producer into an item slot, read by the consumers and the keeper.
struct Item {
  int kind, r, i, s, k, resid;
  int64_t R, Q0, D0;
  int64_t v0, v1;  // vectors [v0, v1) of the row streamed
  int nchunks;
  RowRec rec;
  // results of the consumers
  SlicePart sp;
  U96 ea, ep;
  ff qp;
  int n_amb;
  AmbElem amb[kAmbPerSlice];
};

// The draw's per-CTA exp table (dynamic shared memory): the fixed-point value as two 32-bit words,
// two arrays of 4-byte entries (random 4-byte loads cost far less than random 8-byte ones); hi
// follows lo directly.
struct Tab {
  uint32_t *lo, *hi;
};

struct Sm {
  uint64_t full[kStages], empty[kStages];
  uint64_t iq_full[kItemSlots], iq_empty[kItemSlots], res_ready[kItemSlots];
  uint64_t cons_bar;  // the consumers' barrier (an mbarrier, so that every wait is bounded)
  Item item[kItemSlots];
  float th[256], tl[256];  // 2^(j/256) as double-float pairs (Tang's exp)
  // consumers
  RowStats wst[kCW];
  U96 red[2][2][kCW];  // [buffer][e_all, e_p][warp]
  ff qred[2][kCW];
  unsigned tab_m_bits;
  int tab_valid;
  int tab_mode;
  int amb_n;
  AmbElem amb[kAmbPerSlice];
  int keeper_done;
  int abort_;
};

__device__ __forceinline__ int vload(const int &x) { return *(const volatile int *)&x; }
__device__ __forceinline__ void vstore(int &x, int v) { *(volatile int *)&x = v; }

// Bounded wait for the phase of `bar` with parity `parity`; false after about two seconds or once
// another role gave up (every role then leaves its loop).
__device__ bool wait_bar(uint64_t *bar, uint32_t parity, Sm &sm, const AcceptParams &p) {
  if (ptx::mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  // suspended in the barrier between the checks, so that waiting warps leave the issue slots to
  // the ones that compute
  while (!ptx::mbar_try_wait_sleep(bar, parity, 20000)) {
    if (vload(sm.abort_)) return false;
    if (clock64() - t0 > kWaitCycles) {
      if (atomicExch(&sm.abort_, 1) == 0) report(p.status, WISP_DEV_TIMEOUT, nullptr, -1);
      return false;
    }
  }
  return true;
}

// Barrier of the consumer threads: every consumer arrives, then waits (bounded) for the phase;
// `ph` counts this thread's barriers.
__device__ __forceinline__ void cbar(Sm &sm, uint32_t &ph, const AcceptParams &p) {
  ptx::mbar_arrive(&sm.cons_bar);
  wait_bar(&sm.cons_bar, ph & 1, sm, p);
  ++ph;
}

// The consumers' exp table (Tab) holds round(2^56 exp(u - m)) for the item's row maximum m:
// nothing to do when it already does.  Else from the launch's global copy for this m when one is
// ready (any CTA's draw of a row with the same maximum wrote it), or built here, from
// exp(u) exp(-m) when -m is itself a table value, else directly, both in double-float, and then
// published when the slot for m is free.  Called by every consumer thread.
__device__ void ensure_table(float m, Sm &sm, Tab tab, uint32_t &ph, const AcceptParams &p) {
  constexpr int PER = (kExpTabSize + kConsumers - 1) / kConsumers;
  constexpr int NW4 = (int)(kExpTabBytes / 16);  // 16-byte words of a table
  const unsigned mb = __float_as_uint(m);
  if (sm.tab_valid && sm.tab_m_bits == mb) return;
  const int slot = (int)((mb >> 16) & (kTabCacheSlots - 1));
  uint4 *gt = p.tcache ? reinterpret_cast<uint4 *>(p.tcache + (size_t)slot * 2 * kExpTabEntries) : nullptr;
  if (threadIdx.x == 0) {
    int mode = 0;  // 0 build, 1 build and publish, 2 copy the published table
    if (gt) {
      const int st = ptx::ld_acquire_gpu(&p.ctr->tab_state[slot]);
      if (st == 2 && ld_vol((const int32_t *)&p.ctr->tab_m[slot]) == (int32_t)mb)
        mode = 2;
      else if (st == 0 && atomicCAS(&p.ctr->tab_state[slot], 0, 1) == 0)
        mode = 1;
    }
    sm.tab_mode = mode;
  }
  cbar(sm, ph, p);  // no consumer still reads the previous table; the mode is visible
  const int mode = vload(sm.tab_mode);
  uint4 *st4 = reinterpret_cast<uint4 *>(tab.lo);  // lo and hi are contiguous
  if (mode == 2) {
    uint4 g[(NW4 + kConsumers - 1) / kConsumers];
#pragma unroll
    for (int j = 0; j < (NW4 + kConsumers - 1) / kConsumers; ++j) {
      const int x = threadIdx.x + j * kConsumers;
      if (x < NW4) g[j] = __ldcg(gt + x);
    }
#pragma unroll
    for (int j = 0; j < (NW4 + kConsumers - 1) / kConsumers; ++j) {
      const int x = threadIdx.x + j * kConsumers;
      if (x < NW4) st4[x] = g[j];
    }
  } else {
    const int mi = exp_tab_index((mb >> 16) ^ 0x8000u);  // -m (m is a bf16 value)
    if (mi >= 0) {
      // exp(u - m) = exp(u) exp(-m) = Mu Mm 2^(Eu + Em - 126): the high 64 bits of the 128-bit
      // product times 2^(Eu + Em - 62), rounded to units of 2^-56 (integer operations only)
      const unsigned long long gm = g_exp_m64[mi];
      const unsigned long long Mm = gm & ~0xFFull;
      const int Em = (int)(gm & 0xFFu) - 128;
      constexpr int U = PER;  // entries in flight per thread: every load first
      for (int j0 = 0; j0 < PER; j0 += U) {
        unsigned long long g[U];
#pragma unroll
        for (int j = 0; j < U; ++j) {
          const int idx = threadIdx.x + (j0 + j) * kConsumers;
          g[j] = (j0 + j < PER && idx < kExpTabSize) ? g_exp_m64[idx] : 0ull;
        }
#pragma unroll
        for (int j = 0; j < U; ++j) {
          const int idx = threadIdx.x + (j0 + j) * kConsumers;
          if (j0 + j < PER && idx < kExpTabSize) {
            const int sh = 6 - ((int)(g[j] & 0xFFu) - 128 + Em);  // >= 6 for u <= m
            const unsigned long long hi = __umul64hi(g[j] & ~0xFFull, Mm);
            const bool used = bf16_bits_to_float(exp_tab_bits(idx)) <= m && sh < 64;
            const unsigned long long fx = used ? ((hi >> (sh - 1)) + 1) >> 1 : 0ull;
            tab.lo[exp_tab_entry_of(idx)] = (uint32_t)fx;
            tab.hi[exp_tab_entry_of(idx)] = (uint32_t)(fx >> 32);
          }
        }
      }
    } else {
      for (int idx = threadIdx.x; idx < kExpTabSize; idx += kConsumers) {
        const float u = bf16_bits_to_float(exp_tab_bits(idx));
        const unsigned long long fx = u <= m ? exp_fix_direct(u, m, sm.th, sm.tl).fix : 0ull;
        tab.lo[exp_tab_entry_of(idx)] = (uint32_t)fx;
        tab.hi[exp_tab_entry_of(idx)] = (uint32_t)(fx >> 32);
      }
    }
    for (int x = threadIdx.x; x < kExpTabEntries - kExpTabSize; x += kConsumers) {  // the zero entries
      const int e = x == 0 ? kExpTabHalf : kExpTabSize + x;
      tab.lo[e] = 0u;
      tab.hi[e] = 0u;
    }
    if (mode == 1) {
      cbar(sm, ph, p);  // the whole table is in shared memory
      for (int x = threadIdx.x; x < NW4; x += kConsumers) __stcg(gt + x, st4[x]);
      __threadfence();
    }
  }
  if (threadIdx.x == 0) {
    sm.tab_m_bits = mb;
    sm.tab_valid = 1;
  }
  cbar(sm, ph, p);
  if (mode == 1 && threadIdx.x == 0) {
    // every consumer's part of the copy is fenced and behind the barrier: publish it
    st_vol((int32_t *)&p.ctr->tab_m[slot], (int32_t)mb);
    __threadfence();
    ptx::st_release_gpu(&p.ctr->tab_state[slot], 2);
  }
}

// The E weights of one vector: round(2^56 exp(z - m)).  From the table for bf16 values in its
// range (almost every logit); the others (|z| < 2^-16, |z| >= 64, +-0, a table not given) directly,
// entered once per vector that needs it.
template <typename LT>
__device__ __forceinline__ void weights(const uint4 &w, float m, const Sm &sm, Tab tab,
                                        unsigned long long (&fx)[LTraits<LT>::E]);
__device__ __noinline__ unsigned long long weight_direct1(uint32_t bits, float m, const Sm &sm) {
  return bits == 0xFF80u ? 0ull : exp_fix_direct(__uint_as_float(bits << 16), m, sm.th, sm.tl).fix;
}
template <>
__device__ __forceinline__ void weights<uint16_t>(const uint4 &w, float m, const Sm &sm, Tab tab,
                                                  unsigned long long (&fx)[8]) {
  uint32_t dmax = 0xFFFFFFFFu;
  if (tab.lo) {
    dmax = 0;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const uint32_t u = (i >> 1) == 0 ? w.x : (i >> 1) == 1 ? w.y : (i >> 1) == 2 ? w.z : w.w;
      const uint32_t bits = (i & 1) ? (u >> 16) : (u & 0xFFFFu);
      uint32_t d;
      const uint32_t e = exp_tab_entry(bits, d);
      dmax = max(dmax, d);
      fx[i] = ((unsigned long long)tab.hi[e] << 32) | tab.lo[e];
    }
  }
  if (dmax >= (uint32_t)kExpTabHalf) {
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const uint32_t u = (i >> 1) == 0 ? w.x : (i >> 1) == 1 ? w.y : (i >> 1) == 2 ? w.z : w.w;
      const uint32_t bits = (i & 1) ? (u >> 16) : (u & 0xFFFFu);
      uint32_t d;
      exp_tab_entry(bits, d);
      if (!tab.lo || d >= (uint32_t)kExpTabHalf) fx[i] = weight_direct1(bits, m, sm);
    }
  }
}
template <>
__device__ __forceinline__ void weights<float>(const uint4 &w, float m, const Sm &sm, Tab,
                                               unsigned long long (&fx)[4]) {
  #pragma unroll
  for (int i = 0; i < 4; ++i) fx[i] = exp_fix_direct(vec_elem<float>(w, i), m, sm.th, sm.tl).fix;
}

// A fixed-point weight (units 2^-56, at most 2^56) as a float, within 2^-23 of its value relative:
// the high word converts exactly, the low one with one rounding, and one rounding in the sum.
__device__ __forceinline__ float fix_to_float(unsigned long long x) {
  return __fmaf_rn(__uint2float_rn((uint32_t)(x >> 32)), 0x1p-24f, __uint2float_rn((uint32_t)x) * 0x1p-56f);
}

__device__ __forceinline__ double ff_to_double_(ff a) { return (double)a.hi + (double)a.lo; }

// Draw weight of one element in units of 2^-56, in double: the residual max(0, e - q Z) (Z = Zu in
// the same units) or e itself.  fmax drops a NaN q (no mass), as max(0, p - q) does.
__device__ __forceinline__ double weight_d(unsigned long long e, float q, bool residual, double Zu) {
  return residual ? fmax(0.0, (double)e - (double)q * Zu) : (double)e;
}

// Exact draw weight (units 2^-56, double) of one vector once the normaliser Zu is known: the sign of
// p - q by an fp32 test with a 2^-20 margin, else in double.
template <typename LT>
__device__ __forceinline__ double vec_weight(const uint4 &w, const float *q, bool residual, float m, double Zu,
                                             const Sm &sm, Tab tab) {
  constexpr int E = LTraits<LT>::E;
  unsigned long long fx[E];
  weights<LT>(w, m, sm, tab, fx);
  const float Zf = (float)(Zu * 0x1p-56);
  const float zh = Zf * (1.0f + 0x1p-20f), zl = Zf * (1.0f - 0x1p-20f);
  unsigned long long sp = 0;
  ff sq = {0.0f, 0.0f};
  double ad = 0.0;
#pragma unroll
  for (int i = 0; i < E; ++i) {
    if (!residual) {
      sp += fx[i];
    } else if (q[i] >= 0.0f && fix_to_float(fx[i]) > q[i] * zh) {
      sp += fx[i];
      ff_acc(sq, q[i]);
    } else if (fix_to_float(fx[i]) > q[i] * zl) {
      ad += weight_d(fx[i], q[i], true, Zu);
    }
  }
  return (double)sp - (residual ? Zu * ff_to_double_(sq) : 0.0) + ad;
}

}  // namespace

namespace {

// ---- consumers ----------------------------------------------------------------------------------
// Statistics item: the slice's chunks from the ring (three vectors per thread; a stage is released
// as soon as it is in registers), per-thread streaming statistics, merged into it.sp.
template <typename LT>
__device__ void c_stats(Sm &sm, Item &it, const char *ring, int &c, uint32_t &ph, const AcceptParams &p) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const uint32_t ni = LTraits<LT>::NEG_INF2;
  RowStats st;
  stats_init(st);
  for (int j = 0; j < it.nchunks; ++j) {
    const int stg = c % kStages;
    if (!wait_bar(&sm.full[stg], (c / kStages) & 1, sm, p)) return;
    const uint4 *src = reinterpret_cast<const uint4 *>(ring + (size_t)stg * kStageBytes);
    const int64_t nv = min((int64_t)kStatsChunk, it.v1 - (it.v0 + (int64_t)j * kStatsChunk));
    uint4 w[kStatsChunkVecs];
#pragma unroll
    for (int u = 0; u < kStatsChunkVecs; ++u) {
      const int vi = u * kConsumers + tid;
      w[u] = vi < nv ? src[vi] : make_uint4(ni, ni, ni, ni);
    }
    __syncwarp();
    if (lane == 0) ptx::mbar_arrive(&sm.empty[stg]);
    ++c;
    stats_add_chunk<LT, kStatsChunkVecs>(st, w);
  }
  const RowStats ws = warp_merge(st);
  if (lane == 0) sm.wst[warp] = ws;
  cbar(sm, ph, p);
  if (warp == 0) {
    RowStats q;
    stats_init(q);
    if (lane < kCW) q = sm.wst[lane];
    const RowStats cs = warp_merge(q);
    if (lane == 0) {
      it.sp.m = cs.m;
      it.sp.s_hi = cs.s.hi;
      it.sp.s_lo = cs.s.lo;
      it.sp.A = cs.A;
      it.sp.mfirst = cs.mfirst;
      it.sp.nres = cs.nres;
      it.sp.pad[0] = it.sp.pad[1] = 0;
    }
  }
}

// Warp sum of one value x <= 2^61 per lane as a U96: three 32-bit warp reductions of the 27-bit
// fields of x (each field sum is below 2^32), recombined.
__device__ __forceinline__ U96 warp_sum_u61(unsigned long long x) {
  const unsigned a = __reduce_add_sync(0xffffffffu, (unsigned)(x & 0x7FFFFFFu));
  const unsigned b = __reduce_add_sync(0xffffffffu, (unsigned)((x >> 27) & 0x7FFFFFFu));
  const unsigned c = __reduce_add_sync(0xffffffffu, (unsigned)(x >> 54));  // < 2^13
  U96 r = u96_zero();
  r.lo = (unsigned long long)a + ((unsigned long long)b << 27);  // < 2^60
  r.hi = c >> 10;
  u96_add(r, (unsigned long long)(c & 0x3FFu) << 54);
  return r;
}
// Warp sum of non-negative double-float values (same-sign addition: no cancellation).
__device__ __forceinline__ ff ff_add_pos(ff a, ff b) {
  ff s = ff_two_sum(a.hi, b.hi);
  s.lo = __fadd_rn(s.lo, __fadd_rn(a.lo, b.lo));
  return ff_fast_two_sum(s.hi, s.lo);
}
__device__ __forceinline__ ff ff_warp_sum_pos(ff a) {
  for (int o = 16; o > 0; o >>= 1) a = ff_add_pos(a, ff_shfl_xor(a, o));
  return a;
}

// Draw item: slice of row L in chunks of 256 vectors.  The warps take chunks in two groups (warps
// 0-3 the even chunks of the item, 4-7 the odd ones); in its chunk a warp owns 64 consecutive
// vectors (a tile, two per lane), and the other group only waits for the chunk and releases it.
// Per element the exact weight e = round(2^56 exp(z - m)); after a rejection also the sign of
// p - q, settled with the fp32 normaliser and its certified bound where possible (p > q: e and q go
// into E_P and Q_P; p <= q: no mass), else kept for the finisher.  Sums per tile (written to the
// tile records) and per slice.
template <typename LT>
__device__ void c_draw(Sm &sm, Item &it, Tab tab, const char *ring, int &c, uint32_t &ph, const AcceptParams &p) {
  constexpr int E = LTraits<LT>::E;
  constexpr int TV = kDrawTile;  // vectors per tile
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int grp = warp / (kCW / 2), wi = warp % (kCW / 2);
  const bool residual = it.resid != 0;
  const RowRec rec = it.rec;
  // Z lies in [z_hi (1 - dz), z_hi (1 + dz)]; margins of 2^-20 cover the fp32 roundings of the tests
  const float zhi = rec.z_hi * (1.0f + rec.dz + 0x1p-20f);
  const float zlo = rec.z_hi * (1.0f - rec.dz - 0x1p-20f);
  const float2 zhi2 = make_float2(zhi, zhi), zlo2 = make_float2(zlo, zlo);
  TileRec *trec = p.tiles + (int64_t)it.r * p.ntiles;
  U96 ea = u96_zero(), ep = u96_zero();
  ff qp = {0.0f, 0.0f};
  for (int j = 0; j < it.nchunks; ++j) {
    const int stg = c % kStages;
    if (!wait_bar(&sm.full[stg], (c / kStages) & 1, sm, p)) return;
    const int64_t cv0 = it.v0 + (int64_t)j * kDrawChunk;
    if ((j & 1) != grp) {  // the other group's chunk
      __syncwarp();
      if (lane == 0) ptx::mbar_arrive(&sm.empty[stg]);
      ++c;
      continue;
    }
    const char *sb = ring + (size_t)stg * kStageBytes;
    uint4 w[2];
    float q[2][E];
    bool have[2];
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int loc = wi * TV + h * 32 + lane;  // vector within the chunk
      have[h] = cv0 + loc < it.v1;
      w[h] = have[h] ? reinterpret_cast<const uint4 *>(sb)[loc] : make_uint4(0, 0, 0, 0);
#pragma unroll
      for (int i = 0; i < E; ++i) q[h][i] = 0.0f;
      if (have[h] && residual) {
        const float4 *qs = reinterpret_cast<const float4 *>(sb + kQOffset) + (size_t)loc * (E / 4);
#pragma unroll
        for (int x = 0; x < E / 4; ++x) {
          const float4 t = qs[x];
          q[h][4 * x] = t.x;
          q[h][4 * x + 1] = t.y;
          q[h][4 * x + 2] = t.z;
          q[h][4 * x + 3] = t.w;
        }
      }
    }
    __syncwarp();
    if (lane == 0) ptx::mbar_arrive(&sm.empty[stg]);
    ++c;
    unsigned long long sa = 0, sp = 0;
    // the q sums of the even (x) and odd (y) elements, as double-floats (hi, lo) in packed form
    float2 tqh = make_float2(0.0f, 0.0f), tql = make_float2(0.0f, 0.0f);
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      if (!have[h]) continue;
      unsigned long long fx[E];
      weights<LT>(w[h], rec.m, sm, tab, fx);
      bool amb = false;
#pragma unroll
      for (int i = 0; i < E; i += 2) {
        sa += fx[i];
        sa += fx[i + 1];
        if (residual) {
          // elements i, i + 1 in packed fp32x2 arithmetic (each operation rounds as its scalar
          // form).  p > q for certain (a negative q included: p - q > p; a NaN q never is)
          const float2 qq = make_float2(q[h][i], q[h][i + 1]);
          const float2 hf = make_float2(__uint2float_rn((uint32_t)(fx[i] >> 32)), __uint2float_rn((uint32_t)(fx[i + 1] >> 32)));
          const float2 lf = make_float2(__uint2float_rn((uint32_t)fx[i]), __uint2float_rn((uint32_t)fx[i + 1]));
          const float2 fl = __ffma2_rn(hf, make_float2(0x1p-24f, 0x1p-24f), __fmul2_rn(lf, make_float2(0x1p-56f, 0x1p-56f)));
          const float2 qh = __fmul2_rn(qq, zhi2), ql = __fmul2_rn(qq, zlo2);
          const bool p0 = fl.x > qh.x, p1 = fl.y > qh.y;
          if (p0) sp += fx[i];
          if (p1) sp += fx[i + 1];
          ff_acc2(tqh, tql, make_float2(p0 ? qq.x : 0.0f, p1 ? qq.y : 0.0f));
          // neither certainly positive nor certainly without mass
          amb |= (!p0 && fl.x > ql.x) || (!p1 && fl.y > ql.y);
        }
      }
      if (amb) {
        #pragma unroll
        for (int i = 0; i < E; ++i) {
          const float qi = q[h][i], fl = fix_to_float(fx[i]);
          if (!(fl > qi * zhi) && fl > qi * zlo) {
            const int a = atomicAdd(&sm.amb_n, 1);
            if (a < kAmbPerSlice) {
              sm.amb[a].e = fx[i];
              sm.amb[a].q = qi;
              sm.amb[a].v = (int)((cv0 + wi * TV + h * 32 + lane) * E + i);
            }
          }
        }
      }
    }
    const ff tq = ff_add_pos(ff{tqh.x, tql.x}, ff{tqh.y, tql.y});
    // the warp's tile: its sums, warp-wide, into the tile records
    // per lane at most 16 weights of at most 2^56 each
    const U96 A_ = warp_sum_u61(sa), P_ = residual ? warp_sum_u61(sp) : u96_zero();
    const ff Q_ = residual ? ff_warp_sum_pos(tq) : ff{0.0f, 0.0f};
    if (p.tile_vecs && lane == 0 && cv0 + wi * TV < it.v1) {
      TileRec r;
      r.a_lo = A_.lo;
      r.a_hi = A_.hi;
      r.p_lo = P_.lo;
      r.p_hi = P_.hi;
      r.q_hi = Q_.hi;
      r.q_lo = Q_.lo;
      trec[(cv0 + wi * TV) / TV] = r;
    }
    u96_add(ea, A_);
    u96_add(ep, P_);
    qp = ff_add_pos(qp, Q_);
  }
  // slice totals (each warp holds its own, identical in its lanes)
  if (lane == 0) {
    sm.red[0][0][warp] = ea;
    sm.red[0][1][warp] = ep;
    sm.qred[0][warp] = qp;
  }
  cbar(sm, ph, p);
  if (tid == 0) {
    U96 a = u96_zero(), b = u96_zero();
    ff t = {0.0f, 0.0f};
    for (int x = 0; x < kCW; ++x) {
      u96_add(a, sm.red[0][0][x]);
      u96_add(b, sm.red[0][1][x]);
      t = ff_add_pos(t, sm.qred[0][x]);
    }
    it.ea = a;
    it.ep = b;
    it.qp = t;
    const int na = sm.amb_n;
    it.n_amb = na;
    for (int x = 0; x < na && x < kAmbPerSlice; ++x) it.amb[x] = sm.amb[x];
    __threadfence();  // the tile records before the keeper's completion count
  }
}

// The exp table for row maximum m from the launch's global cache, if a CTA has published it
// (bit-identical to a table built here); else none (the direct exp is then used).
__device__ Tab cached_table(const AcceptParams &p, float m) {
  const unsigned mb = __float_as_uint(m);
  if (!p.tcache) return Tab{nullptr, nullptr};
  const int slot = (int)((mb >> 16) & (kTabCacheSlots - 1));
  if (ptx::ld_acquire_gpu(&p.ctr->tab_state[slot]) != 2 || ld_vol((const int32_t *)&p.ctr->tab_m[slot]) != (int32_t)mb)
    return Tab{nullptr, nullptr};
  uint32_t *t = p.tcache + (size_t)slot * 2 * kExpTabEntries;
  return Tab{t, t + kExpTabEntries};
}

// The extra token (Eq. 3) from vectors [v0, v1) of row L, which hold the crossing of thr (the
// share of u * total left at v0), by the bookkeeping warp right after it has located them: exact
// weights of 32 vectors at a time, a warp scan in token order, then the element of the crossing
// within its vector; with take_last, or when rounding leaves no crossing, the last element with
// weight.  Writes the request's outputs.
template <typename LT>
__device__ void keeper_finish(const AcceptParams &p, const Sm &sm, int r, int i, bool resid, int64_t Q0, int64_t D0,
                              float m, double Zu, int64_t v0, int64_t v1, double thr, bool take_last) {
  constexpr int E = LTraits<LT>::E;
  const int lane = threadIdx.x & 31;
  const LT *row = static_cast<const LT *>(p.logits) + (Q0 + i) * (int64_t)p.V;
  const float *qrow = p.draft_probs + (D0 + i) * (int64_t)p.V;
  const Tab tab = std::is_same<LT, uint16_t>::value ? cached_table(p, m) : Tab{nullptr, nullptr};
  double carry = 0.0;
  int tok = -1;
  int64_t last_vec = -1;  // the last vector with weight so far
  for (int64_t base = v0; base < v1 && tok < 0; base += 32) {
    const int64_t vi = base + lane;
    const bool have = vi < v1;
    uint4 w = make_uint4(0, 0, 0, 0);
    float q[E];
#pragma unroll
    for (int x = 0; x < E; ++x) q[x] = 0.0f;
    if (have) {
      w = load_vec<LT>(row, vi, p.V, p.vec_z != 0);
      if (resid) load_q<E>(qrow, vi * E, p.V, p.vec_q != 0, q);
    }
    const double wv = have ? vec_weight<LT>(w, q, resid, m, Zu, sm, tab) : 0.0;
    double incl = wv;
    for (int o = 1; o < 32; o <<= 1) {
      const double t = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += t;
    }
    incl += carry;
    const unsigned pos = __ballot_sync(0xffffffffu, have && wv > 0.0);
    if (pos) last_vec = base + 31 - __clz(pos);
    const unsigned hit = take_last ? 0u : __ballot_sync(0xffffffffu, have && incl > thr);
    if (hit) {
      const int l0 = __ffs(hit) - 1;
      int t_ = -1;
      if (lane == l0) {
        // this lane's elements in order, with exact weights
        unsigned long long fx[E];
        weights<LT>(w, m, sm, tab, fx);
        double wt[E];
#pragma unroll
        for (int x = 0; x < E; ++x) wt[x] = vi * E + x < p.V ? weight_d(fx[x], q[x], resid, Zu) : 0.0;
        const double r2 = thr - (incl - wv);
        double acc = 0.0;
        int lastv = -1;
#pragma unroll
        for (int x = 0; x < E; ++x) {
          if (t_ < 0) {
            if (wt[x] > 0.0) lastv = (int)(vi * E + x);
            acc += wt[x];
            if (acc > r2) t_ = (int)(vi * E + x);
          }
        }
        if (t_ < 0) t_ = lastv;
      }
      tok = __shfl_sync(0xffffffffu, t_, l0);
      if (tok < 0) tok = -2;  // the crossing vector had no element with weight after all
      break;
    }
    carry = __shfl_sync(0xffffffffu, incl, 31);
  }
  if (tok < 0) {
    // no crossing (take_last, or rounding): the last element with weight
    tok = -1;
    if (last_vec >= 0 && lane == 0) {
      const uint4 w = load_vec<LT>(row, last_vec, p.V, p.vec_z != 0);
      float q[E];
#pragma unroll
      for (int x = 0; x < E; ++x) q[x] = 0.0f;
      if (resid) load_q<E>(qrow, last_vec * E, p.V, p.vec_q != 0, q);
      unsigned long long fx[E];
      weights<LT>(w, m, sm, tab, fx);
#pragma unroll
      for (int x = 0; x < E; ++x) {
        const int64_t v = last_vec * E + x;
        if (v < p.V && weight_d(fx[x], q[x], resid, Zu) > 0.0) tok = (int)v;
      }
    }
  }
  if (lane == 0) {
    p.accepted_len[r] = i;
    p.next_token[r] = tok;
  }
}

}  // namespace

namespace {

// ---- the keeper (warp 9): completions, row decisions, L, the draw's crossing search ------------
struct DecIn {
  float zy, qy, u;
};

// The decision row i scores (Eq. 1 for draft token i + 1), taken by one thread from the row's
// merged statistics: ROW_ACCEPT / ROW_REJECT when u lies outside the certified interval of the
// fp32 ratio p(y) / q(y), ROW_UNCERTAIN otherwise (decided with the exact normaliser).
template <typename LT>
__device__ int decide(const AcceptParams &p, const RowRec &rec, int32_t y, const DecIn &d) {
  if (y < 0 || y >= p.V) return ROW_BAD_TOKEN;
  const float zy = d.zy, qy = d.qy, u = d.u;
  if (!(qy >= 0.0f)) return ROW_BAD_PROB;
  if (qy == 0.0f) return ROW_ACCEPT;                                   // a = 1
  if (!(zy > -INFINITY)) return u <= 0.0f ? ROW_ACCEPT : ROW_REJECT;  // p(y) = 0 exactly
  const float x = zy - rec.m;
  // outside the range of the fp32 ratio (2^x flushes to zero below 2^-126, a subnormal q(y) loses
  // bits): the exact path, in double precision
  if (x * kLog2e < -126.0f || qy < FLT_MIN) return ROW_UNCERTAIN;
  // the decision's own exp (error and argument roundings) and ratio roundings on top of Z's bound
  const float dr = rec.dz + 1.05f * (kEx2RelErr + 3.0f * 0x1p-24f * fabsf(x) + 4.0f * 0x1p-24f);
  const float ratio = ex2_approx(x * kLog2e) / (rec.z_hi * qy);
  const float lo = fminf(1.0f, ratio * (1.0f - dr)), hi = fminf(1.0f, ratio * (1.0f + dr));
  if (u <= lo) return ROW_ACCEPT;
  if (u > hi) return ROW_REJECT;
  return ROW_UNCERTAIN;
}

// Is request r's accepted length now known?  The codes of rows 0..k are read in order (one lane
// each): the first rejection gives L, a valid bonus row L = k, a bad row an error, an unknown row
// means not yet.  The first warp to see the answer claims the request and queues it for its draw
// (or records its error).
__device__ void try_determine(const AcceptParams &p, int r, int k, int64_t Q0) {
  const int lane = threadIdx.x & 31;
  int L = -1, err = 0;
  for (int j0 = 0; j0 <= k; j0 += 32) {
    const int j = j0 + lane;
    const int c = j <= k ? ld_vol(p.row_code + Q0 + j) : ROW_ACCEPT;
    const unsigned nonacc = __ballot_sync(0xffffffffu, c != ROW_ACCEPT);
    if (nonacc == 0) continue;
    const int l0 = __ffs(nonacc) - 1;
    const int c0 = __shfl_sync(0xffffffffu, c, l0);
    if (c0 == ROW_UNKNOWN) return;
    if (c0 == ROW_REJECT)
      L = j0 + l0;
    else if (c0 == ROW_BONUS)
      L = k;
    else
      err = c0 == ROW_BAD_TOKEN ? WISP_DEV_BAD_TOKEN : WISP_DEV_BAD_PROB;
    break;
  }
  if (L < 0 && !err) return;
  if (lane != 0) return;
  if (atomicCAS(p.req_claim + r, 0, 1) != 0) return;
  atomicMin(p.req_rej + r, -1);  // every remaining statistics item of the request is skipped
  if (err) {
    report(p.status, err, p.request_ids, r);
    p.accepted_len[r] = -1;
    p.next_token[r] = -1;
    __threadfence();
    atomicAdd(&p.ctr->n_claimed, 1);
    return;
  }
  st_vol(p.req_L + r, L);
  __threadfence();
  const int pos = atomicAdd(&p.ctr->q_reserve, 1);  // reserve a queue entry
  st_vol(p.queue + pos, r);
  __threadfence();
  atomicAdd(&p.ctr->n_claimed, 1);  // after the queue entry: a CTA that sees every request claimed sees it
}

// Exact draw weight (units 2^-56) of vectors [a, b) of a row, by one warp alone (lanes stride), each
// element's exp computed directly: the rare paths (an uncertain decision's normaliser, a slice
// whose undecided elements overflowed its record).  q = nullptr: the weights exp(z - m) themselves.
template <typename LT>
__device__ double warp_range_weight(const AcceptParams &p, const Sm &sm, const LT *row, const float *qrow, float m,
                                    double Zu, int64_t a, int64_t b) {
  constexpr int E = LTraits<LT>::E;
  const int lane = threadIdx.x & 31;
  double acc = 0.0;
  for (int64_t vi = a + lane; vi < b; vi += 32) {
    const uint4 w = load_vec<LT>(row, vi, p.V, p.vec_z != 0);
    float q[E];
    #pragma unroll
    for (int i = 0; i < E; ++i) q[i] = 0.0f;
    if (qrow) load_q<E>(qrow, vi * E, p.V, p.vec_q != 0, q);
    acc += vec_weight<LT>(w, q, qrow != nullptr, m, Zu, sm, Tab{nullptr, nullptr});
  }
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  return acc;
}

// A statistics item is complete: its slice record, the row's count; the warp that completes the
// row merges its slices, takes the decision, checks the draft (at row 0), publishes the row's code
// and tries to determine L.
template <typename LT>
__device__ void k_stats(const AcceptParams &p, Sm &sm, const Item &it) {
  const int lane = threadIdx.x & 31;
  const int r = it.r, i = it.i, k = it.k;
  const LT *lrow = static_cast<const LT *>(p.logits) + it.R * (int64_t)p.V;
  // the decision's inputs first: the draft token and the uniform, then z(y) and q(y), whose loads
  // overlap the slice bookkeeping and the merge
  const bool dec = i < k;
  const int32_t y = dec ? __ldg(p.draft_tokens + it.D0 + i) : 0;
  DecIn d{0.0f, 0.0f, dec ? __ldg(p.accept_u + it.D0 + i) : 0.0f};
  RowStats q;
  stats_init(q);
  if (p.sslices == 1) {
    // the item is the whole row: its statistics are the row's
    if (lane == 0) {
      q.m = it.sp.m;
      q.s.hi = it.sp.s_hi;
      q.s.lo = it.sp.s_lo;
      q.A = it.sp.A;
      q.mfirst = it.sp.mfirst;
      q.nres = it.sp.nres;
    }
  } else {
    int last = 0;
    if (lane == 0) {
      p.sparts[it.R * p.sslices + it.s] = it.sp;
      __threadfence();
      last = atomicAdd(&p.row_cnt[it.R], 1) == p.sslices - 1;
    }
    if (!__shfl_sync(0xffffffffu, last, 0)) return;
    __threadfence();
    if (lane < p.sslices) {
      const SlicePart *sp = p.sparts + it.R * p.sslices + lane;
      q.m = __ldcg(&sp->m);
      q.s.hi = __ldcg(&sp->s_hi);
      q.s.lo = __ldcg(&sp->s_lo);
      q.A = __ldcg(&sp->A);
      q.mfirst = __ldcg(&sp->mfirst);
      q.nres = __ldcg(&sp->nres);
    }
  }
  if (dec && y >= 0 && y < p.V) {
    d.zy = load_scalar(lrow, y);
    d.qy = __ldg(p.draft_probs + (it.D0 + i) * (int64_t)p.V + y);
  }
  const RowStats rs = warp_merge(q);
  RowRec rec;
  rec.m = rs.m;
  rec.z_hi = rs.s.hi;
  rec.z_lo = rs.s.lo;
  const bool ok = rs.m > -INFINITY && rs.m < INFINITY && rs.s.hi > 0.0f && rs.s.hi < INFINITY && rs.A >= 0.0f;
  rec.dz = ok ? z_bound(rs) : 0.0f;
  int code = 0;
  if (lane == 0) code = !ok ? ROW_BAD_PROB : i == k ? ROW_BONUS : decide<LT>(p, rec, y, d);
  code = __shfl_sync(0xffffffffu, code, 0);
  // the whole draft is validated when row 0 (which the rule always reads) is finished
  if (i == 0 && k > 0) {
    bool bad = false;
    for (int j = lane; j < k; j += 32) {
      const int32_t y = __ldg(p.draft_tokens + it.D0 + j);
      bad |= y < 0 || y >= p.V;
    }
    if (__any_sync(0xffffffffu, bad)) code = ROW_BAD_TOKEN;
  }
  if (code == ROW_UNCERTAIN) {
    const int64_t nvec = (p.V + LTraits<LT>::E - 1) / LTraits<LT>::E;
    const double Zu = warp_range_weight<LT>(p, sm, lrow, nullptr, rec.m, 0.0, 0, nvec);
    // p(y) / q(y) in double precision: z(y) - m is exact, and neither p(y) nor a subnormal q(y)
    // leaves the double range
    const double ratio = exp((double)d.zy - (double)rec.m) * 0x1p56 / (Zu * (double)d.qy);
    code = (double)d.u <= fmin(1.0, ratio) ? ROW_ACCEPT : ROW_REJECT;
  }
  if (lane == 0) {
    p.row_rec[it.R] = rec;
    __threadfence();
    st_vol(p.row_code + it.R, code);
    if (code == ROW_REJECT) atomicMin(p.req_rej + r, i);
  }
  __syncwarp();
  fence_sc();  // this code before the codes read next (against the keeper of another row)
  try_determine(p, r, k, it.Q0);
}

// One of a tile record's integer sums (over the elements with p > q when pos, else all).
__device__ __forceinline__ U96 tile_u96(const TileRec *t, bool pos) {
  U96 r = u96_zero();
  r.lo = __ldcg(pos ? &t->p_lo : &t->a_lo);
  r.hi = __ldcg(pos ? &t->p_hi : &t->a_hi);
  return r;
}


// A draw item is complete: its slice record and the request's count.  The warp that completes the
// request: exact normaliser (the slices' sums of exp(z - m)), residual mass per slice, the slice
// holding the crossing of u * total (Eq. 3), the tile within it (from the tile records), and the
// token within the tile (keeper_finish).
template <typename LT>
__device__ void k_draw(const AcceptParams &p, Sm &sm, const Item &it) {
  constexpr int E = LTraits<LT>::E;
  const int lane = threadIdx.x & 31;
  const int Sd = p.dslices, r = it.r;
  int last = 0;
  if (lane == 0) {
    DrawPart *out = p.dparts + (int64_t)r * Sd + it.s;
    out->e_all = it.ea;
    out->e_p = it.ep;
    out->q_hi = it.qp.hi;
    out->q_lo = it.qp.lo;
    out->n_amb = it.n_amb;
    for (int x = 0; x < it.n_amb && x < kAmbPerSlice; ++x) out->amb[x] = it.amb[x];
    __threadfence();
    last = atomicAdd(p.req_dcnt + r, 1) == Sd - 1;
  }
  if (!__shfl_sync(0xffffffffu, last, 0)) return;
  __threadfence();
  const int64_t nvec = (p.V + E - 1) / E;
  const LT *row = static_cast<const LT *>(p.logits) + (it.Q0 + it.i) * (int64_t)p.V;
  const float *qrow = p.draft_probs + (it.D0 + it.i) * (int64_t)p.V;
  U96 ea = u96_zero(), ep = u96_zero();
  double qp = 0.0;
  int na = 0;
  const DrawPart *dp = p.dparts + (int64_t)r * Sd + lane;
  if (lane < Sd) {
    ea.lo = __ldcg(&dp->e_all.lo);
    ea.hi = __ldcg(&dp->e_all.hi);
    ep.lo = __ldcg(&dp->e_p.lo);
    ep.hi = __ldcg(&dp->e_p.hi);
    qp = (double)__ldcg(&dp->q_hi) + (double)__ldcg(&dp->q_lo);
    na = __ldcg(&dp->n_amb);
  }
  const double Zu = u96_to_double(u96_warp_sum(ea));
  bool resid = it.resid != 0;
  const double se = u96_to_double(ea);
  double sd = se;
  bool over = false;
  if (resid) {
    sd = u96_to_double(ep) - Zu * qp;
    if (na > kAmbPerSlice) {
      over = true;
    } else {
      for (int j = 0; j < na; ++j) sd += weight_d(__ldcg(&dp->amb[j].e), __ldcg(&dp->amb[j].q), true, Zu);
    }
  }
  // slices with more undecided elements than their record holds: their mass by an exact pass
  const unsigned ov = __ballot_sync(0xffffffffu, lane < Sd && over);
  for (unsigned o = ov; o; o &= o - 1) {
    const int d = __ffs(o) - 1;
    const int64_t a = min(nvec, (int64_t)d * p.vpd), b = min(nvec, a + p.vpd);
    const double t = warp_range_weight<LT>(p, sm, row, qrow, it.rec.m, Zu, a, b);
    if (lane == d) sd = t;
  }
  // the slices' masses in slice order: an inclusive warp scan (lane d: slices 0..d), the total from
  // the last lane, so that the crossing search below reads the same prefix sums as the total
  auto slice_scan = [&](double v) {
    double incl = lane < Sd ? v : 0.0;
    for (int o = 1; o < 32; o <<= 1) {
      const double t = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += t;
    }
    return incl;
  };
  double incl = slice_scan(sd);
  double S = __shfl_sync(0xffffffffu, incl, 31);
  if (resid && !(S > 0.0)) {
    // the residual has no mass (only through rounding): draw from p_L instead
    resid = false;
    sd = se;
    incl = slice_scan(sd);
    S = __shfl_sync(0xffffffffu, incl, 31);
  }
  const double thr = (double)__ldg(p.sample_u + r) * S;
  const unsigned hitd = __ballot_sync(0xffffffffu, lane < Sd && incl > thr);
  const unsigned massd = __ballot_sync(0xffffffffu, lane < Sd && sd > 0.0);
  const int owner = hitd ? __ffs(hitd) - 1 : -1;
  const int lastd = massd ? 31 - __clz(massd) : -1;
  // the share of thr left at the owner's first element: thr minus the scan's prefix before it
  const double before = __shfl_sync(0xffffffffu, incl, owner > 0 ? owner - 1 : 0);
  const double thr_d = owner > 0 ? thr - before : owner == 0 ? thr : 0.0;
  double run = 0.0;
  int take_last = owner < 0 ? 1 : 0;  // rounding left no crossing: the last token with mass
  const int d = owner >= 0 ? owner : lastd;
  if (d < 0) {  // no token has mass (cannot happen for a valid row)
    if (lane == 0) {
      p.accepted_len[r] = it.i;
      p.next_token[r] = -1;
    }
    return;
  }
  const int64_t s0 = (int64_t)d * p.vpd, s1 = min(nvec, s0 + p.vpd);
  if (p.tile_vecs == 0) {
    // no tile records (they would not fit): the whole slice is searched
    keeper_finish<LT>(p, sm, r, it.i, resid, it.Q0, it.D0, it.rec.m, Zu, s0, s1, thr_d, take_last != 0);
    return;
  }
  // the tile within slice d
  const int64_t tlo = (int64_t)d * p.vpd / p.tile_vecs;
  const int64_t thi = min((int64_t)p.ntiles, (min(nvec, (int64_t)(d + 1) * p.vpd) + p.tile_vecs - 1) / p.tile_vecs);
  int64_t tile = -1;
  double thr_t = thr_d;
  const bool d_over = (ov >> d) & 1u;
  const int nad = resid && !d_over ? __shfl_sync(0xffffffffu, na, d) : 0;
  const DrawPart *dd = p.dparts + (int64_t)r * Sd + d;
  const TileRec *tr = p.tiles + (int64_t)r * p.ntiles;
  run = 0.0;
  int64_t lastpos = -1;
  for (int64_t t0 = tlo; t0 < thi && tile < 0; t0 += 32) {
    const int64_t t = t0 + lane;
    double w = 0.0;
    if (t < thi) {
      if (d_over) {
        w = 0.0;  // filled below, one tile at a time, by the whole warp
      } else if (resid) {
        w = u96_to_double(tile_u96(tr + t, true)) - Zu * ((double)__ldcg(&tr[t].q_hi) + (double)__ldcg(&tr[t].q_lo));
        for (int j = 0; j < nad; ++j) {
          const int64_t vt = (int64_t)(__ldcg(&dd->amb[j].v) / E) / p.tile_vecs;
          if (vt == t) w += weight_d(__ldcg(&dd->amb[j].e), __ldcg(&dd->amb[j].q), true, Zu);
        }
      } else {
        w = u96_to_double(tile_u96(tr + t, false));
      }
    }
    if (d_over) {
      // the slice's tile sums miss undecided elements: exact tile masses
      for (int x = 0; x < 32 && t0 + x < thi; ++x) {
        const int64_t tt = t0 + x;
        const double m_ = warp_range_weight<LT>(p, sm, row, resid ? qrow : nullptr, it.rec.m, Zu,
                                                tt * p.tile_vecs, min(nvec, (tt + 1) * p.tile_vecs));
        if (lane == x) w = m_;
      }
    }
    double incl = w;
    for (int o = 1; o < 32; o <<= 1) {
      const double u = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += u;
    }
    incl += run;
    const unsigned pos = __ballot_sync(0xffffffffu, t < thi && w > 0.0);
    if (pos) lastpos = t0 + 31 - __clz(pos);
    if (!take_last) {
      const unsigned hit = __ballot_sync(0xffffffffu, t < thi && incl > thr_d);
      if (hit) {
        const int l0 = __ffs(hit) - 1;
        tile = t0 + l0;
        thr_t = thr_d - __shfl_sync(0xffffffffu, incl - w, l0);
      }
    }
    run = __shfl_sync(0xffffffffu, incl, 31);
  }
  if (tile < 0) {
    tile = lastpos;
    take_last = 1;
  }
  if (tile < 0) {
    if (lane == 0) {
      p.accepted_len[r] = it.i;
      p.next_token[r] = -1;
    }
    return;
  }
  const int64_t t0v = tile * p.tile_vecs;
  keeper_finish<LT>(p, sm, r, it.i, resid, it.Q0, it.D0, it.rec.m, Zu, t0v, min(nvec, t0v + p.tile_vecs), thr_t,
                    take_last != 0);
}

template <typename LT>
__device__ void keeper(const AcceptParams &p, Sm &sm) {
  const int lane = threadIdx.x & 31;
  for (int n = 0;; ++n) {
    const int slot = n % kItemSlots;
    if (!wait_bar(&sm.res_ready[slot], (n / kItemSlots) & 1, sm, p)) return;
    const Item &it = sm.item[slot];
    const int kind = it.kind;
    if (kind == WORK_EXIT) return;
    if (kind == WORK_STATS) k_stats<LT>(p, sm, it);
    if (kind == WORK_DRAW) k_draw<LT>(p, sm, it);
    __syncwarp();
    if (lane == 0) {
      __threadfence_block();
      vstore(sm.keeper_done, n + 1);
      ptx::mbar_arrive(&sm.iq_empty[slot]);
    }
    __syncwarp();
  }
}

}  // namespace

namespace {


// ---- the producer (warp 8): next item, bulk copies into the ring ---------------------------------
// Lane 0: the next work item of this CTA: the next statistics item in the level-major order
// (skipping rows past a known rejection and rows of decided requests), else a draw ticket.
// WORK_EXIT once every valid request is decided, every draw ticket taken and this CTA's keeper is
// done with everything issued; WORK_WAIT otherwise.
template <typename LT>
__device__ int pick(const AcceptParams &p, Sm &sm, Item &d, long long &idle_since, int issued, int &pend) {
  constexpr int E = LTraits<LT>::E;
  const int64_t nvec = (p.V + E - 1) / E;
  AccCounters *c = p.ctr;
  const int Sd = p.dslices;
  if (vload(sm.abort_)) return WORK_EXIT;
  // statistics first: every row's decision as early as possible (a draw can wait; the requests
  // decided last bound the pass)
  const int n_items = __ldcg(&c->n_items);
  while (ld_vol(&c->stats_next) < n_items) {
    const int t = atomicAdd(&c->stats_next, 1);
    if (t >= n_items) break;
    const int2 ent = __ldcg(p.row_order + t / p.sslices);
    const int r = ent.x, i = ent.y;
    if (i > ld_vol(p.req_rej + r)) continue;  // past a rejection, or the request is decided
    d.kind = WORK_STATS;
    d.r = r;
    d.i = i;
    d.s = t % p.sslices;
    d.k = __ldg(p.draft_lens + r);
    d.Q0 = __ldg(p.q_row_start + r);
    d.D0 = __ldg(p.draft_start + r);
    d.R = d.Q0 + i;
    d.resid = 0;
    d.v0 = min(nvec, (int64_t)d.s * p.svps);
    d.v1 = min(nvec, d.v0 + p.svps);
    d.nchunks = (int)((d.v1 - d.v0 + kStatsChunk - 1) / kStatsChunk);
    idle_since = -1;
    return WORK_STATS;
  }
  // draw tickets: one atomic increment of the head takes the next ticket.  A ticket taken past the
  // entries reserved so far (a race with other producers) stays pending while this CTA goes on with
  // statistics items; it is used once its entry exists, or lapses once every request is decided.
  if (pend < 0 && ld_vol(&c->q_head) < ld_vol(&c->q_reserve) * Sd) pend = atomicAdd(&c->q_head, 1);
  int r = -1;
  if (pend >= 0 && pend < ld_vol(&c->q_reserve) * Sd) {
    const long long t0 = clock64();
    r = ld_vol(p.queue + pend / Sd);
    while (r < 0) {  // the entry's keeper writes it right after reserving it
      if (clock64() - t0 > kWaitCycles) {
        if (atomicExch(&sm.abort_, 1) == 0) report(p.status, WISP_DEV_TIMEOUT, nullptr, -1);
        return WORK_EXIT;
      }
      __nanosleep(64);
      r = ld_vol(p.queue + pend / Sd);
    }
  }
  if (r >= 0) {
    const unsigned head = (unsigned)pend;
    pend = -1;
    __threadfence();
    d.kind = WORK_DRAW;
    d.r = r;
    d.s = (int)(head % Sd);
    d.i = ld_vol(p.req_L + r);
    d.k = __ldg(p.draft_lens + r);
    d.Q0 = __ldg(p.q_row_start + r);
    d.D0 = __ldg(p.draft_start + r);
    d.R = d.Q0 + d.i;
    d.resid = d.i < d.k;
    const RowRec *rr = p.row_rec + d.R;
    d.rec.m = __ldcg(&rr->m);
    d.rec.z_hi = __ldcg(&rr->z_hi);
    d.rec.z_lo = __ldcg(&rr->z_lo);
    d.rec.dz = __ldcg(&rr->dz);
    d.v0 = min(nvec, (int64_t)d.s * p.vpd);
    d.v1 = min(nvec, d.v0 + p.vpd);
    d.nchunks = (int)((d.v1 - d.v0 + kDrawChunk - 1) / kDrawChunk);
    idle_since = -1;
    return WORK_DRAW;
  }
  if (ld_vol(&c->n_claimed) >= __ldcg(&c->n_valid)) {
    fence_sc();
    const int res = ld_vol(&c->q_reserve) * Sd;
    if (pend >= res) pend = -1;  // no entry will ever hold this ticket
    if (pend < 0 && vload(sm.keeper_done) == issued && ld_vol(&c->q_head) >= res) return WORK_EXIT;
  }
  const long long now = clock64();
  if (idle_since < 0) idle_since = now;
  if (now - idle_since > kWaitCycles) {
    if (atomicExch(&sm.abort_, 1) == 0) report(p.status, WISP_DEV_TIMEOUT, nullptr, -1);
    return WORK_EXIT;
  }
  return WORK_WAIT;
}

// Copy chunk j of item `it` into a stage: bulk copies when the rows are 16-byte aligned (z at the
// stage start, q at kQOffset), else the warp's own loads (padding with -inf / 0 past V).
template <typename LT>
__device__ void issue_chunk(const AcceptParams &p, const Item &it, int j, char *stage, uint64_t *full) {
  constexpr int E = LTraits<LT>::E;
  const int lane = threadIdx.x & 31;
  const bool stats = it.kind == WORK_STATS;
  const int64_t CH = stats ? kStatsChunk : kDrawChunk;
  const int64_t cv0 = it.v0 + (int64_t)j * CH;
  const int nv = (int)min(CH, it.v1 - cv0);
  const bool resid = !stats && it.resid;
  const LT *row = static_cast<const LT *>(p.logits) + it.R * (int64_t)p.V;
  const float *qrow = p.draft_probs + (it.D0 + it.i) * (int64_t)p.V;
  if (p.vec_z && (!resid || p.vec_q)) {
    if (lane == 0) {
      const uint32_t zb = (uint32_t)nv * 16u, qb = resid ? (uint32_t)nv * E * 4u : 0u;
      ptx::mbar_arrive_expect_tx(full, zb + qb);
      ptx::bulk_load(ptx::smem_u32(stage), row + cv0 * E, zb, full);
      if (resid) ptx::bulk_load(ptx::smem_u32(stage + kQOffset), qrow + cv0 * E, qb, full);
    }
    return;
  }
  uint4 *dz = reinterpret_cast<uint4 *>(stage);
  float *dq = reinterpret_cast<float *>(stage + kQOffset);
  for (int v = lane; v < nv; v += 32) {
    dz[v] = load_vec<LT>(row, cv0 + v, p.V, false);
    if (resid) {
      float q[E];
      load_q<E>(qrow, (cv0 + v) * E, p.V, false, q);
      #pragma unroll
      for (int i = 0; i < E; ++i) dq[(size_t)v * E + i] = q[i];
    }
  }
  __syncwarp();
  if (lane == 0) ptx::mbar_arrive(full);
}

template <typename LT>
__device__ void producer(const AcceptParams &p, Sm &sm, char *ring) {
  const int lane = threadIdx.x & 31;
  long long idle_since = -1;
  int pend = -1;  // lane 0: a draw ticket taken but not yet usable
  int n = 0, c = 0;
  bool ok = true;
  for (;;) {
    Item d;
    int kind = WORK_WAIT;
    if (lane == 0) kind = pick<LT>(p, sm, d, idle_since, n, pend);
    kind = __shfl_sync(0xffffffffu, kind, 0);
    if (kind == WORK_WAIT) {
      __nanosleep(256);
      continue;
    }
    const int slot = n % kItemSlots;
    if (!wait_bar(&sm.iq_empty[slot], ((n / kItemSlots) & 1) ^ 1, sm, p)) {
      ok = false;
      break;
    }
    if (lane == 0) {
      d.kind = kind;
      sm.item[slot] = d;
      ptx::mbar_arrive(&sm.iq_full[slot]);
    }
    __syncwarp();
    if (kind == WORK_EXIT) break;
    const Item &it = sm.item[slot];
    for (int j = 0; j < it.nchunks && ok; ++j) {
      const int stg = c % kStages;
      if (!wait_bar(&sm.empty[stg], ((c / kStages) & 1) ^ 1, sm, p)) {
        ok = false;
        break;
      }
      issue_chunk<LT>(p, it, j, ring + (size_t)stg * kStageBytes, &sm.full[stg]);
      ++c;
    }
    if (!ok) break;
    ++n;
  }
  if (!ok) {
    // given up: let the copies still in flight land before the CTA can exit (bounded)
    for (int x = c - kStages < 0 ? 0 : c - kStages; x < c; ++x) wait_bar(&sm.full[x % kStages], (x / kStages) & 1, sm, p);
  }
}

// ---- the consumers (warps 0..7) -------------------------------------------------------------------
template <typename LT>
__device__ void consumers(const AcceptParams &p, Sm &sm, const char *ring, Tab tab) {
  const bool bf = std::is_same<LT, uint16_t>::value;
  uint32_t ph = 0;
  int c = 0;
  for (int n = 0;; ++n) {
    const int slot = n % kItemSlots;
    if (!wait_bar(&sm.iq_full[slot], (n / kItemSlots) & 1, sm, p)) return;
    Item &it = sm.item[slot];
    const int kind = it.kind;
    if (kind != WORK_EXIT && kind != WORK_STATS) {
      if (threadIdx.x == 0) sm.amb_n = 0;
      if (bf) ensure_table(it.rec.m, sm, tab, ph, p);
      cbar(sm, ph, p);
    }
    if (kind == WORK_STATS) c_stats<LT>(sm, it, ring, c, ph, p);
    if (kind == WORK_DRAW) c_draw<LT>(sm, it, bf ? tab : Tab{nullptr, nullptr}, ring, c, ph, p);
    cbar(sm, ph, p);  // every consumer is done with the item
    if (threadIdx.x == 0) ptx::mbar_arrive(&sm.res_ready[slot]);
    if (kind == WORK_EXIT || vload(sm.abort_)) return;
  }
}

}  // namespace

// The acceptance pass (see the file comment): persistent CTAs of consumer, producer and keeper warps.
template <typename LT>
__global__ void __launch_bounds__(kCtaThreads, kAcceptCtasPerSM) accept_kernel(const __grid_constant__ AcceptParams p) {
  extern __shared__ __align__(128) unsigned char s_dyn[];
  __shared__ Sm sm;
  char *ring = reinterpret_cast<char *>(s_dyn);
  const Tab tab{reinterpret_cast<uint32_t *>(s_dyn + kRingBytes),
                reinterpret_cast<uint32_t *>(s_dyn + kRingBytes + kExpTabEntries * sizeof(uint32_t))};
  // launched as a programmatic dependent of the planner: read nothing before it has completed
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int tid = threadIdx.x, warp = tid >> 5;
  for (int j = tid; j < 256; j += kCtaThreads) {
    sm.th[j] = p.tab.hi[j];
    sm.tl[j] = p.tab.lo[j];
  }
  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) {
      ptx::mbar_init(&sm.full[s], 1);
      ptx::mbar_init(&sm.empty[s], kCW);
    }
    for (int s = 0; s < kItemSlots; ++s) {
      ptx::mbar_init(&sm.iq_full[s], 1);
      ptx::mbar_init(&sm.iq_empty[s], 1);
      ptx::mbar_init(&sm.res_ready[s], 1);
    }
    ptx::mbar_init(&sm.cons_bar, kConsumers);
    ptx::fence_mbar_init();
    sm.tab_valid = 0;
    sm.keeper_done = 0;
    sm.abort_ = 0;
  }
  __syncthreads();  // the only CTA-wide barrier: set-up
  if (warp < kCW)
    consumers<LT>(p, sm, ring, tab);
  else if (warp == kProducerWarp)
    producer<LT>(p, sm, ring);
  else
    keeper<LT>(p, sm);
}

// ---- greedy (temperature 0) acceptance -----------------------------------------------------
// Sampling at temperature 0 takes the most likely token, so the rule of Eq. 1-3 becomes: accept
// y_i iff y_i is the argmax of logit row i-1 (the lowest token id among equal maxima), stop at the
// first mismatch, and emit the argmax of row L.  row_argmax_kernel: one warp per (row, slice), every
// row in parallel; greedy_walk_kernel: one warp per request merges the slices of its rows in order.
struct RowArg {
  float m;  // max of the slice (-inf if none)
  int idx;  // lowest token id attaining it
};

template <typename LT>
__global__ void __launch_bounds__(NT) row_argmax_kernel(const __grid_constant__ AcceptParams p) {
  constexpr int E = LTraits<LT>::E;
  const int lane = threadIdx.x & 31;
  const int64_t unit = (int64_t)blockIdx.x * NW + (threadIdx.x >> 5);
  if (unit >= p.total_rows * p.slices) return;
  const int64_t row = unit / p.slices;
  const int sl = (int)(unit % p.slices);
  const int V = p.V;
  const LT *rowp = static_cast<const LT *>(p.logits) + row * (int64_t)V;
  const int64_t nvec = (V + E - 1) / E;
  const int64_t vlo = min(nvec, (int64_t)sl * p.vps);
  const int64_t vhi = min(nvec, vlo + p.vps);
  float m = -INFINITY;
  int idx = INT32_MAX;
  // a lane visits its elements in increasing token order, so a strict ">" keeps the first maximum
  // (the loads of 4 vectors in flight together)
  for (int64_t v0 = vlo + lane; v0 < vhi; v0 += 4 * 32) {
    uint4 w[4];
#pragma unroll
    for (int u = 0; u < 4; ++u)
      if (v0 + u * 32 < vhi) w[u] = load_vec<LT>(rowp, v0 + u * 32, V, p.vec_z != 0);
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int64_t vi = v0 + u * 32;
      if (vi >= vhi) break;
#pragma unroll
      for (int i = 0; i < E; ++i) {
        const float z = vec_elem<LT>(w[u], i);
        if (z > m) {
          m = z;
          idx = (int)(vi * E + i);
        }
      }
    }
  }
  for (int o = 16; o > 0; o >>= 1) {
    const float om = __shfl_xor_sync(0xffffffffu, m, o);
    const int oi = __shfl_xor_sync(0xffffffffu, idx, o);
    if (om > m || (om == m && oi < idx)) {
      m = om;
      idx = oi;
    }
  }
  if (lane == 0) reinterpret_cast<RowArg *>(p.parts)[unit] = RowArg{m, idx};
}

template <typename LT>
__global__ void __launch_bounds__(NT) greedy_walk_kernel(const __grid_constant__ AcceptParams p) {
  const int lane = threadIdx.x & 31;
  const int r = blockIdx.x * NW + (threadIdx.x >> 5);
  if (r >= p.B || p.req_flag[r] != REQ_OK) return;
  const int V = p.V, k = p.draft_lens[r], S = p.slices;
  const int64_t Q0 = p.q_row_start[r], D0 = p.draft_start[r];
  const RowArg *parts = reinterpret_cast<const RowArg *>(p.parts);
  int L = k, tok = -1, err = 0;
  for (int i = 0; i <= k; ++i) {
    RowArg a{-INFINITY, INT32_MAX};
    if (lane < S) a = parts[(Q0 + i) * S + lane];
    for (int o = 16; o > 0; o >>= 1) {
      const float om = __shfl_xor_sync(0xffffffffu, a.m, o);
      const int oi = __shfl_xor_sync(0xffffffffu, a.idx, o);
      if (om > a.m || (om == a.m && oi < a.idx)) {
        a.m = om;
        a.idx = oi;
      }
    }
    if (!(a.m > -INFINITY) || a.idx >= V) {  // no finite logit in the row
      err = WISP_DEV_BAD_PROB;
      break;
    }
    if (i == k) {
      tok = a.idx;
      break;
    }
    const int32_t y = __ldg(p.draft_tokens + D0 + i);
    if (y < 0 || y >= V) {
      err = WISP_DEV_BAD_TOKEN;
      break;
    }
    if (y != a.idx) {
      L = i;
      tok = a.idx;
      break;
    }
  }
  if (lane == 0) {
    if (err) {
      report(p.status, err, p.request_ids, r);
      p.accepted_len[r] = -1;
      p.next_token[r] = -1;
    } else {
      p.accepted_len[r] = L;
      p.next_token[r] = tok;
    }
  }
}

// ---------------------------------------------------------------------------- host side
namespace {

template <typename LT>
cudaError_t set_attr() {
  const int dyn = (int)(kRingBytes + kExpTabBytes);
  cudaError_t e = cudaFuncSetAttribute(accept_kernel<LT>, cudaFuncAttributeMaxDynamicSharedMemorySize, dyn);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(accept_kernel<LT>, cudaFuncAttributePreferredSharedMemoryCarveout,
                             cudaSharedmemCarveoutMaxShared);
  return e;
}

template <typename LT>
cudaError_t launch_t(const AcceptParams &ap, int sms, cudaStream_t s, bool pdl) {
  cudaLaunchConfig_t cfg;
  memset(&cfg, 0, sizeof cfg);
  cfg.gridDim = dim3((unsigned)(sms * kAcceptCtasPerSM));
  cfg.blockDim = dim3(kCtaThreads);
  cfg.dynamicSmemBytes = kRingBytes + kExpTabBytes;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  // programmatic dependent launch: the CTAs may be placed while the planner runs (the kernel
  // waits for it before reading anything)
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, accept_kernel<LT>, ap);
}

// exp(u) for the table's bf16 values, in double (the host's exp), as mantissa and exponent:
// v = f 2^e with f in [0.5, 1) gives M = f 2^64 (exact: 53 significant bits) and E = e - 1.
void host_exp_table(unsigned long long *out) {
  for (int idx = 0; idx < kExpTabSize; ++idx) {
    const uint32_t sign = (uint32_t)idx / (kExpTabBinades * 128), rem = (uint32_t)idx % (kExpTabBinades * 128);
    const uint32_t bits = (sign << 15) | (((rem >> 7) + kExpTabLo) << 7) | (rem & 0x7Fu);
    const uint32_t f32 = bits << 16;
    float u;
    memcpy(&u, &f32, sizeof u);
    int e2 = 0;
    const double f = std::frexp(std::exp((double)u), &e2);
    const unsigned long long M = (unsigned long long)std::ldexp(f, 64);
    out[idx] = (M & ~0xFFull) | (unsigned long long)(e2 - 1 + 128);
  }
}

}  // namespace

cudaError_t accept_setup() {
  cudaError_t e = set_attr<float>();
  if (e == cudaSuccess) e = set_attr<uint16_t>();
  if (e == cudaSuccess) {
    static unsigned long long host[kExpTabSize];
    static bool filled = false;
    if (!filled) {
      host_exp_table(host);
      filled = true;
    }
    e = cudaMemcpyToSymbol(g_exp_m64, host, sizeof host);
  }
  return e;
}

cudaError_t accept_launch(const AcceptParams &p, bool bf16, int sms, cudaStream_t s, bool pdl) {
  return bf16 ? launch_t<uint16_t>(p, sms, s, pdl) : launch_t<float>(p, sms, s, pdl);
}

cudaError_t accept_greedy_launch(const AcceptParams &p, bool bf16, cudaStream_t s) {
  const unsigned g1 = (unsigned)((p.total_rows * p.slices + NW - 1) / NW), g2 = (unsigned)((p.B + NW - 1) / NW);
  if (bf16) {
    row_argmax_kernel<uint16_t><<<g1, NT, 0, s>>>(p);
    greedy_walk_kernel<uint16_t><<<g2, NT, 0, s>>>(p);
  } else {
    row_argmax_kernel<float><<<g1, NT, 0, s>>>(p);
    greedy_walk_kernel<float><<<g2, NT, 0, s>>>(p);
  }
  return cudaGetLastError();
}

}  // namespace wisp
