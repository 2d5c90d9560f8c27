// accept.cu -- the in-order speculative acceptance pass over the vocabulary (Eq. 1-3).
//
// Two launches.
//
// row_stats_kernel: warp (row, slice) streams one vocabulary slice of one logit row once, as
// 16-byte vectors; every lane keeps a running max, a double-float running sum of exp(z - max)
// (fp32 terms, pairwise within a vector) and the terms of a certified bound on the relative
// error of the normaliser Z (exp error, rounding of the argument, every rescale, pairwise sums);
// the warp merges them into the slice's statistics.  Every row of the batch is processed, in
// parallel, so the pass runs at HBM bandwidth; rows past a request's first rejection are read
// although the rule never uses them.
//
// accept_kernel: one thread-block cluster of C CTAs (C = 1..8, chosen from the batch size) per
// request.  Walk (Eq. 1-2): warp w merges the slice statistics of row i0 + w (rows in batches
// of 8; row i scores draft token i+1, row k is the bonus row) and thread 0 takes the decisions
// u_i <= min(1, p(y)/q(y)) in order, in fp32 when u_i lies outside the certified interval of the
// ratio; otherwise the cluster recomputes that row's Z and p(y) in double-float arithmetic
// (Tang's table-driven exp) and decides on those.  The walk stops at the first rejection.
// Draw (Eq. 3): from max(0, p_L - q_{L+1}) after a rejection, else from p_L, by inverse CDF in
// ascending token order: CTA c owns a contiguous slice of the row; one double-float sweep gives
// per-(round, warp) tile sums in shared memory and per-CTA totals (through distributed shared
// memory, summed in rank order so every CTA holds bit-identical values); the CTA holding the
// crossing of u * total scans its tiles, then one warp scans the tile, then one lane its
// elements.
#include <cfloat>
#include <cooperative_groups.h>
#include <cstring>
#include <type_traits>

#include "accept.cuh"

namespace cg = cooperative_groups;

namespace wisp {

namespace {

constexpr int NW = kAcceptThreads / 32;
constexpr int NT = kAcceptThreads;
// vectors (normaliser passes) and rounds (draw sweep) a thread keeps loaded ahead of the one it
// uses, in a ring of registers with one copy of the loop body: with one 16-byte load in flight per
// thread the streams of accept_kernel are latency-bound
constexpr int kZAhead = 8;
constexpr int kSweepAhead = 4;

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

// bf16 logits take few distinct values, so the draw looks exp(u - m) up in a table of the bf16
// values u in the table's range, computed once per CTA with the very same double-float function
// (the results are bit-identical to computing every element); other values are computed directly.
__device__ __forceinline__ int exp_tab_index(uint32_t bits16) {
  const uint32_t d = ((bits16 >> 7) & 0xFFu) - (uint32_t)kExpTabLo;  // wraps below the range
  if (d >= (uint32_t)kExpTabBinades) return -1;
  return (int)((((bits16 >> 15) * kExpTabBinades + d) << 7) | (bits16 & 0x7Fu));
}
__device__ __forceinline__ uint32_t exp_tab_bits(int idx) {
  const uint32_t sign = (uint32_t)idx / (kExpTabBinades * 128), rem = (uint32_t)idx % (kExpTabBinades * 128);
  return (sign << 15) | (((rem >> 7) + kExpTabLo) << 7) | (rem & 0x7Fu);
}

// Double-float weight of one element in the draw: exp(z - m) [- q * Z, clamped at 0].
__device__ __forceinline__ ff draw_weight(float z, float m, bool residual, float q, ff Zff, const float *th,
                                          const float *tl) {
  const ff x = ff_two_sum(z, -m);
  ff e = ff_exp_nonpos(x.hi, x.lo, th, tl);
  if (residual) {
    e = ff_add(e, ff_neg(ff_mul_f(Zff, q)));
    if (!(e.hi > 0.0f)) e = {0.0f, 0.0f};
  }
  return e;
}

// Out-of-table values (rare for logits): the direct double-float exp, kept out of line so that the
// unrolled loops stay small.
__device__ __noinline__ ff exp_direct(float z, float m, const float *th, const float *tl) {
  return draw_weight(z, m, false, 0.0f, ff{}, th, tl);
}

// exp(z - m) of element i of vector w; bf16: from the table when z is in its range.
template <typename LT>
__device__ __forceinline__ ff elem_exp(const uint4 &w, int i, float m, const ff *tab, const float *th, const float *tl);
template <>
__device__ __forceinline__ ff elem_exp<float>(const uint4 &w, int i, float m, const ff *, const float *th, const float *tl) {
  return draw_weight(vec_elem<float>(w, i), m, false, 0.0f, ff{}, th, tl);
}
template <>
__device__ __forceinline__ ff elem_exp<uint16_t>(const uint4 &w, int i, float m, const ff *tab, const float *th,
                                                 const float *tl) {
  const uint32_t u = (i >> 1) == 0 ? w.x : (i >> 1) == 1 ? w.y : (i >> 1) == 2 ? w.z : w.w;
  const int idx = exp_tab_index((i & 1) ? (u >> 16) : (u & 0xFFFFu));
  if (tab && idx >= 0) return tab[idx];
  return exp_direct(vec_elem<uint16_t>(w, i), m, th, tl);
}

// Sum of two non-negative double-float values: Dekker's addition without the TwoSum of the low
// parts.  With operands of one sign no cancellation occurs and the relative error stays within
// about 3 * 2^-48 (the full ff_add is kept wherever a difference is formed).
__device__ __forceinline__ ff ff_add_pos(ff a, ff b) {
  ff s = ff_two_sum(a.hi, b.hi);
  s.lo = __fadd_rn(s.lo, __fadd_rn(a.lo, b.lo));
  return ff_fast_two_sum(s.hi, s.lo);
}

// Pairwise sum of the E non-negative terms of one vector (three levels for E = 8).
template <int E>
__device__ __forceinline__ ff ff_tree_pos(ff (&t)[E]) {
#pragma unroll
  for (int w = 1; w < E; w <<= 1) {
#pragma unroll
    for (int i = 0; i < E; i += 2 * w) t[i] = ff_add_pos(t[i], t[i + w]);
  }
  return t[0];
}

// Draw weight from e = exp(z - m): e itself, or the residual max(0, e - q Z) (as draw_weight).
__device__ __forceinline__ ff weight_from(ff e, bool residual, float q, ff Zff) {
  if (residual) {
    e = ff_add(e, ff_neg(ff_mul_f(Zff, q)));
    if (!(e.hi > 0.0f)) e = {0.0f, 0.0f};
  }
  return e;
}


// Per-thread streaming statistics of one row slice (see the file comment).
struct RowStats {
  float m;       // running max
  ff s;          // sum of exp(z - m)
  float A;       // sum of exp(z - m) * |z - m|  (bounds the effect of rounding z - m)
  int nres;      // rescales so far
  float mfirst;  // first finite max (bounds the size of all rescale arguments)
};

__device__ __forceinline__ void stats_init(RowStats &st) {
  st.m = -INFINITY;
  st.s = {0.0f, 0.0f};
  st.A = 0.0f;
  st.nres = 0;
  st.mfirst = INFINITY;
}

// Move the statistics to a larger reference max mnew.
__device__ __forceinline__ void stats_rebase(RowStats &st, float mnew) {
  if (st.m == -INFINITY) {
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

// Add one chunk of NV vectors (a thread's next elements of its slice): the chunk max first (one
// rescale at most per chunk), then exp(z - m) = 2^((z - m) * log2 e) per element, a pairwise fp32
// sum of the chunk added to the double-float running sum, and the bound term A.
template <typename LT, int NV>
__device__ __forceinline__ void stats_add_chunk(RowStats &st, const uint4 (&w)[NV]) {
  constexpr int E = LTraits<LT>::E;
  constexpr int N = NV * E;
  float z[N];
#pragma unroll
  for (int u = 0; u < NV; ++u) {
#pragma unroll
    for (int i = 0; i < E; ++i) z[u * E + i] = vec_elem<LT>(w[u], i);
  }
  float mx[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) mx[i] = z[i];
#pragma unroll
  for (int i = 8; i < N; ++i) mx[i & 7] = fmaxf(mx[i & 7], z[i]);
  const float cm = fmaxf(fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])), fmaxf(fmaxf(mx[4], mx[5]), fmaxf(mx[6], mx[7])));
  if (cm == -INFINITY) return;  // nothing but padding (or -inf logits)
  if (st.m == -INFINITY) st.mfirst = cm;
  stats_rebase(st, cm);
  float e[N];
  float a[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
  for (int i = 0; i < N; ++i) {
    const float x = z[i] - st.m;
    e[i] = ex2_approx(x * kLog2e);
    a[i & 3] = fmaf(e[i], fminf(-x, 104.0f), a[i & 3]);
  }
#pragma unroll
  for (int w2 = 1; w2 < N; w2 <<= 1) {
#pragma unroll
    for (int i = 0; i < N; i += 2 * w2) e[i] += e[i + w2];
  }
  st.s = ff_add_f(st.s, e[0]);
  st.A += (a[0] + a[1]) + (a[2] + a[3]);
}

struct Decide {
  int flag;  // 0 accept, 1 reject, 2 uncertain, 4 bad prob
  float zy, qy, u;
};

// Warp-wide merge of the S <= 32 slice statistics of one row (lane q reads slice q): the same
// max / rebase / tree-sum, so every lane (and every CTA that does it) holds identical values.
// The slice-to-row rebase is not counted in nres; the decision bound allows for it.
__device__ __forceinline__ RowStats merge_parts(const RowPart *parts, int S) {
  const int lane = threadIdx.x & 31;
  RowStats q;
  stats_init(q);
  if (lane < S) {
    const RowPart t = parts[lane];
    q.m = t.m;
    q.s = {t.s_hi, t.s_lo};
    q.A = t.A;
    q.mfirst = t.mfirst;
    q.nres = t.nres;
  }
  float gm = q.m, gf = q.mfirst;
  int gn = q.nres;
  for (int o = 16; o > 0; o >>= 1) {
    gm = fmaxf(gm, __shfl_xor_sync(0xffffffffu, gm, o));
    gf = fminf(gf, __shfl_xor_sync(0xffffffffu, gf, o));
    gn = max(gn, __shfl_xor_sync(0xffffffffu, gn, o));
  }
  if (q.m > -INFINITY) stats_rebase(q, gm);
  ff gs = q.m > -INFINITY ? q.s : ff{0.0f, 0.0f};
  float ga = q.m > -INFINITY ? q.A : 0.0f;
  for (int o = 16; o > 0; o >>= 1) {
    gs = ff_add(gs, ff_shfl_xor(gs, o));
    ga += __shfl_xor_sync(0xffffffffu, ga, o);
  }
  RowStats r;
  r.m = gm;
  r.s = gs;
  r.A = ga;
  r.nres = gn;
  r.mfirst = gf;
  return r;
}

}  // namespace

// Statistics of one vocabulary slice of one logit row (Eq. 1 needs p = softmax of the row):
// warp (row, slice) streams its slice once, every lane keeping a running max, a double-float sum
// of exp(z - m) and the error terms over chunks of 4 vectors (the next chunk's loads are issued
// before the current one is reduced); the lanes are merged with shuffles (max, rebase, tree sum)
// and lane 0 writes the slice's statistics.  No shared memory, no block barrier.
template <typename LT>
__global__ void __launch_bounds__(NT) row_stats_kernel(const __grid_constant__ AcceptParams p) {
  constexpr int E = LTraits<LT>::E;
  const int lane = threadIdx.x & 31;
  const int64_t unit = (int64_t)blockIdx.x * NW + (threadIdx.x >> 5);
  if (unit >= p.total_rows * p.slices) return;
  const int64_t row = unit / p.slices;
  const int sl = (int)(unit % p.slices);
  const int V = p.V;
  const LT *rowp = static_cast<const LT *>(p.logits) + row * (int64_t)V;
  const bool vec_z = p.vec_z != 0;
  const int64_t nvec = (V + E - 1) / E;
  const int64_t vlo = min(nvec, (int64_t)sl * p.vps);
  const int64_t vhi = min(nvec, vlo + p.vps);
  const uint32_t ni = LTraits<LT>::NEG_INF2;
  auto load4 = [&](int64_t base, uint4 (&w)[4]) {
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int64_t vi = base + u * 32;
      w[u] = vi < vhi ? load_vec<LT>(rowp, vi, V, vec_z) : make_uint4(ni, ni, ni, ni);
    }
  };
  RowStats st;
  stats_init(st);
  uint4 cur[4];
  load4(vlo + lane, cur);
  for (int64_t base = vlo + lane; base < vhi; base += 4 * 32) {
    uint4 nxt[4];
    load4(base + 4 * 32, nxt);
    stats_add_chunk<LT, 4>(st, cur);
#pragma unroll
    for (int u = 0; u < 4; ++u) cur[u] = nxt[u];
  }
  // lanes -> slice: max, rebase, tree sum (the lane-to-slice rebase counts as one more rescale)
  float wm = st.m, wf = st.mfirst;
  int wn = st.nres;
  for (int o = 16; o > 0; o >>= 1) {
    wm = fmaxf(wm, __shfl_xor_sync(0xffffffffu, wm, o));
    wf = fminf(wf, __shfl_xor_sync(0xffffffffu, wf, o));
    wn = max(wn, __shfl_xor_sync(0xffffffffu, wn, o));
  }
  if (wm > -INFINITY) stats_rebase(st, wm);
  ff ws = st.m > -INFINITY ? st.s : ff{0.0f, 0.0f};
  float wa = st.m > -INFINITY ? st.A : 0.0f;
  for (int o = 16; o > 0; o >>= 1) {
    ws = ff_add(ws, ff_shfl_xor(ws, o));
    wa += __shfl_xor_sync(0xffffffffu, wa, o);
  }
  if (lane == 0) {
    RowPart out;
    out.m = wm;
    out.s_hi = ws.hi;
    out.s_lo = ws.lo;
    out.A = wa;
    out.mfirst = wf;
    out.nres = wn + 1;
    p.parts[unit] = out;
  }
}

template <typename LT>
__global__ void __launch_bounds__(NT, 2) accept_kernel(const __grid_constant__ AcceptParams p) {
  constexpr int E = LTraits<LT>::E;
  extern __shared__ ff s_tile[];  // [rounds * NW] per-(round, warp) draw sums, then the exp table (bf16)
  __shared__ float s_th[256], s_tl[256];
  __shared__ RowStats s_wst[NW];
  __shared__ RowStats s_pub[2];   // this CTA's published totals (ring of 2)
  __shared__ ff s_tot[kMaxAcceptCluster];
  __shared__ RowStats s_rows[NW]; // merged statistics of the rows being walked
  __shared__ int s_walk[2];       // walk state, row within the batch
  __shared__ float s_zy[kPreload], s_qy[kPreload], s_u[kPreload];
  __shared__ Decide s_dec;
  __shared__ int s_bad;
  __shared__ int s_owner, s_take_last;
  __shared__ ff s_thr;

  // launched as a programmatic dependent of the kernel before it: nothing is read before that
  // grid has completed and its writes are visible
  asm volatile("griddepcontrol.wait;" ::: "memory");
  cg::cluster_group cluster = cg::this_cluster();
  const int C = p.cluster;
  const int rank = (int)cluster.block_rank();
  const int r = blockIdx.x / C;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  if (r >= p.B) return;                 // whole clusters only (grid = B * C)
  if (p.req_flag[r] != REQ_OK) return;  // uniform across the cluster

  const int V = p.V;
  const int k = p.draft_lens[r];
  const int64_t Q0 = p.q_row_start[r], D0 = p.draft_start[r];
  const LT *logits = static_cast<const LT *>(p.logits);
  const bool vec_z = p.vec_z != 0, vec_q = p.vec_q != 0;
  const int64_t nvec = (V + E - 1) / E;
  const int64_t vlo = min((int64_t)nvec, (int64_t)rank * p.vpc);
  const int64_t vhi = min((int64_t)nvec, vlo + p.vpc);
  const int rounds = (int)((vhi - vlo + NT - 1) / NT);
  int xslot = 0;

  for (int i = tid; i < 256; i += NT) {
    s_th[i] = p.tab.hi[i];
    s_tl[i] = p.tab.lo[i];
  }
  if (tid == 0) s_bad = 0;
  __syncthreads();
  // validate every draft token and gather the decision inputs of the first rows
  for (int i = tid; i < k; i += NT) {
    const int32_t y = __ldg(p.draft_tokens + D0 + i);
    if (y < 0 || y >= V) {
      atomicOr(&s_bad, 1);
    } else if (i < kPreload) {
      s_zy[i] = load_scalar(logits + (Q0 + i) * (int64_t)V, y);
      s_qy[i] = __ldg(p.draft_probs + (D0 + i) * (int64_t)V + y);
      s_u[i] = __ldg(p.accept_u + D0 + i);
    }
  }
  __syncthreads();

  // ---- reductions across the cluster -----------------------------------------------
  // ff total over the CTA (per-thread values), every CTA's total gathered into s_tot,
  // and their sum in rank order
  auto cluster_total = [&](ff a) -> ff {
    for (int o = 16; o > 0; o >>= 1) a = ff_add(a, ff_shfl_xor(a, o));
    if (lane == 0) s_wst[warp].s = a;
    __syncthreads();
    if (tid == 0) {
      ff t = {0.0f, 0.0f};
      for (int w = 0; w < NW; ++w) t = ff_add(t, s_wst[w].s);
      s_pub[xslot].s = t;
    }
    cluster.sync();
    if (tid < C) s_tot[tid] = cluster.map_shared_rank(&s_pub[xslot], tid)->s;
    __syncthreads();
    ff t = {0.0f, 0.0f};
    for (int q = 0; q < C; ++q) t = ff_add(t, s_tot[q]);
    xslot ^= 1;
    return t;
  };
  // double-float sum of f(element) over this thread's vectors of a row, in vector order; w[u] holds
  // the vector u rounds ahead of the current one
  auto thread_sum = [&](const LT *row, auto &&f) -> ff {
    ff acc = {0.0f, 0.0f};
    uint4 w[kZAhead];
#pragma unroll
    for (int u = 0; u < kZAhead; ++u) {
      const int64_t vi = vlo + tid + (int64_t)u * NT;
      if (vi < vhi) w[u] = load_vec<LT>(row, vi, V, vec_z);
    }
#pragma unroll 1
    for (int64_t vi = vlo + tid; vi < vhi; vi += NT) {
      const uint4 cur = w[0];
#pragma unroll
      for (int u = 0; u + 1 < kZAhead; ++u) w[u] = w[u + 1];
      const int64_t vn = vi + (int64_t)kZAhead * NT;
      if (vn < vhi) w[kZAhead - 1] = load_vec<LT>(row, vn, V, vec_z);
      ff t[E];
#pragma unroll
      for (int i = 0; i < E; ++i) t[i] = f(cur, i);
      acc = ff_add_pos(acc, ff_tree_pos<E>(t));
    }
    return acc;
  };
  // double-float normaliser of a row (re-streamed); m is the row's exact max
  auto row_Zff = [&](const LT *row, float m) -> ff {
    return cluster_total(thread_sum(row, [&](const uint4 &w, int i) {
      const ff x = ff_two_sum(vec_elem<LT>(w, i), -m);
      return ff_exp_nonpos(x.hi, x.lo, s_th, s_tl);
    }));
  };

  // ---- the in-order walk (Eq. 1-2) -------------------------------------------
  // The rows' statistics come from row_stats_kernel: warp w merges the slices of row i0 + w,
  // then thread 0 takes the decisions of the batch in order; a decision inside the certified
  // interval of the fp32 ratio stops it, the whole cluster recomputes that row's normaliser in
  // double-float arithmetic, and the walk resumes after it.
  int L = k;
  int err = s_bad ? WISP_DEV_BAD_TOKEN : 0;
  float m = 0.0f;
  ff Zff = {0.0f, 0.0f};
  bool have_Zff = false;
  bool done = err != 0;
  const int nsl = p.slices;
  for (int i0 = 0; i0 <= k && !done; i0 += NW) {
    if (i0 + warp <= k) {
      const RowStats rs = merge_parts(p.parts + (Q0 + i0 + warp) * (int64_t)nsl, nsl);
      if (lane == 0) s_rows[warp] = rs;
    }
    __syncthreads();
    int j = 0;
    while (!done) {
      if (tid == 0) {
        // state: 0 batch exhausted, 1 bonus row reached, 2 rejected, 3 bad row, 4 uncertain
        int state = 0, jj = j;
        Decide d;
        d.flag = 0;
        for (; jj < NW && i0 + jj <= k; ++jj) {
          const int i = i0 + jj;
          const RowStats rs = s_rows[jj];
          const float mi = rs.m;
          const ff Z = rs.s;
          if (!(mi > -INFINITY) || !(mi < INFINITY) || !(Z.hi > 0.0f) || !(Z.hi < INFINITY) || !(rs.A >= 0.0f)) {
            state = 3;
            break;
          }
          if (i == k) {
            state = 1;  // every draft token accepted
            break;
          }
          if (i < kPreload) {
            d.zy = s_zy[i];
            d.qy = s_qy[i];
            d.u = s_u[i];
          } else {
            const int32_t y = __ldg(p.draft_tokens + D0 + i);
            d.zy = load_scalar(logits + (Q0 + i) * (int64_t)V, y);
            d.qy = __ldg(p.draft_probs + (D0 + i) * (int64_t)V + y);
            d.u = __ldg(p.accept_u + D0 + i);
          }
          if (!(d.qy >= 0.0f)) {
            state = 3;
            break;
          }
          if (d.qy == 0.0f) continue;  // a = 1: accepted
          if (!(d.zy > -INFINITY)) {  // a masked token: p(y) = 0 exactly, accepted only if u = 0
            if (d.u <= 0.0f) continue;
            state = 2;
            break;
          }
          // certified relative error of Z (see RowStats) and of the ratio p(y)/q(y)
          // terms: one exp error per element and per rescale on its way (thread, CTA, row), three
          // roundings in the argument (z - m, log2 e, the product) of every element and every
          // rescale, the 32-term pairwise sums; the decision's own exp and ratio on top
          const float x = d.zy - mi;
          // outside the range of the fp32 ratio (2^x flushes to zero below 2^-126, a subnormal q(y)
          // loses bits): decide in double precision
          if (x * kLog2e < -126.0f || d.qy < FLT_MIN) {
            state = 4;
            break;
          }
          const float dz = 1.05f * ((float)(rs.nres + 2) * kEx2RelErr + 3.0f * 0x1p-24f * (mi - rs.mfirst) +
                                    3.0f * 0x1p-24f * (rs.A / Z.hi) + 6.0f * 0x1p-24f) +
                           1e-12f;
          const float dr = dz + 1.05f * (kEx2RelErr + 3.0f * 0x1p-24f * fabsf(x) + 4.0f * 0x1p-24f);
          const float ratio = ex2_approx(x * kLog2e) / (Z.hi * d.qy);
          const float lo = fminf(1.0f, ratio * (1.0f - dr)), hi = fminf(1.0f, ratio * (1.0f + dr));
          if (d.u <= lo) continue;
          state = d.u > hi ? 2 : 4;
          break;
        }
        s_walk[0] = state;
        s_walk[1] = jj;
        s_dec = d;
      }
      __syncthreads();
      const int state = s_walk[0], jj = s_walk[1];
      if (state == 0) break;  // next batch
      if (state == 3) {
        err = WISP_DEV_BAD_PROB;
        done = true;
      } else if (state == 1 || state == 2) {
        L = i0 + jj;
        m = s_rows[jj].m;
        done = true;
      } else {
        // inside the certified interval: decide with the double-float normaliser
        const int i = i0 + jj;
        const float mi = s_rows[jj].m;
        const ff zf = row_Zff(logits + (Q0 + i) * (int64_t)V, mi);
        if (tid == 0) {
          const Decide d = s_dec;
          // p(y) / q(y) in double precision: z(y) - m is exact as a double, and neither p(y) nor a
          // subnormal q(y) leaves the double range
          const double ratio = exp((double)d.zy - (double)mi) / (ff_to_double(zf) * (double)d.qy);
          s_walk[0] = (double)d.u <= fmin(1.0, ratio) ? 0 : 1;
        }
        __syncthreads();
        if (s_walk[0] == 1) {
          L = i;
          m = mi;
          Zff = zf;
          have_Zff = true;
          done = true;
        } else {
          j = jj + 1;  // accepted: resume the walk after this row
        }
      }
      __syncthreads();  // s_walk / s_dec are rewritten by the next round
    }
  }

  if (err) {
    if (rank == 0 && tid == 0) {
      report(p.status, err, p.request_ids, r);
      p.accepted_len[r] = -1;
      p.next_token[r] = -1;
    }
    cluster.sync();
    return;
  }

  // ---- the extra token (Eq. 3) --------------------------------------------------
  const LT *row = logits + (Q0 + L) * (int64_t)V;
  const float *qrow = p.draft_probs + (D0 + L) * (int64_t)V;
  bool residual = L < k;
  // exp(u - m) of row L for the bf16 values u of the table's range
  // (only for rows much longer than the table)
  ff *s_etab = std::is_same<LT, uint16_t>::value && V >= kExpTabMinV ? s_tile + rounds * NW : nullptr;
  if (s_etab) {
#pragma unroll 2
    for (int idx = tid; idx < kExpTabSize; idx += NT) {
      const float u = bf16_bits_to_float(exp_tab_bits(idx));
      s_etab[idx] = u > m ? ff{0.0f, 0.0f} : draw_weight(u, m, false, 0.0f, ff{}, s_th, s_tl);  // u > m never occurs
    }
    __syncthreads();
  }
  if (residual && !have_Zff)
    Zff = cluster_total(thread_sum(row, [&](const uint4 &w, int i) { return elem_exp<LT>(w, i, m, s_etab, s_th, s_tl); }));
  ff S = {0.0f, 0.0f};
  for (;;) {
    ff run = {0.0f, 0.0f};
    // the row's and the draft's vectors of round rd + u in w[u], q[u]
    uint4 w[kSweepAhead];
    float q[kSweepAhead][E];
    auto load_round = [&](int rd, uint4 &wv, float (&qv)[E]) {
      const int64_t vi = vlo + (int64_t)rd * NT + tid;
      if (rd < rounds && vi < vhi) {
        wv = load_vec<LT>(row, vi, V, vec_z);
        if (residual) {
          load_q<E>(qrow, vi * E, V, vec_q, qv);
        } else {
#pragma unroll
          for (int i = 0; i < E; ++i) qv[i] = 0.0f;
        }
      }
    };
#pragma unroll
    for (int u = 0; u < kSweepAhead; ++u) load_round(u, w[u], q[u]);
#pragma unroll 1
    for (int rd = 0; rd < rounds; ++rd) {
      const uint4 cw = w[0];
      float cq[E];
#pragma unroll
      for (int i = 0; i < E; ++i) cq[i] = q[0][i];
#pragma unroll
      for (int u = 0; u + 1 < kSweepAhead; ++u) {
        w[u] = w[u + 1];
#pragma unroll
        for (int i = 0; i < E; ++i) q[u][i] = q[u + 1][i];
      }
      load_round(rd + kSweepAhead, w[kSweepAhead - 1], q[kSweepAhead - 1]);
      const int64_t vi = vlo + (int64_t)rd * NT + tid;
      ff part = {0.0f, 0.0f};
      if (vi < vhi) {
        ff t[E];
#pragma unroll
        for (int i = 0; i < E; ++i) t[i] = weight_from(elem_exp<LT>(cw, i, m, s_etab, s_th, s_tl), residual, cq[i], Zff);
        part = ff_tree_pos<E>(t);
      }
      for (int o = 16; o > 0; o >>= 1) part = ff_add_pos(part, ff_shfl_xor(part, o));
      if (lane == 0) s_tile[rd * NW + warp] = part;
      run = ff_add_pos(run, part);
    }
    // run is the warp's sum over all rounds (same value in every lane): count it once
    if (lane != 0) run = {0.0f, 0.0f};
    S = cluster_total(run);
    if (residual && !(S.hi > 0.0f)) {
      residual = false;  // the residual has no mass (only through rounding): draw from p_L instead
      continue;
    }
    break;
  }

  // which CTA holds the crossing of u * S (every CTA computes the same answer)
  if (tid == 0) {
    const ff thr = ff_mul_f(S, __ldg(p.sample_u + r));
    ff run = {0.0f, 0.0f};
    int owner = -1, last_pos = -1;
    ff local = thr;
    for (int q = 0; q < C; ++q) {
      const ff nxt = ff_add(run, s_tot[q]);
      if (s_tot[q].hi > 0.0f) last_pos = q;
      if (owner < 0 && ff_gt(nxt, thr)) {
        owner = q;
        local = ff_add(thr, ff_neg(run));
      }
      run = nxt;
    }
    s_owner = owner >= 0 ? owner : last_pos;
    s_take_last = owner >= 0 ? 0 : 1;
    s_thr = local;
  }
  __syncthreads();
  const int owner = s_owner;
  if (rank == owner && warp == 0) {
    // tile entries (round, warp) are in token order: find the one holding the crossing
    const int n_ent = rounds * NW;
    bool take_last = s_take_last != 0;
    const ff thr = s_thr;
    int entry = -1;
    ff before = {0.0f, 0.0f};
    if (!take_last) {
      ff base = {0.0f, 0.0f};
      for (int e0 = 0; e0 < n_ent && entry < 0; e0 += 32) {
        const ff v = e0 + lane < n_ent ? s_tile[e0 + lane] : ff{0.0f, 0.0f};
        ff incl = v;
        for (int d = 1; d < 32; d <<= 1) {
          const ff o = ff_shfl_up(incl, d);
          if (lane >= d) incl = ff_add(incl, o);
        }
        incl = ff_add(base, incl);
        ff excl = ff_shfl_up(incl, 1);
        if (lane == 0) excl = base;
        const unsigned hit = __ballot_sync(0xffffffffu, e0 + lane < n_ent && ff_gt(incl, thr));
        if (hit) {
          const int l0 = __ffs(hit) - 1;
          entry = e0 + l0;
          before = {__shfl_sync(0xffffffffu, excl.hi, l0), __shfl_sync(0xffffffffu, excl.lo, l0)};
        }
        base = {__shfl_sync(0xffffffffu, incl.hi, 31), __shfl_sync(0xffffffffu, incl.lo, 31)};
      }
      if (entry < 0) take_last = true;  // rounding left no crossing inside this CTA
    }
    if (take_last) {
      entry = -1;
      for (int e0 = ((n_ent - 1) / 32) * 32; e0 >= 0 && entry < 0; e0 -= 32) {
        const bool pos = e0 + lane < n_ent && s_tile[e0 + lane].hi > 0.0f;
        const unsigned b = __ballot_sync(0xffffffffu, pos);
        if (b) entry = e0 + 31 - __clz(b);
      }
    }
    if (entry >= 0) {
      // re-derive the tile's weights: lane sums, inclusive scan, then one lane's elements
      const int rd = entry / NW, ww = entry % NW;
      const int64_t vi = vlo + (int64_t)rd * NT + ww * 32 + lane;
      float q[E];
      ff wts[E];
      ff lsum = {0.0f, 0.0f};
#pragma unroll
      for (int i = 0; i < E; ++i) wts[i] = {0.0f, 0.0f};
      if (vi < vhi) {
        const uint4 w = load_vec<LT>(row, vi, V, vec_z);
        if (residual) {
          load_q<E>(qrow, vi * E, V, vec_q, q);
        } else {
#pragma unroll
          for (int i = 0; i < E; ++i) q[i] = 0.0f;
        }
#pragma unroll
        for (int i = 0; i < E; ++i) {
          wts[i] = weight_from(elem_exp<LT>(w, i, m, s_etab, s_th, s_tl), residual, q[i], Zff);
          lsum = ff_add(lsum, wts[i]);
        }
      }
      const ff rem = ff_add(thr, ff_neg(before));
      ff incl = lsum;
      for (int d = 1; d < 32; d <<= 1) {
        const ff o = ff_shfl_up(incl, d);
        if (lane >= d) incl = ff_add(incl, o);
      }
      ff excl = ff_shfl_up(incl, 1);
      if (lane == 0) excl = {0.0f, 0.0f};
      int l0 = -1;
      if (!take_last) {
        const unsigned hit = __ballot_sync(0xffffffffu, ff_gt(incl, rem));
        if (hit) l0 = __ffs(hit) - 1;
      }
      const bool last_mode = take_last || l0 < 0;
      if (last_mode) {
        const unsigned b = __ballot_sync(0xffffffffu, lsum.hi > 0.0f);
        l0 = b ? 31 - __clz(b) : -1;
      }
      if (l0 >= 0 && lane == l0) {
        const ff r2 = ff_add(rem, ff_neg(excl));
        ff acc = {0.0f, 0.0f};
        int tok = -1, last = -1;
        for (int i = 0; i < E; ++i) {
          const int64_t v = vi * E + i;
          if (v >= V) break;
          if (wts[i].hi > 0.0f) last = (int)v;
          acc = ff_add(acc, wts[i]);
          if (!last_mode && ff_gt(acc, r2)) {
            tok = (int)v;
            break;
          }
        }
        p.next_token[r] = tok >= 0 ? tok : last;
      }
    } else if (lane == 0) {
      p.next_token[r] = -1;  // no element with mass: cannot happen for a finite row
    }
  }
  if (rank == 0 && tid == 0) {
    p.accepted_len[r] = L;
    if (owner < 0) p.next_token[r] = -1;
  }
  cluster.sync();  // no CTA leaves while another may still read its shared memory
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
  // the maximum shared-memory carveout, like the attention kernel, so that these CTAs can share an
  // SM with an attention CTA when wisp_verify_step runs both at once
  cudaError_t e = cudaFuncSetAttribute(accept_kernel<LT>, cudaFuncAttributeMaxDynamicSharedMemorySize, 96 * 1024);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(accept_kernel<LT>, cudaFuncAttributePreferredSharedMemoryCarveout, cudaSharedmemCarveoutMaxShared);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(row_stats_kernel<LT>, cudaFuncAttributePreferredSharedMemoryCarveout, cudaSharedmemCarveoutMaxShared);
  return e;
}

template <typename LT>
cudaError_t stats_t(const AcceptParams &ap, cudaStream_t s) {
  row_stats_kernel<LT><<<(unsigned)((ap.total_rows * ap.slices + NW - 1) / NW), NT, 0, s>>>(ap);
  return cudaGetLastError();
}

template <typename LT>
cudaError_t walk_t(const AcceptParams &ap, cudaStream_t s) {
  const int rounds = (ap.vpc + NT - 1) / NT;
  cudaLaunchConfig_t cfg;
  memset(&cfg, 0, sizeof cfg);
  cfg.gridDim = dim3((unsigned)((int64_t)ap.B * ap.cluster));
  cfg.blockDim = dim3(NT);
  const bool tab = std::is_same<LT, uint16_t>::value && ap.V >= kExpTabMinV;
  cfg.dynamicSmemBytes = (size_t)rounds * NW * sizeof(ff) + (tab ? kExpTabSize * sizeof(ff) : 0);
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)ap.cluster;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  // programmatic dependent launch: the clusters may be placed while the previous kernel's last
  // CTAs run (the kernel waits for it before it reads anything)
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, accept_kernel<LT>, ap);
}

}  // namespace

cudaError_t accept_setup() {
  cudaError_t e = set_attr<float>();
  if (e == cudaSuccess) e = set_attr<uint16_t>();
  return e;
}

cudaError_t accept_stats_launch(const AcceptParams &p, bool bf16, cudaStream_t s) {
  return bf16 ? stats_t<uint16_t>(p, s) : stats_t<float>(p, s);
}

cudaError_t accept_walk_launch(const AcceptParams &p, bool bf16, cudaStream_t s) {
  return bf16 ? walk_t<uint16_t>(p, s) : walk_t<float>(p, s);
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
