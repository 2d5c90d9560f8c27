// accept.cu -- the in-order speculative acceptance pass over the vocabulary (Eq. 1-3).
//
// One thread-block cluster of C CTAs serves one request; each CTA owns a contiguous
// slice of the vocabulary (16-byte tiles of 32 lanes).  For logit rows i = 0, 1, ...
// of the request (row i scores draft token i+1, Sec. 4.5):
//   1. the row max m_i and normaliser Z_i = sum_v exp(z_v - m_i) are reduced within
//      each CTA (warp shuffles) and across the cluster through distributed shared
//      memory, every CTA combining the C partials in rank order so that all CTAs hold
//      bit-identical values and take identical branches;
//   2. the acceptance of Eq. 1, u_i <= min(1, p(y)/q(y)), is decided with a certified
//      error bound on the fp32 normaliser; a decision inside the bound is re-taken
//      with the normaliser recomputed in double-float arithmetic;
//   3. the walk stops at the first rejection (Eq. 2), so rows after it are never read.
// The extra token of Eq. 3 is then drawn by inverse CDF from max(0, p_L - q_{L+1})
// (rejection) or p_L (all accepted), with every weight and prefix sum in double-float
// arithmetic: per-(tile, lane) partial sums in shared memory, per-CTA totals exchanged
// across the cluster, and a final element scan by the one thread whose range holds the
// crossing.
#include <cooperative_groups.h>
#include <cstring>

#include "accept.cuh"

namespace cg = cooperative_groups;

namespace wisp {

namespace {

template <typename LT>
struct LTraits;
template <>
struct LTraits<float> {
  static constexpr int E = 4;  // elements per 16-byte vector
};
template <>
struct LTraits<uint16_t> {
  static constexpr int E = 8;
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

// The E elements of one lane of one tile; elements at or past V read as -inf.
template <typename LT>
__device__ __forceinline__ uint4 load_vec(const LT *row, int64_t v0, int V, bool vec_ok) {
  constexpr int E = LTraits<LT>::E;
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

// Four draft probabilities for elements v0..v0+3 (0 past V).
__device__ __forceinline__ float4 load_q4(const float *qrow, int64_t v0, int V, bool vec_ok) {
  if (vec_ok && v0 + 4 <= V) return __ldg(reinterpret_cast<const float4 *>(qrow + v0));
  float f[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) f[i] = v0 + i < V ? __ldg(qrow + v0 + i) : 0.0f;
  return make_float4(f[0], f[1], f[2], f[3]);
}

__device__ __forceinline__ float q4_elem(const float4 &q, int i) {
  return i == 0 ? q.x : i == 1 ? q.y : i == 2 ? q.z : q.w;
}

// Double-float weight of one element in the draw: exp(z - m) [- q * Z, clamped at 0].
__device__ __forceinline__ ff draw_weight(float z, float m, bool residual, float q, ff Zff,
                                          const float *th, const float *tl) {
  const ff x = ff_two_sum(z, -m);
  ff e = ff_exp_nonpos(x.hi, x.lo, th, tl);
  if (residual) {
    e = ff_add(e, ff_neg(ff_mul_f(Zff, q)));
    if (!(e.hi > 0.0f)) e = {0.0f, 0.0f};
  }
  return e;
}

struct Bcast {
  float m;
  ff Z;
  float bnd;
  int flag;
  int aux;
};

}  // namespace

template <typename LT, int NW, int MAXT>
__global__ void __launch_bounds__(NW * 32) accept_kernel(const __grid_constant__ AcceptParams p) {
  constexpr int E = LTraits<LT>::E;
  constexpr int TILE = 32 * E;
  constexpr int NT = NW * 32;
  extern __shared__ ff s_part[];  // [MAXT * NW * 32] per-(tile, lane) draw partials
  __shared__ float s_th[256], s_tl[256];
  __shared__ float4 s_pub[2];     // value this CTA publishes to the cluster (ring of 2)
  __shared__ float4 s_red[NW];
  __shared__ ff s_all[8];         // per-CTA totals gathered from the cluster
  __shared__ Bcast s_b;
  __shared__ int s_sel_entry, s_sel_last;
  __shared__ ff s_sel_before;

  cg::cluster_group cluster = cg::this_cluster();
  const int C = p.cluster;
  const int rank = (int)cluster.block_rank();
  const int r = blockIdx.x / C;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  if (r >= p.B) return;                    // whole clusters only (grid = B * C)
  if (p.req_flag[r] != REQ_OK) return;     // uniform across the cluster

  for (int i = tid; i < 256; i += NT) {
    s_th[i] = p.tab.hi[i];
    s_tl[i] = p.tab.lo[i];
  }

  const int V = p.V;
  const int k = p.draft_lens[r];
  const int64_t Q0 = p.q_row_start[r], D0 = p.draft_start[r];
  const LT *logits = static_cast<const LT *>(p.logits);
  const bool vec_z = p.vec_z != 0, vec_q = p.vec_q != 0;
  const int n_tiles = (V + TILE - 1) / TILE;
  const int tpc = (n_tiles + C - 1) / C;
  const int tile_lo = min(n_tiles, rank * tpc);
  const int tile_hi = min(n_tiles, tile_lo + tpc);
  const int my_tiles = tile_hi - tile_lo;
  int xslot = 0;

  // ---- reductions -------------------------------------------------------
  auto cta_max = [&](float v) -> float {
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    if (lane == 0) s_red[warp].x = v;
    __syncthreads();
    float m = -INFINITY;
    for (int w = 0; w < NW; ++w) m = fmaxf(m, s_red[w].x);
    __syncthreads();
    return m;
  };
  // ff sum + plain float sum, deterministic order
  auto cta_sum = [&](ff a, float b) -> float4 {
    for (int o = 16; o > 0; o >>= 1) {
      a = ff_add(a, ff_shfl_xor(a, o));
      b += __shfl_xor_sync(0xffffffffu, b, o);
    }
    if (lane == 0) s_red[warp] = make_float4(a.hi, a.lo, b, 0.0f);
    __syncthreads();
    ff t = {0.0f, 0.0f};
    float tb = 0.0f;
    for (int w = 0; w < NW; ++w) {
      t = ff_add(t, ff{s_red[w].x, s_red[w].y});
      tb += s_red[w].z;
    }
    __syncthreads();
    return make_float4(t.hi, t.lo, tb, 0.0f);
  };
  // publish this CTA's value, then every CTA reads all C values in rank order
  auto cluster_gather = [&](float4 mine) {
    if (tid == 0) s_pub[xslot] = mine;
    cluster.sync();
    if (warp == 0 && lane < C) {
      const float4 *rp = cluster.map_shared_rank(&s_pub[xslot], lane);
      const float4 v = *rp;
      s_all[lane] = ff{v.x, v.y};
      s_red[lane] = v;  // keep .z (bound) too; s_red is free here
    }
    __syncthreads();
    xslot ^= 1;
  };
  auto cluster_max = [&](float v) -> float {
    cluster_gather(make_float4(v, 0.f, 0.f, 0.f));
    float m = -INFINITY;
    for (int c = 0; c < C; ++c) m = fmaxf(m, s_all[c].hi);
    __syncthreads();
    return m;
  };
  auto cluster_sum = [&](float4 v) -> float4 {
    cluster_gather(v);
    ff t = {0.0f, 0.0f};
    float tb = 0.0f;
    for (int c = 0; c < C; ++c) {
      t = ff_add(t, s_all[c]);
      tb += s_red[c].z;
    }
    __syncthreads();
    return make_float4(t.hi, t.lo, tb, 0.0f);
  };

  // double-float normaliser of a row held in global memory (re-read through L2)
  auto row_Zff = [&](const LT *row, float m) -> ff {
    ff acc = {0.0f, 0.0f};
    for (int tl = warp; tl < my_tiles; tl += NW) {
      const uint4 w = load_vec<LT>(row, (int64_t)(tile_lo + tl) * TILE + lane * E, V, vec_z);
#pragma unroll
      for (int i = 0; i < E; ++i) {
        const ff x = ff_two_sum(vec_elem<LT>(w, i), -m);
        acc = ff_add(acc, ff_exp_nonpos(x.hi, x.lo, s_th, s_tl));
      }
    }
    const float4 c = cta_sum(acc, 0.0f);
    const float4 t = cluster_sum(c);
    return ff{t.x, t.y};
  };

  // ---- the in-order walk over rows (Eq. 1-2) -----------------------------
  int L = k;
  int err = 0;
  float m = 0.0f;
  ff Zff = {0.0f, 0.0f};
  bool have_Zff = false;
  for (int i = 0; i <= k; ++i) {
    const LT *row = logits + (Q0 + i) * (int64_t)V;
    int32_t y = 0;
    if (tid == 0 && i < k) y = __ldg(p.draft_tokens + D0 + i);
    uint4 zr[MAXT];
#pragma unroll
    for (int t = 0; t < MAXT; ++t) {
      const int tl = warp + t * NW;
      zr[t] = tl < my_tiles ? load_vec<LT>(row, (int64_t)(tile_lo + tl) * TILE + lane * E, V, vec_z)
                            : make_uint4(0, 0, 0, 0);
    }
    float lm = -INFINITY;
#pragma unroll
    for (int t = 0; t < MAXT; ++t) {
      if (warp + t * NW < my_tiles) {
#pragma unroll
        for (int e = 0; e < E; ++e) lm = fmaxf(lm, vec_elem<LT>(zr[t], e));
      }
    }
    m = cluster_max(cta_max(lm));
    // gather what the decision needs while the sum runs
    float zy = 0.0f, qy = 0.0f, u = 0.0f;
    int tok_bad = 0;
    if (tid == 0 && i < k) {
      if (y < 0 || y >= V) {
        tok_bad = 1;
      } else {
        zy = load_scalar(row, y);
        qy = __ldg(p.draft_probs + (D0 + i) * (int64_t)V + y);
        u = __ldg(p.accept_u + D0 + i);
      }
    }
    // Z = sum exp(z - m): fp32 terms, pairwise within a vector, double-float across vectors;
    // bnd = sum e * |x| bounds the effect of rounding x = z - m.
    ff zs = {0.0f, 0.0f};
    float bnd = 0.0f;
#pragma unroll
    for (int t = 0; t < MAXT; ++t) {
      if (warp + t * NW < my_tiles) {
        float ev[E];
#pragma unroll
        for (int e = 0; e < E; ++e) {
          const float x = vec_elem<LT>(zr[t], e) - m;
          ev[e] = expf(x);
          bnd = fmaf(ev[e], fminf(-x, 104.0f), bnd);
        }
#pragma unroll
        for (int w = 1; w < E; w <<= 1) {
#pragma unroll
          for (int e = 0; e < E; e += 2 * w) ev[e] += ev[e + w];
        }
        zs = ff_add_f(zs, ev[0]);
      }
    }
    const float4 zc = cluster_sum(cta_sum(zs, bnd));
    const ff Z = {zc.x, zc.y};
    const float zbnd = zc.z;
    have_Zff = false;
    if (!(m > -INFINITY) || !(m < INFINITY) || !(Z.hi > 0.0f) || !(Z.hi < INFINITY)) {
      err = WISP_DEV_BAD_PROB;
      break;
    }
    if (i == k) break;  // bonus row reached: every draft token accepted

    // Eq. 1 decision, taken identically by thread 0 of every CTA
    if (tid == 0) {
      int flag = 0;  // 0 accept, 1 reject, 2 uncertain, 3 bad token, 4 bad prob
      if (tok_bad) {
        flag = 3;
      } else if (!(qy >= 0.0f)) {
        flag = 4;
      } else if (qy == 0.0f) {
        flag = 0;  // a = 1
      } else {
        const double Zd = ff_to_double(Z);
        const double ratio = exp((double)zy - (double)m) / Zd / (double)qy;
        // relative error of Zd: expf (2 ulp), rounding of x (bnd), pairwise depth 3, ff sums
        const double delta =
            1.02 * (0x1p-22 + 3.0 * 0x1p-24 + 0x1p-24 * ((double)zbnd / Zd)) + 1e-12;
        const double lo = fmin(1.0, ratio / (1.0 + delta)), hi = fmin(1.0, ratio * (1.0 + delta));
        const double ud = (double)u;
        flag = ud <= lo ? 0 : (ud > hi ? 1 : 2);
      }
      s_b.flag = flag;
      s_b.m = zy;
      s_b.bnd = qy;
      s_b.aux = __float_as_int(u);
    }
    __syncthreads();
    int flag = s_b.flag;
    if (flag == 3 || flag == 4) {
      err = flag == 3 ? WISP_DEV_BAD_TOKEN : WISP_DEV_BAD_PROB;
      break;
    }
    if (flag == 2) {
      // certified fp32 bound not enough: decide with the double-float normaliser
      const float zy_b = s_b.m, qy_b = s_b.bnd, u_b = __int_as_float(s_b.aux);
      Zff = row_Zff(row, m);
      have_Zff = true;
      if (tid == 0) {
        const double ratio = exp((double)zy_b - (double)m) / ff_to_double(Zff) / (double)qy_b;
        s_b.flag = (double)u_b <= fmin(1.0, ratio) ? 0 : 1;
      }
      __syncthreads();
      flag = s_b.flag;
    }
    __syncthreads();
    if (flag == 1) {
      L = i;
      break;
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

  // ---- the extra token (Eq. 3) ---------------------------------------------
  const LT *row = logits + (Q0 + L) * (int64_t)V;
  const float *qrow = p.draft_probs + (D0 + L) * (int64_t)V;
  bool residual = L < k;
  if (residual && !have_Zff) Zff = row_Zff(row, m);
  ff S = {0.0f, 0.0f};
  for (;;) {
    ff my_total = {0.0f, 0.0f};
    for (int tl = warp; tl < my_tiles; tl += NW) {
      const int64_t v0 = (int64_t)(tile_lo + tl) * TILE + lane * E;
      const uint4 w = load_vec<LT>(row, v0, V, vec_z);
      float qv[E];
#pragma unroll
      for (int i = 0; i < E; ++i) qv[i] = 0.0f;
      if (residual) {
#pragma unroll
        for (int i = 0; i < E; i += 4) {
          const float4 q4 = load_q4(qrow, v0 + i, V, vec_q);
#pragma unroll
          for (int j = 0; j < 4; ++j) qv[i + j] = q4_elem(q4, j);
        }
      }
      ff part = {0.0f, 0.0f};
#pragma unroll
      for (int i = 0; i < E; ++i) part = ff_add(part, draw_weight(vec_elem<LT>(w, i), m, residual, qv[i], Zff, s_th, s_tl));
      s_part[tl * 32 + lane] = part;
      my_total = ff_add(my_total, part);
    }
    const float4 t = cluster_sum(cta_sum(my_total, 0.0f));  // also leaves every CTA's total in s_all
    S = ff{t.x, t.y};
    if (residual && !(S.hi > 0.0f)) {
      residual = false;  // the residual has no mass (only through rounding): draw from p_L instead
      continue;
    }
    break;
  }

  // which CTA holds the crossing of u * S?  (every CTA computes the same answer)
  if (tid == 0) {
    const ff thr = ff_mul_f(S, __ldg(p.sample_u + r));
    ff run = {0.0f, 0.0f};
    int owner = -1, last_pos = -1;
    ff local = thr;
    for (int c = 0; c < C; ++c) {
      const ff nxt = ff_add(run, s_all[c]);
      if (s_all[c].hi > 0.0f) last_pos = c;
      if (owner < 0 && ff_gt(nxt, thr)) {
        owner = c;
        local = ff_add(thr, ff_neg(run));
      }
      run = nxt;
    }
    s_b.flag = owner >= 0 ? owner : last_pos;
    s_b.aux = owner >= 0 ? 0 : 1;  // 1: no crossing (u >= 1, or rounding): the last element with mass
    s_b.Z = local;
    s_sel_entry = -1;
    s_sel_last = 0;
  }
  cluster.sync();  // orders s_b / s_sel_* for the CTA as well
  const int owner = s_b.flag;
  const ff thr = s_b.Z;
  if (rank == owner) {
    const int n_entries = my_tiles * 32;
    const int ept = (n_entries + NT - 1) / NT;
    const int e_lo = min(n_entries, tid * ept), e_hi = min(n_entries, e_lo + ept);
    if (s_b.aux == 0) {
      ff tot = {0.0f, 0.0f};
      for (int e = e_lo; e < e_hi; ++e) tot = ff_add(tot, s_part[e]);
      // inclusive / exclusive block scan of the per-thread totals (entries in token order)
      ff incl = tot;
      for (int d = 1; d < 32; d <<= 1) {
        const ff o = ff_shfl_up(incl, d);
        if (lane >= d) incl = ff_add(incl, o);
      }
      if (lane == 31) s_red[warp] = make_float4(incl.hi, incl.lo, 0.f, 0.f);
      __syncthreads();
      ff wbase = {0.0f, 0.0f};
      for (int w = 0; w < warp; ++w) wbase = ff_add(wbase, ff{s_red[w].x, s_red[w].y});
      incl = ff_add(wbase, incl);
      ff excl = ff_shfl_up(incl, 1);
      if (lane == 0) excl = wbase;
      if (ff_gt(incl, thr) && (tid == 0 || !ff_gt(excl, thr))) {
        ff run = excl;
        int entry = -1;
        bool hit = false;
        for (int e = e_lo; e < e_hi; ++e) {
          const ff nxt = ff_add(run, s_part[e]);
          if (ff_gt(nxt, thr)) {
            entry = e;
            hit = true;
            break;
          }
          if (s_part[e].hi > 0.0f) entry = e;
          run = nxt;
        }
        s_sel_entry = entry;
        s_sel_before = run;
        s_sel_last = hit ? 0 : 1;
      }
      __syncthreads();
    }
    const int sel0 = s_sel_entry;
    __syncthreads();
    if (sel0 < 0) {
      // no crossing inside this CTA (caller's u >= 1, or rounding): last entry with mass
      for (int e = e_hi - 1; e >= e_lo; --e) {
        if (s_part[e].hi > 0.0f) {
          atomicMax(&s_sel_entry, e);
          break;
        }
      }
      if (tid == 0) s_sel_last = 1;
      __syncthreads();
    }
    if (tid == 0) {
      int tok = -1;
      const int entry = s_sel_entry;
      if (entry >= 0) {
        // element scan of the entry, accumulating in the same order as the sweep
        const int tl = entry >> 5, ln = entry & 31;
        const int64_t v0 = (int64_t)(tile_lo + tl) * TILE + ln * E;
        const ff rem = ff_add(thr, ff_neg(s_sel_before));
        ff acc = {0.0f, 0.0f};
        int last = -1;
        for (int i = 0; i < E; ++i) {
          const int64_t v = v0 + i;
          if (v >= V) break;
          const ff w = draw_weight(load_scalar(row, v), m, residual, residual ? __ldg(qrow + v) : 0.0f, Zff,
                                   s_th, s_tl);
          if (w.hi > 0.0f) last = (int)v;
          acc = ff_add(acc, w);
          if (!s_sel_last && ff_gt(acc, rem)) {
            tok = (int)v;
            break;
          }
        }
        if (tok < 0) tok = last;
      }
      p.next_token[r] = tok;
    }
  }
  if (rank == 0 && tid == 0) {
    p.accepted_len[r] = L;
    if (owner < 0) p.next_token[r] = -1;  // no element with mass: cannot happen for finite rows
  }
  cluster.sync();  // no CTA leaves while another may still read its shared memory
}

namespace {

constexpr int kSmallNW = 2, kSmallMaxT = 8;    // 16 tiles
constexpr int kLargeNW = 16, kLargeMaxT = 16;  // 256 tiles per CTA
static_assert(kSmallNW * kSmallMaxT == kSmallTiles, "small shape");
static_assert(kLargeNW * kLargeMaxT == kLargeTilesPerCta, "large shape");

template <int NW, int MAXT>
constexpr size_t smem_bytes() { return (size_t)MAXT * NW * 32 * sizeof(ff); }

template <typename LT, int NW, int MAXT>
cudaError_t set_attr() {
  return cudaFuncSetAttribute(accept_kernel<LT, NW, MAXT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)smem_bytes<NW, MAXT>());
}

template <typename LT, int NW, int MAXT>
cudaError_t launch_shape(const AcceptParams &ap, cudaStream_t s) {
  cudaLaunchConfig_t cfg;
  memset(&cfg, 0, sizeof cfg);
  cfg.gridDim = dim3((unsigned)((int64_t)ap.B * ap.cluster));
  cfg.blockDim = dim3(NW * 32);
  cfg.dynamicSmemBytes = smem_bytes<NW, MAXT>();
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)ap.cluster;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, accept_kernel<LT, NW, MAXT>, ap);
}

}  // namespace

cudaError_t accept_setup() {
  cudaError_t e = set_attr<float, kSmallNW, kSmallMaxT>();
  if (e == cudaSuccess) e = set_attr<float, kLargeNW, kLargeMaxT>();
  if (e == cudaSuccess) e = set_attr<uint16_t, kSmallNW, kSmallMaxT>();
  if (e == cudaSuccess) e = set_attr<uint16_t, kLargeNW, kLargeMaxT>();
  return e;
}

cudaError_t accept_launch(const AcceptParams &p, bool bf16, bool large, cudaStream_t s) {
  if (large) {
    return bf16 ? launch_shape<uint16_t, kLargeNW, kLargeMaxT>(p, s) : launch_shape<float, kLargeNW, kLargeMaxT>(p, s);
  }
  return bf16 ? launch_shape<uint16_t, kSmallNW, kSmallMaxT>(p, s) : launch_shape<float, kSmallNW, kSmallMaxT>(p, s);
}

}  // namespace wisp
