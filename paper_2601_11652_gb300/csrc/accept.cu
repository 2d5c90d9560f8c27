// accept.cu -- the in-order speculative acceptance pass over the vocabulary (Eq. 1-3).
//
// One thread-block cluster of C CTAs (C = 1..8, chosen from the batch size) serves one
// request; CTA c owns a contiguous slice of every logit row, streamed as 16-byte vectors.
//
// Walk (Eq. 1-2): for logit rows i = 0, 1, ... of the request (row i scores draft token
// i+1; row k is the bonus row):
//   * one streaming pass gives each thread a running max and a double-float running sum
//     of exp(z - max) (fp32 terms, pairwise within a vector); threads, then CTAs (through
//     distributed shared memory, in rank order so every CTA holds bit-identical values)
//     combine them.  Alongside, a certified bound on the relative error of the normaliser
//     Z is accumulated (fp32 exp error, rounding of z - m, every rescale, pairwise sums);
//   * the decision u_i <= min(1, p(y)/q(y)) is taken in fp32 when u_i lies outside the
//     certified interval of the ratio; otherwise Z and p(y) are recomputed in double-float
//     arithmetic (Tang's table-driven exp) and the decision is taken on those;
//   * the walk stops at the first rejection, so later rows are never read.
// Draw (Eq. 3): from max(0, p_L - q_{L+1}) after a rejection, else from p_L, by inverse
// CDF in ascending token order: one double-float sweep of the row gives per-(round, warp)
// tile sums in shared memory and per-CTA totals; the CTA holding the crossing of
// u * total scans its tiles, then one warp scans the tile, then one lane its elements.
#include <cooperative_groups.h>
#include <cstring>

#include "accept.cuh"

namespace cg = cooperative_groups;

namespace wisp {

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

__device__ __forceinline__ void prefetch_l2(const void *p, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
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
  const float f = expf(st.m - mnew);
  const float d = mnew - st.m;
  st.s = ff_mul_f(st.s, f);
  st.A = fmaf(st.A, f, d * st.s.hi);
  st.m = mnew;
  st.nres += 1;
}

template <typename LT>
__device__ __forceinline__ void stats_add_vec(RowStats &st, const uint4 &w) {
  constexpr int E = LTraits<LT>::E;
  float z[E];
  float vm = -INFINITY;
#pragma unroll
  for (int i = 0; i < E; ++i) {
    z[i] = vec_elem<LT>(w, i);
    vm = fmaxf(vm, z[i]);
  }
  if (vm == -INFINITY) return;  // nothing but padding (or -inf logits)
  if (st.m == -INFINITY) st.mfirst = vm;
  stats_rebase(st, vm);
  float e[E];
#pragma unroll
  for (int i = 0; i < E; ++i) {
    const float x = z[i] - st.m;
    e[i] = expf(x);
    st.A = fmaf(e[i], fminf(-x, 104.0f), st.A);
  }
#pragma unroll
  for (int w2 = 1; w2 < E; w2 <<= 1) {
#pragma unroll
    for (int i = 0; i < E; i += 2 * w2) e[i] += e[i + w2];
  }
  st.s = ff_add_f(st.s, e[0]);
}

// Combine `o` into `st` (both may be empty).
__device__ __forceinline__ void stats_merge(RowStats &st, const RowStats &o) {
  if (o.m == -INFINITY) return;
  RowStats b = o;
  const float mm = fmaxf(st.m, b.m);
  stats_rebase(st, mm);
  stats_rebase(b, mm);
  st.s = ff_add(st.s, b.s);
  st.A += b.A;
  st.nres = max(st.nres, b.nres);
  st.mfirst = fminf(st.mfirst, b.mfirst);
}

struct Decide {
  int flag;  // 0 accept, 1 reject, 2 uncertain, 4 bad prob
  float zy, qy, u;
};

}  // namespace

template <typename LT>
__global__ void __launch_bounds__(NT) accept_kernel(const __grid_constant__ AcceptParams p) {
  constexpr int E = LTraits<LT>::E;
  extern __shared__ ff s_tile[];  // [rounds * NW] per-(round, warp) draw sums
  __shared__ float s_th[256], s_tl[256];
  __shared__ RowStats s_wst[NW];
  __shared__ RowStats s_pub[2];   // this CTA's published statistics (ring of 2)
  __shared__ ff s_tot[8];
  __shared__ RowStats s_row;      // combined statistics of the current row
  __shared__ float s_zy[kPreload], s_qy[kPreload], s_u[kPreload];
  __shared__ Decide s_dec;
  __shared__ int s_bad;
  __shared__ int s_owner, s_take_last;
  __shared__ ff s_thr;

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

  // ---- reductions -----------------------------------------------------------
  // CTA-wide merge of per-thread statistics (max first, then every thread rebases to it and
  // the sums are tree-reduced), then the cluster-wide merge: lane q of warp 0 reads CTA q's
  // published statistics and the same max / rebase / tree-sum runs across those lanes, so
  // every CTA ends with bit-identical values.
  auto cluster_stats = [&](RowStats st) -> RowStats {
    float wm = st.m, wf = st.mfirst;
    int wn = st.nres;
    for (int o = 16; o > 0; o >>= 1) {
      wm = fmaxf(wm, __shfl_xor_sync(0xffffffffu, wm, o));
      wf = fminf(wf, __shfl_xor_sync(0xffffffffu, wf, o));
      wn = max(wn, __shfl_xor_sync(0xffffffffu, wn, o));
    }
    if (lane == 0) {
      s_wst[warp].m = wm;
      s_wst[warp].mfirst = wf;
      s_wst[warp].nres = wn;
    }
    __syncthreads();
    float cm = -INFINITY, cf = INFINITY;
    int cn = 0;
    for (int w = 0; w < NW; ++w) {
      cm = fmaxf(cm, s_wst[w].m);
      cf = fminf(cf, s_wst[w].mfirst);
      cn = max(cn, s_wst[w].nres);
    }
    if (cm > -INFINITY) stats_rebase(st, cm);
    ff ws = st.s;
    float wa = st.A;
    for (int o = 16; o > 0; o >>= 1) {
      ws = ff_add(ws, ff_shfl_xor(ws, o));
      wa += __shfl_xor_sync(0xffffffffu, wa, o);
    }
    __syncthreads();  // everyone has read s_wst[*].m
    if (lane == 0) {
      s_wst[warp].s = ws;
      s_wst[warp].A = wa;
    }
    __syncthreads();
    if (tid == 0) {
      RowStats c;
      c.m = cm;
      c.mfirst = cf;
      c.nres = cn + 1;  // the thread-to-CTA rebase
      c.s = {0.0f, 0.0f};
      c.A = 0.0f;
      for (int w = 0; w < NW; ++w) {
        c.s = ff_add(c.s, s_wst[w].s);
        c.A += s_wst[w].A;
      }
      s_pub[xslot] = c;
    }
    cluster.sync();
    if (warp == 0) {
      RowStats q;
      stats_init(q);
      if (lane < C) q = *cluster.map_shared_rank(&s_pub[xslot], lane);
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
      if (lane == 0) {
        s_row.m = gm;
        s_row.s = gs;
        s_row.A = ga;
        s_row.nres = gn;  // + the CTA-to-cluster rebase, counted in the bound
        s_row.mfirst = gf;
      }
    }
    __syncthreads();
    xslot ^= 1;
    return s_row;
  };
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
  // double-float normaliser of a row (re-streamed); m is the row's exact max
  auto row_Zff = [&](const LT *row, float m) -> ff {
    ff acc = {0.0f, 0.0f};
    for (int64_t vi = vlo + tid; vi < vhi; vi += NT) {
      const uint4 w = load_vec<LT>(row, vi, V, vec_z);
#pragma unroll
      for (int i = 0; i < E; ++i) {
        const ff x = ff_two_sum(vec_elem<LT>(w, i), -m);
        acc = ff_add(acc, ff_exp_nonpos(x.hi, x.lo, s_th, s_tl));
      }
    }
    return cluster_total(acc);
  };

  // ---- the in-order walk (Eq. 1-2) -------------------------------------------
  int L = k;
  int err = s_bad ? WISP_DEV_BAD_TOKEN : 0;
  float m = 0.0f;
  ff Zff = {0.0f, 0.0f};
  bool have_Zff = false;
  for (int i = 0; i <= k && !err; ++i) {
    const LT *row = logits + (Q0 + i) * (int64_t)V;
    if (p.prefetch && i < k && tid == 0 && vhi > vlo) {
      const LT *nrow = row + V;
      const uint64_t a0 = reinterpret_cast<uint64_t>(nrow + vlo * E) & ~uint64_t(15);
      const uint64_t a1 = reinterpret_cast<uint64_t>(nrow + min((int64_t)V, vhi * E)) & ~uint64_t(15);
      for (uint64_t a = a0; a < a1; a += 32768) {
        const uint64_t n = a1 - a < 32768 ? a1 - a : 32768;
        prefetch_l2(reinterpret_cast<const void *>(a), (uint32_t)n);
      }
    }
    RowStats st;
    stats_init(st);
    for (int64_t base = vlo + tid; base < vhi; base += 4 * NT) {
      uint4 w[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int64_t vi = base + u * NT;
        const uint32_t ni = LTraits<LT>::NEG_INF2;
        w[u] = vi < vhi ? load_vec<LT>(row, vi, V, vec_z) : make_uint4(ni, ni, ni, ni);
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) stats_add_vec<LT>(st, w[u]);
    }
    const RowStats rs = cluster_stats(st);
    m = rs.m;
    const ff Z = rs.s;
    have_Zff = false;
    if (!(m > -INFINITY) || !(m < INFINITY) || !(Z.hi > 0.0f) || !(Z.hi < INFINITY) || !(rs.A >= 0.0f)) {
      err = WISP_DEV_BAD_PROB;
      break;
    }
    if (i == k) break;  // bonus row reached: every draft token accepted

    // Eq. 1, taken identically by thread 0 of every CTA
    if (tid == 0) {
      Decide d;
      if (i < kPreload) {
        d.zy = s_zy[i];
        d.qy = s_qy[i];
        d.u = s_u[i];
      } else {
        const int32_t y = __ldg(p.draft_tokens + D0 + i);
        d.zy = load_scalar(row, y);
        d.qy = __ldg(p.draft_probs + (D0 + i) * (int64_t)V + y);
        d.u = __ldg(p.accept_u + D0 + i);
      }
      if (!(d.qy >= 0.0f)) {
        d.flag = 4;
      } else if (d.qy == 0.0f) {
        d.flag = 0;  // a = 1
      } else {
        // certified relative error of Z (see RowStats) and of the ratio p(y)/q(y)
        const float x = d.zy - m;
        const float dz = 1.05f * ((float)(rs.nres + 2) * 0x1p-22f + 0x1p-24f * (m - rs.mfirst) +
                                  0x1p-24f * (rs.A / Z.hi) + 4.0f * 0x1p-24f) +
                         1e-12f;
        const float dr = dz + 1.05f * (0x1p-22f + 0x1p-24f * fabsf(x) + 4.0f * 0x1p-24f);
        const float ratio = expf(x) / (Z.hi * d.qy);
        const float lo = fminf(1.0f, ratio * (1.0f - dr)), hi = fminf(1.0f, ratio * (1.0f + dr));
        d.flag = d.u <= lo ? 0 : (d.u > hi ? 1 : 2);
      }
      s_dec = d;
    }
    __syncthreads();
    Decide d = s_dec;
    if (d.flag == 4) {
      err = WISP_DEV_BAD_PROB;
      break;
    }
    if (d.flag == 2) {
      // inside the certified interval: decide with the double-float normaliser
      Zff = row_Zff(row, m);
      have_Zff = true;
      if (tid == 0) {
        const ff x = ff_two_sum(d.zy, -m);
        const ff e = ff_exp_nonpos(x.hi, x.lo, s_th, s_tl);
        const double ratio = ff_to_double(e) / (ff_to_double(Zff) * (double)d.qy);
        s_dec.flag = (double)d.u <= fmin(1.0, ratio) ? 0 : 1;
      }
      __syncthreads();
      d.flag = s_dec.flag;
    }
    __syncthreads();
    if (d.flag == 1) {
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

  // ---- the extra token (Eq. 3) --------------------------------------------------
  const LT *row = logits + (Q0 + L) * (int64_t)V;
  const float *qrow = p.draft_probs + (D0 + L) * (int64_t)V;
  bool residual = L < k;
  if (residual && !have_Zff) Zff = row_Zff(row, m);
  ff S = {0.0f, 0.0f};
  for (;;) {
    ff run = {0.0f, 0.0f};
    for (int rd = 0; rd < rounds; ++rd) {
      const int64_t vi = vlo + (int64_t)rd * NT + tid;
      ff part = {0.0f, 0.0f};
      if (vi < vhi) {
        const uint4 w = load_vec<LT>(row, vi, V, vec_z);
        float q[E];
        if (residual) {
          load_q<E>(qrow, vi * E, V, vec_q, q);
        } else {
#pragma unroll
          for (int i = 0; i < E; ++i) q[i] = 0.0f;
        }
#pragma unroll
        for (int i = 0; i < E; ++i)
          part = ff_add(part, draw_weight(vec_elem<LT>(w, i), m, residual, q[i], Zff, s_th, s_tl));
      }
      for (int o = 16; o > 0; o >>= 1) part = ff_add(part, ff_shfl_xor(part, o));
      if (lane == 0) s_tile[rd * NW + warp] = part;
      run = ff_add(run, part);
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
          wts[i] = draw_weight(vec_elem<LT>(w, i), m, residual, q[i], Zff, s_th, s_tl);
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

// ---------------------------------------------------------------------------- host side
namespace {

template <typename LT>
cudaError_t set_attr() {
  return cudaFuncSetAttribute(accept_kernel<LT>, cudaFuncAttributeMaxDynamicSharedMemorySize, 96 * 1024);
}

template <typename LT>
cudaError_t launch_t(const AcceptParams &ap, cudaStream_t s) {
  const int rounds = (ap.vpc + NT - 1) / NT;
  cudaLaunchConfig_t cfg;
  memset(&cfg, 0, sizeof cfg);
  cfg.gridDim = dim3((unsigned)((int64_t)ap.B * ap.cluster));
  cfg.blockDim = dim3(NT);
  cfg.dynamicSmemBytes = (size_t)rounds * NW * sizeof(ff);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)ap.cluster;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, accept_kernel<LT>, ap);
}

}  // namespace

cudaError_t accept_setup() {
  cudaError_t e = set_attr<float>();
  if (e == cudaSuccess) e = set_attr<uint16_t>();
  return e;
}

cudaError_t accept_launch(const AcceptParams &p, bool bf16, cudaStream_t s) {
  return bf16 ? launch_t<uint16_t>(p, s) : launch_t<float>(p, s);
}

}  // namespace wisp
