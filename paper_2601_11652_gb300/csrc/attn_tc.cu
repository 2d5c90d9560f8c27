// attn_tc.cu -- tensor-core paged GQA attention for the verification forward (bf16 KV).
//
// Same contract as attn_simt.cu (Sec. 4.4-4.5: request r's k+1 new queries over its
// L_total = L_cached + L_new paged keys, query j seeing keys 0..c_r + j), built for sm_103a.
//
// Persistent CTAs (one per SM) take work items (request, KV head, key chunk) from a global
// counter.  Per CTA:
//   * warp 0 (producer) fetches the next item, publishes it to the other warps through a
//     4-slot shared ring, copies the item's query rows into shared memory (128-byte-swizzled
//     K-major layout), and streams K and V tiles of 64 tokens with TMA tiled loads: one
//     2 KB box per (16-token block, 64-wide half of the head dim), block ids from the block
//     table; blocks past the item are out-of-range boxes that read as zeros;
//   * warp 1 (one thread) issues tcgen05.mma: S = Q K^T (M = 128, N = 64, K = D) into a
//     double-buffered TMEM tile, and O += P V (M = 128, N = D, K = 64) into a TMEM
//     accumulator that lives across the whole item;
//   * warps 2-5 (softmax): the g*(k+1) query rows of an item are placed in a row group of
//     G = 32, 64 or 128 MMA rows and replicated 128/G times, so that each of the four TMEM
//     lane quadrants holds a copy; the warp of each quadrant then handles 64/rep of the 64
//     columns of every S tile.  The replicas of a row agree on a reference max through
//     shared memory each tile; the reference only moves when the tile max exceeds it by
//     more than 2^8 (then the O rows are rescaled in TMEM), so P = 2^(s - m_ref) <= 2^8.
//     Each warp writes its columns of P (bf16, swizzled) for the PV product and keeps its
//     share of the row sum; the item's epilogue adds the shares, reads O from TMEM and
//     writes the normalised output, or, for a split item, the (O, m, l) partials -- the
//     last chunk of a split (request, head) to finish merges all its chunks.
// Every mbarrier wait is bounded in time; an expired wait records WISP_DEV_TIMEOUT and the
// CTA drains.  Rows past g*(k+1) are padding: computed from stale data, never written.
#include "attn.cuh"
#include "sm100_ptx.cuh"

#include <cudaTypedefs.h>
#include <type_traits>

namespace wisp {

namespace {

constexpr int kBN = 64;             // KV tokens per tile
constexpr int kM = 128;             // MMA rows
constexpr int kThreads = 192;       // warp 0 producer, warp 1 MMA, warps 2-5 softmax
constexpr uint32_t kTmemCols = 256; // S[2] at columns 0 / 64, O at column 128
constexpr long long kWaitCycles = 4000000000LL;  // about two seconds: a wait that long is a failure
constexpr float kTau = 8.0f;        // lazy rescale threshold (log2 units)

template <int D>
struct Cfg {
  static constexpr int HALVES = D / 64;
  static constexpr int Q_BYTES = kM * D * 2;
  static constexpr int KV_TILE = kBN * D * 2;  // K (or V) of one tile
  static constexpr int NSTAGE = D == 128 ? 4 : 6;
  static constexpr int P_BYTES = kM * kBN * 2;
  static constexpr int RING = 4;               // slots of the item ring
  static constexpr int OFF_Q = 0;
  static constexpr int OFF_K = OFF_Q + 2 * Q_BYTES;
  static constexpr int OFF_V = OFF_K + NSTAGE * KV_TILE;
  static constexpr int OFF_P = OFF_V + NSTAGE * KV_TILE;
  static constexpr int OFF_BAR = OFF_P + 2 * P_BYTES;
  static constexpr int N_BAR = 2 * NSTAGE + 15 + 2 * RING;
  static constexpr int OFF_RED = OFF_BAR + N_BAR * 8;        // float [2][128] tile maxima, [128] row sums
  static constexpr int OFF_MISC = OFF_RED + 3 * 128 * 4;
  static constexpr int SMEM = OFF_MISC + 64 + 1024;          // + slack to align the base to 1024
};

constexpr uint32_t IDESC_S = ptx::idesc_bf16_f32(kM, kBN, false);

struct Bars {
  uint64_t *kv_full, *kv_empty, *q_full, *q_empty, *s_full, *s_empty, *p_full, *o_full, *o_empty, *mma_done;
  uint64_t *it_full, *it_empty, *grp;
};

__device__ __forceinline__ bool wait_bar(uint64_t *b, uint32_t parity, volatile int *abort) {
  if (ptx::mbar_try_wait(b, parity)) return true;
  const long long t0 = clock64();
  while (true) {
    if (ptx::mbar_try_wait(b, parity)) return true;
    if (*abort) return false;
    if (clock64() - t0 > kWaitCycles) {
      *abort = 1;
      return false;
    }
  }
}

__device__ __forceinline__ bool item_ok(const AttnParams &p, const WorkItem &w) {
  return w.r >= 0 && w.r < p.B && p.req_flag[w.r] == REQ_OK && w.t1 > w.t0 && w.rows > 0 && w.rows <= kM;
}

__device__ __forceinline__ int row_group(int rows) { return rows <= 32 ? 32 : (rows <= 64 ? 64 : 128); }

__device__ __forceinline__ uint32_t pack_bf16(float a, float b) {
  __nv_bfloat162 v = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t *>(&v);
}

}  // namespace

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    attn_tc_kernel(const __grid_constant__ AttnParams p, const __grid_constant__ CUtensorMap tmk,
                   const __grid_constant__ CUtensorMap tmv) {
  using C = Cfg<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t sbase = ptx::smem_u32(smem);
  uint64_t *bar = reinterpret_cast<uint64_t *>(smem + C::OFF_BAR);
  Bars B;
  B.kv_full = bar;
  B.kv_empty = bar + C::NSTAGE;
  B.q_full = bar + 2 * C::NSTAGE;
  B.q_empty = B.q_full + 2;
  B.s_full = B.q_empty + 2;
  B.s_empty = B.s_full + 2;
  B.p_full = B.s_empty + 2;
  B.o_full = B.p_full + 2;
  B.o_empty = B.o_full + 1;
  B.mma_done = B.o_empty + 1;
  B.it_full = B.mma_done + 1;
  B.it_empty = B.it_full + C::RING;
  B.grp = B.it_empty + C::RING;
  float *s_cmax = reinterpret_cast<float *>(smem + C::OFF_RED);  // [2][128]
  float *s_lsum = s_cmax + 2 * 128;                               // [128]
  uint32_t *s_tmem = reinterpret_cast<uint32_t *>(smem + C::OFF_MISC);
  volatile int *s_abort = reinterpret_cast<volatile int *>(smem + C::OFF_MISC + 4);
  volatile int *s_last = reinterpret_cast<volatile int *>(smem + C::OFF_MISC + 8);
  int *s_item = reinterpret_cast<int *>(smem + C::OFF_MISC + 16);  // [RING]

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < C::NSTAGE; ++s) {
      ptx::mbar_init(B.kv_full + s, 1);
      ptx::mbar_init(B.kv_empty + s, 1);
    }
    for (int b = 0; b < 2; ++b) {
      ptx::mbar_init(B.q_full + b, 1);
      ptx::mbar_init(B.q_empty + b, 1);
      ptx::mbar_init(B.s_full + b, 1);
      ptx::mbar_init(B.s_empty + b, 4);
      ptx::mbar_init(B.p_full + b, 4);
    }
    ptx::mbar_init(B.o_full, 1);
    ptx::mbar_init(B.o_empty, 4);
    ptx::mbar_init(B.mma_done, 1);
    for (int i = 0; i < C::RING; ++i) {
      ptx::mbar_init(B.it_full + i, 1);
      ptx::mbar_init(B.it_empty + i, 5);  // the MMA thread and the four softmax warps
    }
    ptx::mbar_init(B.grp, 4);  // the four softmax warps
    *s_abort = 0;
    ptx::fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    ptx::prefetch_tmap(&tmk);
    ptx::prefetch_tmap(&tmv);
  }
  if (warp == 1) {
    ptx::tmem_alloc(s_tmem, kTmemCols);
    ptx::tmem_relinquish();
  }
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem = *s_tmem;

  const int n_items = p.header->n_items;
  const int g = p.Hq / p.Hkv;

  if (warp == 0) {
    // ------------------------------------------------------------------ producer
    uint32_t tile_n = 0;
    int li = 0;
    bool ok = true;
    for (uint32_t j = 0; ok; ++j) {
      // fetch the next work item and publish it to the MMA thread and the softmax warps
      const int slot = j % C::RING;
      if (!wait_bar(B.it_empty + slot, ((j / C::RING) & 1) ^ 1, s_abort)) { ok = false; break; }
      int it = 0;
      if (lane == 0) {
        it = atomicAdd(&p.header_mut->next_item, 1);
        if (it >= n_items) it = -1;
        s_item[slot] = it;
        ptx::mbar_arrive(B.it_full + slot);
      }
      it = __shfl_sync(0xffffffffu, it, 0);
      if (it < 0) break;
      const WorkItem w = p.items[it];
      if (!item_ok(p, w)) continue;
      const int qb = li & 1;
      if (!wait_bar(B.q_empty + qb, ((li >> 1) & 1) ^ 1, s_abort)) { ok = false; break; }
      ++li;
      // query rows of this KV head -> Q[qb]: row rho = j*g + hh, copied to MMA rows rr*G + rho
      const int G = row_group(w.rows), rep = kM / G;
      const uint16_t *qg = static_cast<const uint16_t *>(p.q);
      uint8_t *qs = smem + C::OFF_Q + qb * C::Q_BYTES;
      constexpr int CPR = D / 8;  // 16-byte chunks per row
      for (int c = lane; c < w.rows * CPR; c += 32) {
        const int row = c / CPR, cc = c % CPR;
        const int jj = row / g, hh = row % g;
        const uint4 v = __ldg(reinterpret_cast<const uint4 *>(
                                  qg + ((int64_t)(w.q0 + jj) * p.Hq + w.h * g + hh) * D) + cc);
        for (int rr = 0; rr < rep; ++rr) {
          const int m = rr * G + row;
          *reinterpret_cast<uint4 *>(qs + (cc >> 3) * (kM * 128) + m * 128 + (((cc & 7) ^ (m & 7)) << 4)) = v;
        }
      }
      ptx::fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) ptx::mbar_arrive(B.q_full + qb);

      // K/V tiles
      const int32_t *bt = p.block_tables + (int64_t)w.r * p.max_blocks_per_seq + w.t0 / 16;
      const int nblk = (w.t1 - w.t0 + 15) / 16;
      auto fetch = [&](int base) -> int {
        const int i = base + lane;
        return i < nblk ? __ldg(bt + i) : -1;
      };
      int cur = fetch(0), nxt = fetch(32);
      const int ntiles = (w.t1 - w.t0 + kBN - 1) / kBN;
      for (int t = 0; t < ntiles; ++t, ++tile_n) {
        if (t > 0 && (t & 7) == 0) {
          cur = nxt;
          nxt = fetch(32 * ((t >> 3) + 1));
        }
        const int s = (int)(tile_n % C::NSTAGE);
        const uint32_t round = tile_n / C::NSTAGE;
        if (!wait_bar(B.kv_empty + s, (round & 1) ^ 1, s_abort)) { ok = false; break; }
        if (lane == 0) ptx::mbar_arrive_expect_tx(B.kv_full + s, 2 * C::KV_TILE);
        __syncwarp();
        int bid = __shfl_sync(0xffffffffu, cur, (4 * t + (lane & 3)) & 31);
        if (lane < 4) {
          const int rel = 4 * t + lane;
          if (rel >= nblk) {
            bid = p.num_blocks;  // past the item: the box is out of range and reads zeros
          } else if (bid < 0 || bid >= p.num_blocks) {
            report(p.status, WISP_DEV_BAD_BLOCK, p.request_ids, w.r);
            bid = p.num_blocks;
          }
#pragma unroll
          for (int hf = 0; hf < C::HALVES; ++hf) {
            const uint32_t off = s * C::KV_TILE + hf * (kBN * 128) + lane * (16 * 128);
            ptx::tma_load_4d(sbase + C::OFF_K + off, &tmk, B.kv_full + s, hf * 64, 0, w.h, bid);
            ptx::tma_load_4d(sbase + C::OFF_V + off, &tmv, B.kv_full + s, hf * 64, 0, w.h, bid);
          }
        }
      }
    }
    if (!ok && lane == 0) report(p.status, WISP_DEV_TIMEOUT, p.request_ids, 0);
    // drain: every stage issued must land before the CTA's shared memory goes away
    if (lane == 0) {
      for (uint32_t k = 0; k < (uint32_t)C::NSTAGE && k < tile_n; ++k) {
        const uint32_t n = tile_n - 1 - k;
        const long long t0 = clock64();
        while (!ptx::mbar_try_wait(B.kv_full + n % C::NSTAGE, (n / C::NSTAGE) & 1) && clock64() - t0 < kWaitCycles) {
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t IDESC_PV = ptx::idesc_bf16_f32(kM, D, true);
      uint32_t n = 0;
      int li = 0;
      bool ok = true;
      // O (+)= P V for global tile m; `first` = first tile of its item (overwrite O)
      auto issue_pv = [&](uint32_t m, bool first, int item_no) -> bool {
        const int pb = m & 1;
        if (!wait_bar(B.p_full + pb, (m >> 1) & 1, s_abort)) return false;
        if (first && !wait_bar(B.o_empty, (item_no & 1) ^ 1, s_abort)) return false;
        ptx::tc_fence_after();
        const int st = (int)(m % C::NSTAGE);
        const uint32_t pa = sbase + C::OFF_P + pb * C::P_BYTES;
        const uint32_t va = sbase + C::OFF_V + st * C::KV_TILE;
#pragma unroll
        for (int ks = 0; ks < kBN / 16; ++ks) {
          const uint64_t a = ptx::sdesc_sw128(pa + ks * 32, 16, 1024);
          const uint64_t b = ptx::sdesc_sw128(va + ks * 16 * 128, kBN * 128, 1024);
          ptx::umma_f16(tmem + 128, a, b, IDESC_PV, (!first || ks > 0) ? 1u : 0u);
        }
        ptx::umma_commit(B.o_full);
        ptx::umma_commit(B.kv_empty + st);
        return true;
      };
      for (uint32_t j = 0; ok; ++j) {
        const int slot = j % C::RING;
        if (!wait_bar(B.it_full + slot, (j / C::RING) & 1, s_abort)) { ok = false; break; }
        const int it = s_item[slot];
        ptx::mbar_arrive(B.it_empty + slot);
        if (it < 0) break;
        const WorkItem w = p.items[it];
        if (!item_ok(p, w)) continue;
        const int qb = li & 1;
        if (!wait_bar(B.q_full + qb, (li >> 1) & 1, s_abort)) { ok = false; break; }
        ptx::tc_fence_after();
        const uint32_t qa = sbase + C::OFF_Q + qb * C::Q_BYTES;
        const int ntiles = (w.t1 - w.t0 + kBN - 1) / kBN;
        for (int t = 0; t < ntiles && ok; ++t, ++n) {
          const int s = (int)(n % C::NSTAGE);
          if (!wait_bar(B.kv_full + s, (n / C::NSTAGE) & 1, s_abort)) { ok = false; break; }
          const int sb = n & 1;
          if (!wait_bar(B.s_empty + sb, ((n >> 1) & 1) ^ 1, s_abort)) { ok = false; break; }
          ptx::tc_fence_after();
          const uint32_t ka = sbase + C::OFF_K + s * C::KV_TILE;
#pragma unroll
          for (int ks = 0; ks < D / 16; ++ks) {
            const uint32_t koff = (ks >> 2) * (kBN * 128) + (ks & 3) * 32;
            const uint32_t qoff = (ks >> 2) * (kM * 128) + (ks & 3) * 32;
            ptx::umma_f16(tmem + sb * 64, ptx::sdesc_sw128(qa + qoff, 16, 1024), ptx::sdesc_sw128(ka + koff, 16, 1024),
                          IDESC_S, ks > 0);
          }
          ptx::umma_commit(B.s_full + sb);
          if (t == ntiles - 1) ptx::umma_commit(B.q_empty + qb);
          if (t > 0 && !issue_pv(n - 1, t == 1, li)) { ok = false; break; }
        }
        if (ok && !issue_pv(n - 1, ntiles == 1, li)) ok = false;
        ++li;
      }
      if (!ok) report(p.status, WISP_DEV_TIMEOUT, p.request_ids, 0);
      // every MMA this thread issued must finish before the TMEM is released
      ptx::umma_commit(B.mma_done);
      const long long t0 = clock64();
      while (!ptx::mbar_try_wait(B.mma_done, 0) && clock64() - t0 < kWaitCycles) {
      }
    }
  } else {
    // ------------------------------------------------------------------ softmax warps
    const int qd = warp & 3;          // TMEM lane quadrant of this warp
    const int mrow = qd * 32 + lane;  // this thread's MMA row
    const uint32_t lane_addr = (uint32_t)(qd * 32) << 16;
    const float scale_log2 = 1.4426950408889634f / sqrtf((float)D);
    uint32_t n = 0, gph = 0;
    bool ok = true;
    // barrier of the four softmax warps (an mbarrier, so that the wait is bounded)
    auto group_sync = [&]() -> bool {
      __syncwarp();
      if (lane == 0) ptx::mbar_arrive(B.grp);
      return wait_bar(B.grp, (gph++) & 1, s_abort);
    };
    for (uint32_t j = 0; ok; ++j) {
      const int slot = j % C::RING;
      if (!wait_bar(B.it_full + slot, (j / C::RING) & 1, s_abort)) { ok = false; break; }
      const int it = s_item[slot];
      __syncwarp();
      if (lane == 0) ptx::mbar_arrive(B.it_empty + slot);
      if (it < 0) break;
      const WorkItem w = p.items[it];
      if (!item_ok(p, w)) continue;
      const int G = row_group(w.rows), rep = kM / G;
      const int rid = (qd * 32) / G;      // replica handled by this warp
      const int row = mrow - rid * G;     // query row of this thread (j*g + hh)
      const bool owner = rid == 0;        // O rows live in the first G lanes
      const int cw = kBN / rep;           // columns of each S tile handled by this warp
      const int c0 = rid * cw;
      const int jq = row / g;
      const int vis = w.ctx + jq;         // last key position this row may see
      float m_ref = -INFINITY, l = 0.0f;

      const int ntiles = (w.t1 - w.t0 + kBN - 1) / kBN;
      // the tile loop, specialised for the CW columns of each S tile this warp handles
      auto run_tiles = [&](auto cw_tag) -> bool {
        constexpr int CW = decltype(cw_tag)::value;
        for (int t = 0; t < ntiles; ++t, ++n) {
          const int sb = n & 1;
          if (!wait_bar(B.s_full + sb, (n >> 1) & 1, s_abort)) return false;
          ptx::tc_fence_after();
          float sv[CW];
          const uint32_t saddr = tmem + lane_addr + sb * 64 + c0;
          if constexpr (CW == 16) {
            uint32_t x[16];
            ptx::tmem_ld16(saddr, x);
            ptx::tmem_wait_ld();
#pragma unroll
            for (int i = 0; i < 16; ++i) sv[i] = __uint_as_float(x[i]);
          } else {
#pragma unroll
            for (int h = 0; h < CW / 32; ++h) {
              uint32_t x[32];
              ptx::tmem_ld32(saddr + h * 32, x);
              ptx::tmem_wait_ld();
#pragma unroll
              for (int i = 0; i < 32; ++i) sv[h * 32 + i] = __uint_as_float(x[i]);
            }
          }
          ptx::tc_fence_before();
          __syncwarp();
          if (lane == 0) ptx::mbar_arrive(B.s_empty + sb);

          // mask, scale, this warp's share of the row max; replicas agree through shared memory
          const int tok0 = w.t0 + t * kBN + c0;
          float mx = -INFINITY;
#pragma unroll
          for (int i = 0; i < CW; ++i) {
            const int tok = tok0 + i;
            const bool valid = tok < w.t1 && tok <= vis;
            sv[i] = valid ? sv[i] * scale_log2 : -INFINITY;
            mx = fmaxf(mx, sv[i]);
          }
          float m_tile = mx;
          if constexpr (CW < kBN) {
            float *cmax = s_cmax + (n & 1) * 128;
            cmax[mrow] = mx;
            if (!group_sync()) return false;
#pragma unroll
            for (int rr = 0; rr < kBN / CW; ++rr) m_tile = fmaxf(m_tile, cmax[rr * G + row]);
          }
          float fac = 1.0f;
          bool rescale = false;
          if (m_ref == -INFINITY) {
            m_ref = m_tile;  // O holds nothing for this row yet
          } else if (m_tile > m_ref + kTau) {
            fac = ptx::ex2(m_ref - m_tile);
            rescale = true;
            m_ref = m_tile;
          }
          const float m_use = m_ref == -INFINITY ? 0.0f : m_ref;
          l *= fac;
          uint32_t pk[CW / 2];
#pragma unroll
          for (int i = 0; i < CW; i += 2) {
            const float e0 = ptx::ex2(sv[i] - m_use), e1 = ptx::ex2(sv[i + 1] - m_use);
            l += e0 + e1;
            pk[i / 2] = pack_bf16(e0, e1);
          }
          // Owners consume every PV completion in order: PV(n-1) is waited for at tile n, after
          // S(n) has landed (so PV(n-2) is complete) and before P(n) is published (so PV(n) cannot
          // have completed): the parity (n-1) & 1 always names that PV.  A rescale of the O rows
          // needs PV(n-1) complete and must precede PV(n).
          const bool need_pv = owner && t > 0;
          if (need_pv && __ballot_sync(0xffffffffu, rescale)) {
            if (!wait_bar(B.o_full, (n - 1) & 1, s_abort)) return false;
            ptx::tc_fence_after();
#pragma unroll
            for (int c = 0; c < D / 32; ++c) {
              uint32_t x[32];
              ptx::tmem_ld32(tmem + lane_addr + 128 + c * 32, x);
              ptx::tmem_wait_ld();
#pragma unroll
              for (int i = 0; i < 32; ++i) x[i] = __float_as_uint(__uint_as_float(x[i]) * fac);
              ptx::tmem_st32(tmem + lane_addr + 128 + c * 32, x);
            }
            ptx::tmem_wait_st();
            ptx::tc_fence_before();
          } else if (need_pv) {
            if (!wait_bar(B.o_full, (n - 1) & 1, s_abort)) return false;
          }
          // this warp's columns of P row `row` (bf16, 128-byte swizzle)
          uint8_t *prow = smem + C::OFF_P + sb * C::P_BYTES + row * 128;
#pragma unroll
          for (int c = 0; c < CW / 8; ++c) {
            const int cc = c0 / 8 + c;
            *reinterpret_cast<uint4 *>(prow + ((cc ^ (row & 7)) << 4)) =
                make_uint4(pk[4 * c], pk[4 * c + 1], pk[4 * c + 2], pk[4 * c + 3]);
          }
          ptx::fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) ptx::mbar_arrive(B.p_full + sb);
        }
        return true;
      };
      if (cw == 16) {
        ok = run_tiles(std::integral_constant<int, 16>{});
      } else if (cw == 32) {
        ok = run_tiles(std::integral_constant<int, 32>{});
      } else {
        ok = run_tiles(std::integral_constant<int, 64>{});
      }
      if (!ok) break;

      // ---- epilogue: row sum from the replicas, O from TMEM ----
      s_lsum[mrow] = l;
      if (owner) {
        if (!wait_bar(B.o_full, (n - 1) & 1, s_abort)) ok = false;  // PV of the item's last tile
        ptx::tc_fence_after();
      }
      if (!group_sync()) ok = false;
      if (!ok) break;
      float lt = 0.0f;
      for (int rr = 0; rr < rep; ++rr) lt += s_lsum[rr * G + row];
      const bool ract = owner && row < w.rows;
      const int hh = row % g;
      if (owner) {
#pragma unroll
        for (int c = 0; c < D / 32; ++c) {
          uint32_t x[32];
          ptx::tmem_ld32(tmem + lane_addr + 128 + c * 32, x);
          ptx::tmem_wait_ld();
          if (ract) {
            if (w.poff < 0) {
              const float inv = 1.0f / lt;
              uint16_t *og =
                  static_cast<uint16_t *>(p.out) + ((int64_t)(w.q0 + jq) * p.Hq + w.h * g + hh) * D + c * 32;
#pragma unroll
              for (int v = 0; v < 4; ++v) {
                uint4 o;
                o.x = pack_bf16(__uint_as_float(x[8 * v + 0]) * inv, __uint_as_float(x[8 * v + 1]) * inv);
                o.y = pack_bf16(__uint_as_float(x[8 * v + 2]) * inv, __uint_as_float(x[8 * v + 3]) * inv);
                o.z = pack_bf16(__uint_as_float(x[8 * v + 4]) * inv, __uint_as_float(x[8 * v + 5]) * inv);
                o.w = pack_bf16(__uint_as_float(x[8 * v + 6]) * inv, __uint_as_float(x[8 * v + 7]) * inv);
                reinterpret_cast<uint4 *>(og)[v] = o;
              }
            } else {
              float *part = p.partials + w.poff + (int64_t)row * D + c * 32;
#pragma unroll
              for (int v = 0; v < 8; ++v) {
                reinterpret_cast<float4 *>(part)[v] =
                    make_float4(__uint_as_float(x[4 * v]), __uint_as_float(x[4 * v + 1]),
                                __uint_as_float(x[4 * v + 2]), __uint_as_float(x[4 * v + 3]));
              }
            }
          }
        }
        if (ract && w.poff >= 0) {
          p.partials[w.poff + w.rows * D + row] = m_ref;
          p.partials[w.poff + w.rows * D + w.rows + row] = lt;
        }
      }
      ptx::tc_fence_before();
      __syncwarp();
      if (lane == 0) ptx::mbar_arrive(B.o_empty);

      // ---- split item: the last chunk of this (request, head) to finish merges all chunks ----
      if (w.poff >= 0) {
        __threadfence();
        if (!group_sync()) { ok = false; break; }
        if (threadIdx.x == 64) {
          const int chunks = p.req_chunks[w.r];
          const int done = atomicAdd(p.pair_done + (int64_t)w.r * p.Hkv + w.h, 1);
          *s_last = done == chunks - 1 ? chunks : 0;
          __threadfence();
        }
        if (!group_sync()) { ok = false; break; }
        const int chunks = *s_last;
        if (chunks > 0 && ract) {
          const WorkItem *ci = p.items + p.req_item_begin[w.r] + w.h * chunks;
          float mstar = -INFINITY;
          for (int c = 0; c < chunks; ++c)
            mstar = fmaxf(mstar, __ldcg(p.partials + ci[c].poff + w.rows * D + row));
          float den = 0.0f;
          float acc[D];
#pragma unroll
          for (int d = 0; d < D; ++d) acc[d] = 0.0f;
          for (int c = 0; c < chunks; ++c) {
            const float *part = p.partials + ci[c].poff;
            const float mc = __ldcg(part + w.rows * D + row);
            if (mc == -INFINITY) continue;
            const float wgt = ptx::ex2(mc - mstar);
            den = fmaf(__ldcg(part + w.rows * D + w.rows + row), wgt, den);
            const float4 *src = reinterpret_cast<const float4 *>(part + (int64_t)row * D);
#pragma unroll
            for (int v = 0; v < D / 4; ++v) {
              const float4 a = __ldcg(src + v);
              acc[4 * v] = fmaf(a.x, wgt, acc[4 * v]);
              acc[4 * v + 1] = fmaf(a.y, wgt, acc[4 * v + 1]);
              acc[4 * v + 2] = fmaf(a.z, wgt, acc[4 * v + 2]);
              acc[4 * v + 3] = fmaf(a.w, wgt, acc[4 * v + 3]);
            }
          }
          const float inv = 1.0f / den;
          uint16_t *og = static_cast<uint16_t *>(p.out) + ((int64_t)(w.q0 + jq) * p.Hq + w.h * g + hh) * D;
#pragma unroll
          for (int v = 0; v < D / 8; ++v) {
            uint4 o;
            o.x = pack_bf16(acc[8 * v + 0] * inv, acc[8 * v + 1] * inv);
            o.y = pack_bf16(acc[8 * v + 2] * inv, acc[8 * v + 3] * inv);
            o.z = pack_bf16(acc[8 * v + 4] * inv, acc[8 * v + 5] * inv);
            o.w = pack_bf16(acc[8 * v + 6] * inv, acc[8 * v + 7] * inv);
            reinterpret_cast<uint4 *>(og)[v] = o;
          }
        }
      }
    }
    if (!ok && lane == 0) report(p.status, WISP_DEV_TIMEOUT, p.request_ids, 0);
  }

  ptx::tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc(tmem, kTmemCols);
  }
}

// ---------------------------------------------------------------------------- host side
namespace {

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

cudaError_t get_encode() {
  if (g_encode) return cudaSuccess;
  void *fn = nullptr;
  cudaDriverEntryPointQueryResult q;
  cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
  if (e != cudaSuccess || q != cudaDriverEntryPointSuccess || !fn) return cudaErrorNotSupported;
  g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  return cudaSuccess;
}

// The paged pool [num_blocks, Hkv, 16, D] bf16 as a 4-D tensor (d, slot, head, block);
// one box = 64 head-dim elements (128 bytes, swizzled) x 16 slots of one block and head.
cudaError_t encode_pool(CUtensorMap *map, const void *base, int D, int Hkv, int num_blocks) {
  const cuuint64_t dims[4] = {(cuuint64_t)D, 16, (cuuint64_t)Hkv, (cuuint64_t)num_blocks};
  const cuuint64_t strides[3] = {(cuuint64_t)D * 2, (cuuint64_t)16 * D * 2, (cuuint64_t)Hkv * 16 * D * 2};
  const cuuint32_t box[4] = {64, 16, 1, 1};
  const cuuint32_t estr[4] = {1, 1, 1, 1};
  const CUresult r = g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void *>(base), dims, strides, box,
                              estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

}  // namespace

cudaError_t attn_tc_setup() {
  cudaError_t e = get_encode();
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(attn_tc_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg<128>::SMEM);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(attn_tc_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg<64>::SMEM);
  return e;
}

cudaError_t attn_tc_launch(const AttnParams &p, int grid, cudaStream_t s) {
  alignas(64) CUtensorMap tk, tv;
  cudaError_t e = encode_pool(&tk, p.k_cache, p.D, p.Hkv, p.num_blocks);
  if (e == cudaSuccess) e = encode_pool(&tv, p.v_cache, p.D, p.Hkv, p.num_blocks);
  if (e != cudaSuccess) return e;
  if (p.D == 128) {
    attn_tc_kernel<128><<<grid, kThreads, Cfg<128>::SMEM, s>>>(p, tk, tv);
  } else {
    attn_tc_kernel<64><<<grid, kThreads, Cfg<64>::SMEM, s>>>(p, tk, tv);
  }
  return cudaGetLastError();
}

}  // namespace wisp
