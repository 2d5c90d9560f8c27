// attn_tc.cu -- tensor-core paged GQA attention for the verification forward (bf16 KV).
//
// Same contract as attn_simt.cu (Sec. 4.4-4.5: request r's k+1 new queries over its
// L_total = L_cached + L_new paged keys, query j seeing keys 0..c_r + j), built for sm_103a.
//
// Persistent CTAs (one per SM) take work items (request, KV head, key chunk) from a global
// counter, in the planner's longest-first order.  Warp roles in a CTA:
//   * warp 6 (item loader) takes the next item, publishes it to the other warps through a
//     4-slot shared ring, and copies its query rows into one of two shared Q buffers
//     (128-byte-swizzled K-major layout);
//   * warps 0 and 7 (K and V producers) stream the item's K and V tiles of 64 tokens with TMA
//     tiled loads into two separate rings, one 8 KB box per 64-wide half of the head dim when
//     the tile's four 16-token blocks are consecutive in the pool, else one 2 KB box per block;
//     blocks past the item read as zeros (out-of-range box).  A K stage is free again once S of
//     its tile is done, a V stage once PV is;
//   * warp 1 (one thread) issues tcgen05.mma: S = Q K^T (M = 128, N = 64, K = D) into one of two
//     TMEM tiles, and O += P V (M = 128, N = D, K = 64) into the item's TMEM accumulator (two
//     accumulators, alternating between items);
//   * warps 2-5 (softmax): the g*(k+1) query rows of an item are placed in a row group of
//     G = 32, 64 or 128 MMA rows and replicated 128/G times, so that each of the four TMEM lane
//     quadrants holds a copy.  Each warp reads the whole 64-column S row of its lane (so the
//     replicas agree on the row max without talking to each other) and handles 64/rep of the
//     columns: exponentials, its share of the row sum, and P (bf16, swizzled, written to every
//     replica row) for the PV product.  The reference max only moves when a tile max exceeds it
//     by more than 2^8 (then the warp rescales its slice of the O rows in TMEM), so
//     P = 2^(s - m_ref) <= 2^8.  At the item's end the row-sum share and the max go to spare
//     TMEM columns and the item is handed over;
//   * warps 8-11 (epilogue) add the row-sum shares, read O from TMEM and write the normalised
//     output or, for a split item, the (O, m, l) partials; the last chunk of a split
//     (request, head) to finish merges all its chunks.  This runs while the softmax warps are
//     already on the next item.
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
constexpr int kThreads = 384;       // warp 0 K producer, warp 1 MMA, warps 2-5 softmax, warp 6 item loader,
                                    // warp 7 V producer, warps 8-11 epilogue
constexpr uint32_t kTmemCols = 512; // S[2] at columns 0 / 64, O[2] at 128 / 256, (l, m) hand-over at 384
constexpr long long kWaitCycles = 4000000000LL;  // about two seconds: a wait that long is a failure
constexpr float kTau = 8.0f;        // lazy rescale threshold (log2 units)

template <int D>
struct Cfg {
  static constexpr int HALVES = D / 64;
  static constexpr int Q_BYTES = kM * D * 2;
  static constexpr int KV_TILE = kBN * D * 2;  // K (or V) of one tile
  static constexpr int NSTAGE = D == 128 ? 3 : 6;
  static constexpr int P_BYTES = kM * kBN * 2;
  static constexpr int RING = 4;               // slots of the item ring
  static constexpr int OFF_Q = 0;
  static constexpr int OFF_K = OFF_Q + 2 * Q_BYTES;
  static constexpr int OFF_V = OFF_K + NSTAGE * KV_TILE;
  static constexpr int OFF_P = OFF_V + NSTAGE * KV_TILE;
  static constexpr int NPBUF = 3;                // P buffers: P(n) in buffer n % 3
  static constexpr int OFF_BAR = OFF_P + NPBUF * P_BYTES;
  static constexpr int N_BAR = 4 * NSTAGE + 24 + 2 * RING;
  static constexpr int OFF_RED = OFF_BAR + N_BAR * 8;        // float [2][128] row sums (epilogue)
  static constexpr int OFF_MISC = OFF_RED + 2 * 128 * 4;     // tmem base, flags
  static constexpr int OFF_RING = OFF_MISC + 64;             // RING x (index, WorkItem)
  static constexpr int SMEM = OFF_RING + RING * 48 + 1024;   // + slack to align the base to 1024
  static_assert(SMEM <= 227 * 1024, "shared memory of one CTA on sm_103a");
};

constexpr uint32_t IDESC_S = ptx::idesc_bf16_f32(kM, kBN, false);

struct Bars {
  uint64_t *k_full, *k_empty, *v_full, *v_empty, *q_full, *q_empty, *s_full, *s_empty, *p_full, *o_full;
  uint64_t *o_empty, *o_done, *ep_full, *mma_done, *it_full, *it_empty, *egrp;
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
                   const __grid_constant__ CUtensorMap tmv, const __grid_constant__ CUtensorMap tmk4,
                   const __grid_constant__ CUtensorMap tmv4) {
  using C = Cfg<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t sbase = ptx::smem_u32(smem);
  uint64_t *bar = reinterpret_cast<uint64_t *>(smem + C::OFF_BAR);
  Bars B;
  B.k_full = bar;
  B.k_empty = bar + C::NSTAGE;
  B.v_full = bar + 2 * C::NSTAGE;
  B.v_empty = bar + 3 * C::NSTAGE;
  B.q_full = bar + 4 * C::NSTAGE;
  B.q_empty = B.q_full + 2;
  B.s_full = B.q_empty + 2;
  B.s_empty = B.s_full + 2;
  B.p_full = B.s_empty + 2;  // [3] per P buffer
  B.o_full = B.p_full + 3;  // [3] per P buffer: PV of tiles n with n % 3 == b
  B.o_empty = B.o_full + 3;  // [2] per O buffer: its epilogue is done
  B.o_done = B.o_empty + 2;  // [2] per O buffer: the item's last PV is done
  B.ep_full = B.o_done + 2;  // [2] per O buffer: the softmax warps handed the item over
  B.mma_done = B.ep_full + 2;
  B.it_full = B.mma_done + 1;
  B.it_empty = B.it_full + C::RING;
  B.egrp = B.it_empty + C::RING;
  float *s_lsum = reinterpret_cast<float *>(smem + C::OFF_RED);  // [2][128]
  uint32_t *s_tmem = reinterpret_cast<uint32_t *>(smem + C::OFF_MISC);
  volatile int *s_abort = reinterpret_cast<volatile int *>(smem + C::OFF_MISC + 4);
  volatile int *s_last = reinterpret_cast<volatile int *>(smem + C::OFF_MISC + 8);
  struct RingSlot {
    int it;
    int pad[3];
    WorkItem w;
  };
  RingSlot *s_ring = reinterpret_cast<RingSlot *>(smem + C::OFF_RING);
  static_assert(C::OFF_RING + C::RING * sizeof(RingSlot) + 1024 <= C::SMEM, "item ring overflows its region");

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < C::NSTAGE; ++s) {
      ptx::mbar_init(B.k_full + s, 1);
      ptx::mbar_init(B.k_empty + s, 1);
      ptx::mbar_init(B.v_full + s, 1);
      ptx::mbar_init(B.v_empty + s, 1);
    }
    for (int b = 0; b < 2; ++b) {
      ptx::mbar_init(B.q_full + b, 1);
      ptx::mbar_init(B.q_empty + b, 1);
      ptx::mbar_init(B.s_full + b, 1);
      ptx::mbar_init(B.s_empty + b, 4);
    }
    for (int b = 0; b < 3; ++b) {
      ptx::mbar_init(B.p_full + b, 4);
      ptx::mbar_init(B.o_full + b, 1);
    }
    for (int b = 0; b < 2; ++b) {
      ptx::mbar_init(B.o_empty + b, 4);  // the four epilogue warps
      ptx::mbar_init(B.o_done + b, 1);
      ptx::mbar_init(B.ep_full + b, 4);  // the four softmax warps
    }
    ptx::mbar_init(B.mma_done, 1);
    for (int i = 0; i < C::RING; ++i) {
      ptx::mbar_init(B.it_full + i, 1);
      ptx::mbar_init(B.it_empty + i, 11);  // KV producers, MMA thread, softmax and epilogue warps
    }
    ptx::mbar_init(B.egrp, 4);  // the four epilogue warps
    *s_abort = 0;
    ptx::fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    ptx::prefetch_tmap(&tmk);
    ptx::prefetch_tmap(&tmv);
    ptx::prefetch_tmap(&tmk4);
    ptx::prefetch_tmap(&tmv4);
  }
  __syncwarp();
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

  if (warp == 0 || warp == 7) {
    // ------------------------------------------------------------------ K / V producers
    // K and V have rings of their own: a K stage is free again once S of its tile is done, a V
    // stage once PV is, so each tensor is fetched about NSTAGE tiles ahead of its use.
    const bool is_k = warp == 0;
    const CUtensorMap *tm1 = is_k ? &tmk : &tmv;
    const CUtensorMap *tm4 = is_k ? &tmk4 : &tmv4;
    const uint32_t off_t = sbase + (is_k ? C::OFF_K : C::OFF_V);
    uint64_t *full = is_k ? B.k_full : B.v_full;
    uint64_t *empty = is_k ? B.k_empty : B.v_empty;
    uint32_t tile_n = 0;
    bool ok = true;
    for (uint32_t j = 0; ok; ++j) {
      const int slot = j % C::RING;
      if (!wait_bar(B.it_full + slot, (j / C::RING) & 1, s_abort)) { ok = false; break; }
      const int it = s_ring[slot].it;
      const WorkItem w = s_ring[slot].w;
      __syncwarp();
      if (lane == 0) ptx::mbar_arrive(B.it_empty + slot);
      if (it < 0) break;
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
        if (!wait_bar(empty + s, (round & 1) ^ 1, s_abort)) { ok = false; break; }
        if (lane == 0) ptx::mbar_arrive_expect_tx(full + s, C::KV_TILE);
        __syncwarp();
        int bid = __shfl_sync(0xffffffffu, cur, (4 * t + (lane & 3)) & 31);
        const int rel = 4 * t + (lane & 3);
        bool valid = rel < nblk && bid >= 0 && bid < p.num_blocks;
        if (is_k && lane < 4 && rel < nblk && !valid) report(p.status, WISP_DEV_BAD_BLOCK, p.request_ids, w.r);
        const int b0 = __shfl_sync(0xffffffffu, bid, 0);
        // four consecutive valid blocks: one 8 KB box per (tensor, half) with the 4-block maps
        const unsigned contig = __ballot_sync(0xffffffffu, lane < 4 && valid && bid == b0 + lane);
        if (contig == 0xFu) {
          if (lane == 0) {
#pragma unroll
            for (int hf = 0; hf < C::HALVES; ++hf) {
              ptx::tma_load_4d(off_t + s * C::KV_TILE + hf * (kBN * 128), tm4, full + s, hf * 64, 0, w.h, b0);
            }
          }
        } else if (lane < 4) {
          if (!valid) bid = p.num_blocks;  // past the item (or invalid): out-of-range box, reads zeros
#pragma unroll
          for (int hf = 0; hf < C::HALVES; ++hf) {
            const uint32_t off = s * C::KV_TILE + hf * (kBN * 128) + lane * (16 * 128);
            ptx::tma_load_4d(off_t + off, tm1, full + s, hf * 64, 0, w.h, bid);
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
        while (!ptx::mbar_try_wait(full + n % C::NSTAGE, (n / C::NSTAGE) & 1) && clock64() - t0 < kWaitCycles) {
        }
      }
    }
  } else if (warp == 6) {
    // ------------------------------------------------------------------ item loader
    int li = 0;
    bool ok = true;
    for (uint32_t j = 0; ok; ++j) {
      // next valid work item: publish it to the other warps, then load its query rows
      const int slot = j % C::RING;
      if (!wait_bar(B.it_empty + slot, ((j / C::RING) & 1) ^ 1, s_abort)) { ok = false; break; }
      int it = -1;
      if (lane == 0) {
        while (true) {
          it = atomicAdd(&p.header_mut->next_item, 1);
          if (it >= n_items) { it = -1; break; }
          it = p.order[it];
          if (item_ok(p, p.items[it])) break;
        }
        s_ring[slot].it = it;
        if (it >= 0) s_ring[slot].w = p.items[it];
        ptx::mbar_arrive(B.it_full + slot);
      }
      it = __shfl_sync(0xffffffffu, it, 0);
      if (it < 0) break;
      const WorkItem w = p.items[it];
      const int qb = li & 1;
      if (!wait_bar(B.q_empty + qb, ((li >> 1) & 1) ^ 1, s_abort)) { ok = false; break; }
      ++li;
      // query rows of this KV head -> Q[qb]: row rho = j*g + hh, copied to MMA rows rr*G + rho.
      // Loads are issued QBATCH at a time per lane before any store.
      const int G = row_group(w.rows), rep = kM / G;
      const uint16_t *qg = static_cast<const uint16_t *>(p.q);
      uint8_t *qs = smem + C::OFF_Q + qb * C::Q_BYTES;
      constexpr int CPR = D / 8;  // 16-byte chunks per row
      constexpr int QBATCH = 16;
      const int nchunks = w.rows * CPR;
      for (int base = 0; base < nchunks; base += 32 * QBATCH) {
        uint4 v[QBATCH];
#pragma unroll
        for (int u = 0; u < QBATCH; ++u) {
          const int c = base + u * 32 + lane;
          if (c < nchunks) {
            const int row = c / CPR, cc = c % CPR;
            const int jj = row / g, hh = row % g;
            v[u] = __ldg(reinterpret_cast<const uint4 *>(qg + ((int64_t)(w.q0 + jj) * p.Hq + w.h * g + hh) * D) + cc);
          }
        }
#pragma unroll
        for (int u = 0; u < QBATCH; ++u) {
          const int c = base + u * 32 + lane;
          if (c < nchunks) {
            const int row = c / CPR, cc = c % CPR;
            for (int rr = 0; rr < rep; ++rr) {
              const int m = rr * G + row;
              *reinterpret_cast<uint4 *>(qs + (cc >> 3) * (kM * 128) + m * 128 + (((cc & 7) ^ (m & 7)) << 4)) = v[u];
            }
          }
        }
      }
      ptx::fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) ptx::mbar_arrive(B.q_full + qb);
    }
    if (!ok && lane == 0) report(p.status, WISP_DEV_TIMEOUT, p.request_ids, 0);
  } else if (warp == 1) {
    // ------------------------------------------------------------------ MMA issuer
    // One thread polls two queues: S(n) is issued as soon as tile n has landed, its Q is loaded
    // and its TMEM buffer has been read; PV(m) as soon as P(m) is published (and, for an item's
    // first tile, the previous item's O has been read).  S therefore runs ahead of PV instead of
    // waiting behind it.
    if (lane == 0) {
      constexpr uint32_t IDESC_PV = ptx::idesc_bf16_f32(kM, D, true);
      uint32_t n_s = 0, n_pv = 0, j = 0;
      int li = 0, s_t = 0, s_nt = 0, s_qb = 0, s_li = 0;
      bool s_have = false, items_done = false, ok = true;
      uint8_t tflag[4];  // per issued S tile: bit 0 first tile of its item, bit 1 its last
      int tli[4];        // item number of the tile (o_empty parity)
      long long last = clock64();
      while (true) {
        bool prog = false;
        if (!s_have && !items_done) {
          const int slot = j % C::RING;
          if (ptx::mbar_test_wait(B.it_full + slot, (j / C::RING) & 1)) {
            const int it = s_ring[slot].it;
            const WorkItem w = s_ring[slot].w;
            ptx::mbar_arrive(B.it_empty + slot);
            ++j;
            if (it < 0) {
              items_done = true;
            } else {
              s_have = true;
              s_t = 0;
              s_nt = (w.t1 - w.t0 + kBN - 1) / kBN;
              s_qb = li & 1;
              s_li = li;
              ++li;
            }
            prog = true;
          }
        }
        if (s_have && n_s < n_pv + 4) {
          const int st = (int)(n_s % C::NSTAGE), sb = n_s & 1;
          if ((s_t > 0 || ptx::mbar_test_wait(B.q_full + s_qb, (s_li >> 1) & 1)) &&
              ptx::mbar_test_wait(B.k_full + st, (n_s / C::NSTAGE) & 1) &&
              ptx::mbar_test_wait(B.s_empty + sb, ((n_s >> 1) & 1) ^ 1)) {
            ptx::tc_fence_after();
            const uint32_t qa = sbase + C::OFF_Q + s_qb * C::Q_BYTES;
            const uint32_t ka = sbase + C::OFF_K + st * C::KV_TILE;
#pragma unroll
            for (int ks = 0; ks < D / 16; ++ks) {
              const uint32_t koff = (ks >> 2) * (kBN * 128) + (ks & 3) * 32;
              const uint32_t qoff = (ks >> 2) * (kM * 128) + (ks & 3) * 32;
              ptx::umma_f16(tmem + sb * 64, ptx::sdesc_sw128(qa + qoff, 16, 1024),
                            ptx::sdesc_sw128(ka + koff, 16, 1024), IDESC_S, ks > 0);
            }
            ptx::umma_commit(B.s_full + sb);
            ptx::umma_commit(B.k_empty + st);
            if (s_t == s_nt - 1) ptx::umma_commit(B.q_empty + s_qb);
            tflag[n_s & 3] = (s_t == 0 ? 1 : 0) | (s_t == s_nt - 1 ? 2 : 0);
            tli[n_s & 3] = s_li;
            ++n_s;
            if (++s_t == s_nt) s_have = false;
            prog = true;
          }
        }
        if (n_pv < n_s) {
          const int pb = (int)(n_pv % 3);
          const bool first = tflag[n_pv & 3] & 1, last = tflag[n_pv & 3] & 2;
          const int tl = tli[n_pv & 3], ob = tl & 1;  // the item's O buffer
          const int st = (int)(n_pv % C::NSTAGE);
          if (ptx::mbar_test_wait(B.p_full + pb, (n_pv / 3) & 1) &&
              ptx::mbar_test_wait(B.v_full + st, (n_pv / C::NSTAGE) & 1) &&
              (!first || ptx::mbar_test_wait(B.o_empty + ob, ((tl >> 1) & 1) ^ 1))) {
            ptx::tc_fence_after();
            const uint32_t pa = sbase + C::OFF_P + pb * C::P_BYTES;
            const uint32_t va = sbase + C::OFF_V + st * C::KV_TILE;
#pragma unroll
            for (int ks = 0; ks < kBN / 16; ++ks) {
              const uint64_t a = ptx::sdesc_sw128(pa + ks * 32, 16, 1024);
              const uint64_t b = ptx::sdesc_sw128(va + ks * 16 * 128, kBN * 128, 1024);
              ptx::umma_f16(tmem + 128 + ob * 128, a, b, IDESC_PV, (!first || ks > 0) ? 1u : 0u);
            }
            ptx::umma_commit(B.o_full + pb);
            ptx::umma_commit(B.v_empty + st);
            if (last) ptx::umma_commit(B.o_done + ob);
            ++n_pv;
            prog = true;
          }
        }
        if (items_done && !s_have && n_pv == n_s) break;
        if (prog) {
          last = clock64();
        } else {
          if (*s_abort) { ok = false; break; }
          if (clock64() - last > kWaitCycles) {
            *s_abort = 1;
            ok = false;
            break;
          }
          __nanosleep(20);
        }
      }
      if (!ok) report(p.status, WISP_DEV_TIMEOUT, p.request_ids, 0);
      // every MMA this thread issued must finish before the TMEM is released
      ptx::umma_commit(B.mma_done);
      const long long t0 = clock64();
      while (!ptx::mbar_try_wait(B.mma_done, 0) && clock64() - t0 < kWaitCycles) {
      }
    }
  } else if (warp >= 8) {
    // ------------------------------------------------------------------ epilogue warps
    // One warp per TMEM lane quadrant.  Item li's O (buffer li & 1) is read once the softmax warps
    // have handed the item over and its last PV is done; the output (or, for a split item, the
    // partial O, m, l) is written, the buffer released, and the last chunk of a split
    // (request, head) to finish merges all of its chunks.
    const int qd = warp & 3;
    const int mrow = qd * 32 + lane;
    const uint32_t lane_addr = (uint32_t)(qd * 32) << 16;
    uint32_t gph = 0;
    int li = 0;
    bool ok = true;
    // barrier of the four epilogue warps (an mbarrier, so that the wait is bounded)
    auto group_sync = [&]() -> bool {
      __syncwarp();
      if (lane == 0) ptx::mbar_arrive(B.egrp);
      return wait_bar(B.egrp, (gph++) & 1, s_abort);
    };
    for (uint32_t j = 0; ok; ++j) {
      const int slot = j % C::RING;
      if (!wait_bar(B.it_full + slot, (j / C::RING) & 1, s_abort)) { ok = false; break; }
      const int it = s_ring[slot].it;
      const WorkItem w = s_ring[slot].w;
      __syncwarp();
      if (lane == 0) ptx::mbar_arrive(B.it_empty + slot);
      if (it < 0) break;
      const int G = row_group(w.rows), rep = kM / G;
      const int rid = (qd * 32) / G;   // replica of this warp's rows
      const int row = mrow - rid * G;  // query row of this thread (j*g + hh)
      const int dcw = D / rep;         // this warp writes the output columns [d0, d0 + dcw)
      const int d0 = rid * dcw;
      const int jq = row / g;
      const int ob = li & 1;
      const uint32_t o_col = 128 + ob * 128;
      // the softmax warps' hand-over and the item's last PV
      if (!wait_bar(B.ep_full + ob, (li >> 1) & 1, s_abort)) { ok = false; break; }
      if (!wait_bar(B.o_done + ob, (li >> 1) & 1, s_abort)) { ok = false; break; }
      ++li;
      ptx::tc_fence_after();
      uint32_t lm[2];
      ptx::tmem_ld2(tmem + lane_addr + 384 + 2 * ob, lm);
      ptx::tmem_wait_ld();
      const float m_ref = __uint_as_float(lm[1]);
      // row sum: the shares of the row's replicas
      s_lsum[ob * 128 + mrow] = __uint_as_float(lm[0]);
      if (!group_sync()) { ok = false; break; }
      float lt = 0.0f;
      for (int rr = 0; rr < rep; ++rr) lt += s_lsum[ob * 128 + rr * G + row];
      const bool ract = row < w.rows;
      const int hh = row % g;
      const float inv = 1.0f / lt;
      for (int c = 0; c < dcw; c += 16) {
        uint32_t x[16];
        ptx::tmem_ld16(tmem + lane_addr + o_col + d0 + c, x);
        ptx::tmem_wait_ld();
        if (ract) {
          if (w.poff < 0) {
            uint16_t *og = static_cast<uint16_t *>(p.out) + ((int64_t)(w.q0 + jq) * p.Hq + w.h * g + hh) * D + d0 + c;
#pragma unroll
            for (int v = 0; v < 2; ++v) {
              uint4 o;
              o.x = pack_bf16(__uint_as_float(x[8 * v + 0]) * inv, __uint_as_float(x[8 * v + 1]) * inv);
              o.y = pack_bf16(__uint_as_float(x[8 * v + 2]) * inv, __uint_as_float(x[8 * v + 3]) * inv);
              o.z = pack_bf16(__uint_as_float(x[8 * v + 4]) * inv, __uint_as_float(x[8 * v + 5]) * inv);
              o.w = pack_bf16(__uint_as_float(x[8 * v + 6]) * inv, __uint_as_float(x[8 * v + 7]) * inv);
              reinterpret_cast<uint4 *>(og)[v] = o;
            }
          } else {
            float4 *part = reinterpret_cast<float4 *>(p.partials + w.poff + (int64_t)row * D + d0 + c);
#pragma unroll
            for (int v = 0; v < 4; ++v)
              part[v] = make_float4(__uint_as_float(x[4 * v]), __uint_as_float(x[4 * v + 1]),
                                    __uint_as_float(x[4 * v + 2]), __uint_as_float(x[4 * v + 3]));
          }
        }
      }
      if (ract && rid == 0 && w.poff >= 0) {
        p.partials[w.poff + w.rows * D + row] = m_ref;
        p.partials[w.poff + w.rows * D + w.rows + row] = lt;
      }
      ptx::tc_fence_before();
      __syncwarp();
      if (lane == 0) ptx::mbar_arrive(B.o_empty + ob);

      // ---- split item: the last chunk of this (request, head) to finish merges all chunks ----
      if (w.poff >= 0) {
        __threadfence();
        if (!group_sync()) { ok = false; break; }
        if (warp == 8 && lane == 0) {
          const int chunks = p.req_chunks[w.r];
          const int done = atomicAdd(p.pair_done + (int64_t)w.r * p.Hkv + w.h, 1);
          *s_last = done == chunks - 1 ? chunks : 0;
          __threadfence();
        }
        if (!group_sync()) { ok = false; break; }
        const int chunks = *s_last;
        if (chunks > 0 && ract) {
          // every warp merges its column slice of its rows
          const WorkItem *ci = p.items + p.req_item_begin[w.r] + w.h * chunks;
          float mstar = -INFINITY;
          for (int c = 0; c < chunks; ++c)
            mstar = fmaxf(mstar, __ldcg(p.partials + ci[c].poff + w.rows * D + row));
          float den = 0.0f;
          for (int c = 0; c < chunks; ++c) {
            const float *part = p.partials + ci[c].poff;
            const float mc = __ldcg(part + w.rows * D + row);
            if (mc != -INFINITY) den = fmaf(__ldcg(part + w.rows * D + w.rows + row), ptx::ex2(mc - mstar), den);
          }
          const float dinv = 1.0f / den;
          uint16_t *og = static_cast<uint16_t *>(p.out) + ((int64_t)(w.q0 + jq) * p.Hq + w.h * g + hh) * D;
          for (int d = d0; d < d0 + dcw; d += 16) {
            float acc[16];
#pragma unroll
            for (int i = 0; i < 16; ++i) acc[i] = 0.0f;
            for (int c = 0; c < chunks; ++c) {
              const float *part = p.partials + ci[c].poff;
              const float mc = __ldcg(part + w.rows * D + row);
              if (mc == -INFINITY) continue;
              const float wgt = ptx::ex2(mc - mstar);
              const float4 *src = reinterpret_cast<const float4 *>(part + (int64_t)row * D + d);
#pragma unroll
              for (int v = 0; v < 4; ++v) {
                const float4 a = __ldcg(src + v);
                acc[4 * v] = fmaf(a.x, wgt, acc[4 * v]);
                acc[4 * v + 1] = fmaf(a.y, wgt, acc[4 * v + 1]);
                acc[4 * v + 2] = fmaf(a.z, wgt, acc[4 * v + 2]);
                acc[4 * v + 3] = fmaf(a.w, wgt, acc[4 * v + 3]);
              }
            }
#pragma unroll
            for (int v = 0; v < 2; ++v) {
              uint4 o;
              o.x = pack_bf16(acc[8 * v + 0] * dinv, acc[8 * v + 1] * dinv);
              o.y = pack_bf16(acc[8 * v + 2] * dinv, acc[8 * v + 3] * dinv);
              o.z = pack_bf16(acc[8 * v + 4] * dinv, acc[8 * v + 5] * dinv);
              o.w = pack_bf16(acc[8 * v + 6] * dinv, acc[8 * v + 7] * dinv);
              reinterpret_cast<uint4 *>(og + d)[v] = o;
            }
          }
        }
      }
    }
    if (!ok && lane == 0) report(p.status, WISP_DEV_TIMEOUT, p.request_ids, 0);
  } else {
    // ------------------------------------------------------------------ softmax warps
    const int qd = warp & 3;          // TMEM lane quadrant of this warp
    const int mrow = qd * 32 + lane;  // this thread's MMA row
    const uint32_t lane_addr = (uint32_t)(qd * 32) << 16;
    const float scale_log2 = 1.4426950408889634f / sqrtf((float)D);
    uint32_t n = 0;
    int li = 0;  // items so far: item li accumulates into O buffer li & 1
    bool ok = true;
    for (uint32_t j = 0; ok; ++j) {
      const int slot = j % C::RING;
      if (!wait_bar(B.it_full + slot, (j / C::RING) & 1, s_abort)) { ok = false; break; }
      const int it = s_ring[slot].it;
      const WorkItem w = s_ring[slot].w;
      __syncwarp();
      if (lane == 0) ptx::mbar_arrive(B.it_empty + slot);
      if (it < 0) break;
      const int G = row_group(w.rows), rep = kM / G;
      const int rid = (qd * 32) / G;      // replica handled by this warp
      const int row = mrow - rid * G;     // query row of this thread (j*g + hh)
      const int cw = kBN / rep;           // columns of each S tile handled by this warp
      const int c0 = rid * cw;
      // P is written to every replica row, so O = P V comes out replicated in all four lane
      // quadrants; this warp rescales the O columns [d0, d0 + dcw) of its quadrant
      const int dcw = D / rep;
      const int d0 = rid * dcw;
      const int jq = row / g;
      const int vis = w.ctx + jq;         // last key position this row may see
      const int ob = li & 1;
      const uint32_t o_col = 128 + ob * 128;
      float m_ref = -INFINITY, l = 0.0f;

      const int ntiles = (w.t1 - w.t0 + kBN - 1) / kBN;
      // the tile loop, specialised for the CW columns of each S tile this warp handles
      auto run_tiles = [&](auto cw_tag) -> bool {
        constexpr int CW = decltype(cw_tag)::value;
        for (int t = 0; t < ntiles; ++t, ++n) {
          const int sb = n & 1;
          if (!wait_bar(B.s_full + sb, (n >> 1) & 1, s_abort)) return false;
          ptx::tc_fence_after();
          // the whole 64-column row (replicas hold identical rows, so each warp gets the row max
          // without talking to the others), then this warp's CW columns
          float sr[kBN];
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            uint32_t x[32];
            ptx::tmem_ld32(tmem + lane_addr + sb * 64 + h * 32, x);
            ptx::tmem_wait_ld();
#pragma unroll
            for (int i = 0; i < 32; ++i) sr[h * 32 + i] = __uint_as_float(x[i]);
          }

          const int tok0 = w.t0 + t * kBN;
          // interior tile: every token visible to every row of the item
          const bool interior = tok0 + kBN <= w.t1 && tok0 + kBN - 1 <= w.ctx;
          if (!interior) {
#pragma unroll
            for (int i = 0; i < kBN; ++i) {
              const int tok = tok0 + i;
              if (!(tok < w.t1 && tok <= vis)) sr[i] = -INFINITY;
            }
          }
          // row max with eight independent partial maxima (short dependency chains)
          float m8[8];
#pragma unroll
          for (int k = 0; k < 8; ++k) m8[k] = sr[k];
#pragma unroll
          for (int i = 8; i < kBN; ++i) m8[i & 7] = fmaxf(m8[i & 7], sr[i]);
#pragma unroll
          for (int k = 0; k < 4; ++k) m8[k] = fmaxf(m8[k], m8[k + 4]);
          const float m_tile = fmaxf(fmaxf(m8[0], m8[2]), fmaxf(m8[1], m8[3])) * scale_log2;  // scale > 0
          float sv[CW];
          if constexpr (CW == kBN) {
#pragma unroll
            for (int i = 0; i < CW; ++i) sv[i] = sr[i] * scale_log2;  // -inf stays -inf
          } else {
            // this warp's own CW columns, taken from the (already masked) row in registers; the
            // replica index is warp-uniform, so each case reads registers at constant indices
            auto take = [&](auto part) {
              constexpr int o = decltype(part)::value * CW;
#pragma unroll
              for (int i = 0; i < CW; ++i) sv[i] = sr[o + i] * scale_log2;
            };
            const int part = c0 / CW;
            if (part == 0) take(std::integral_constant<int, 0>{});
            else if (part == 1) take(std::integral_constant<int, 1>{});
            if constexpr (CW == 16) {
              if (part == 2) take(std::integral_constant<int, 2>{});
              else if (part == 3) take(std::integral_constant<int, 3>{});
            }
          }
          // S(n) has been read: its TMEM buffer may be overwritten by S(n+2)
          ptx::tc_fence_before();
          __syncwarp();
          if (lane == 0) ptx::mbar_arrive(B.s_empty + sb);
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
          float ev[CW];
#pragma unroll
          for (int i = 0; i < CW; ++i) ev[i] = ptx::ex2(sv[i] - m_use);
#pragma unroll
          for (int i = 0; i < CW; i += 2) pk[i / 2] = pack_bf16(ev[i], ev[i + 1]);
#pragma unroll
          for (int w2 = 1; w2 < CW; w2 <<= 1) {
#pragma unroll
            for (int i = 0; i < CW; i += 2 * w2) ev[i] += ev[i + w2];
          }
          l += ev[0];
          // PV(m) completes barrier o_full[m % 3] for the (m / 3)-th time.  Every softmax warp
          // waits PV(n-3) here (P buffer n % 3 is free again); since it waited PV(n-6) three tiles
          // ago and PV(n) needs the P(n) it is about to publish, the parity names exactly PV(n-3).
          const int pbuf = (int)(n % 3);
          if (n >= 3 && !wait_bar(B.o_full + pbuf, ((n - 3) / 3) & 1, s_abort)) return false;
          // a rescale of the O rows needs PV(n-1) complete (exact for the same reason) and
          // precedes PV(n); each warp rescales its own column slice of its quadrant's rows
          if (t > 0 && __ballot_sync(0xffffffffu, rescale)) {
            if (!wait_bar(B.o_full + (n - 1) % 3, ((n - 1) / 3) & 1, s_abort)) return false;
            ptx::tc_fence_after();
            for (int c = 0; c < dcw; c += 16) {
              uint32_t x[16];
              ptx::tmem_ld16(tmem + lane_addr + o_col + d0 + c, x);
              ptx::tmem_wait_ld();
#pragma unroll
              for (int i = 0; i < 16; ++i) x[i] = __float_as_uint(__uint_as_float(x[i]) * fac);
              ptx::tmem_st16(tmem + lane_addr + o_col + d0 + c, x);
            }
            ptx::tmem_wait_st();
            ptx::tc_fence_before();
          }
          // this warp's columns of P row `row` (bf16, 128-byte swizzle)
#pragma unroll
          for (int rr = 0; rr < kBN / CW; ++rr) {
            uint8_t *prow = smem + C::OFF_P + pbuf * C::P_BYTES + (rr * G + row) * 128;  // (rr*G + row) & 7 == row & 7
#pragma unroll
            for (int c = 0; c < CW / 8; ++c) {
              const int cc = c0 / 8 + c;
              *reinterpret_cast<uint4 *>(prow + ((cc ^ (row & 7)) << 4)) =
                  make_uint4(pk[4 * c], pk[4 * c + 1], pk[4 * c + 2], pk[4 * c + 3]);
            }
          }
          ptx::fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) ptx::mbar_arrive(B.p_full + pbuf);
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

      // ---- hand the item over to the epilogue warps: this thread's share of the row sum and the
      // reference max go to two spare TMEM columns of its lane.  The epilogue of item li - 2 (same
      // O buffer and columns) must be done with them first.
      if (!wait_bar(B.o_empty + ob, ((li >> 1) & 1) ^ 1, s_abort)) { ok = false; break; }
      ptx::tc_fence_after();
      {
        const uint32_t lm[2] = {__float_as_uint(l), __float_as_uint(m_ref)};
        ptx::tmem_st2(tmem + lane_addr + 384 + 2 * ob, lm);
        ptx::tmem_wait_st();
      }
      ptx::tc_fence_before();
      __syncwarp();
      if (lane == 0) ptx::mbar_arrive(B.ep_full + ob);
      ++li;
    }
    if (!ok && lane == 0) report(p.status, WISP_DEV_TIMEOUT, p.request_ids, 0);
  }

  // __syncthreads is an aligned barrier: each warp must reach it converged, and the roles above
  // leave lane 0 alone in its loop (MMA issue, drains)
  __syncwarp();
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
// one box = 64 head-dim elements (128 bytes, swizzled) x 16 slots of one head in `box_blocks`
// consecutive blocks (1, or 4 for a whole 64-token tile of consecutive blocks).
cudaError_t encode_pool(CUtensorMap *map, const void *base, int D, int Hkv, int num_blocks, int box_blocks) {
  const cuuint64_t dims[4] = {(cuuint64_t)D, 16, (cuuint64_t)Hkv, (cuuint64_t)num_blocks};
  const cuuint64_t strides[3] = {(cuuint64_t)D * 2, (cuuint64_t)16 * D * 2, (cuuint64_t)Hkv * 16 * D * 2};
  const cuuint32_t box[4] = {64, 16, 1, (cuuint32_t)box_blocks};
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
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(attn_tc_kernel<128>, cudaFuncAttributePreferredSharedMemoryCarveout, cudaSharedmemCarveoutMaxShared);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(attn_tc_kernel<64>, cudaFuncAttributePreferredSharedMemoryCarveout, cudaSharedmemCarveoutMaxShared);
  return e;
}

cudaError_t attn_tc_launch(const AttnParams &p, int grid, cudaStream_t s) {
  alignas(64) CUtensorMap tk, tv, tk4, tv4;
  cudaError_t e = encode_pool(&tk, p.k_cache, p.D, p.Hkv, p.num_blocks, 1);
  if (e == cudaSuccess) e = encode_pool(&tv, p.v_cache, p.D, p.Hkv, p.num_blocks, 1);
  if (e == cudaSuccess) e = encode_pool(&tk4, p.k_cache, p.D, p.Hkv, p.num_blocks, 4);
  if (e == cudaSuccess) e = encode_pool(&tv4, p.v_cache, p.D, p.Hkv, p.num_blocks, 4);
  if (e != cudaSuccess) return e;
  if (p.D == 128) {
    attn_tc_kernel<128><<<grid, kThreads, Cfg<128>::SMEM, s>>>(p, tk, tv, tk4, tv4);
  } else {
    attn_tc_kernel<64><<<grid, kThreads, Cfg<64>::SMEM, s>>>(p, tk, tv, tk4, tv4);
  }
  return cudaGetLastError();
}

}  // namespace wisp
