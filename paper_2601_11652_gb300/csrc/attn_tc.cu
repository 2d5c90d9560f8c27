// attn_tc.cu -- tensor-core paged GQA attention for the verification forward (bf16 KV).
//
// Same contract as attn_simt.cu (Sec. 4.4-4.5: request r's k+1 new queries over its
// L_total = L_cached + L_new paged keys, query j seeing keys 0..c_r + j), built for sm_103a.
//
// A verification item has few query rows (g * (k+1), at most 64 per item) and many keys, so the
// products run transposed: the keys are the MMA's M dimension and the query rows its N.
//   S^T = K Q^T       (M = 128 keys of a tile, N = the item's rows rounded up to 16, K = D)
//   O^T += V^T P^T    (M = D, N = rows, K = 128 keys)
// Nothing is replicated to fill the 128-row MMA, and the tensor core reads each K and V tile from
// shared memory once.
//
// Persistent CTAs (one per SM) take work items (request, KV head, key chunk, row group) from a
// global counter, in the planner's longest-first order.  Warp roles in a CTA:
//   * warp 6 (item loader) takes the next item just in time (when the K producer is three tiles
//     from the end of the current one), publishes it to the other warps through a 4-slot shared
//     ring, and copies its query rows into one of two shared Q buffers (128-byte-swizzled,
//     K-major: the B operand of S^T);
//   * warps 0 and 7 (K and V producers) stream the item's K and V tiles of 128 tokens with TMA
//     tiled loads into two rings: one 16 KB box per 64-wide half of the head dim when the tile's
//     eight 16-token blocks are consecutive in the pool, else one 2 KB box per block; blocks past
//     the item read as zeros (out-of-range box).  A K stage is free again once S^T of its tile is
//     done, a V stage once its PV product is;
//   * warp 1 (one thread) issues tcgen05.mma: S^T into one of two TMEM tiles (key t in TMEM lane
//     t, query row j in column j), and O^T into the item's TMEM accumulator (head-dim index d in
//     lane d, row j in column j; two accumulators alternating between items);
//   * warps 2-5 and 12-15 (softmax): the first group takes rows 0-31 of an item, the second rows
//     32-63; within a group one warp per TMEM lane quadrant, i.e. 32 keys of each tile per warp: a
//     thread holds one key's scores for the group's rows.  The rows' reference maxima live in
//     shared memory; a tile whose scores exceed a reference by more than 2^8 anywhere (the first
//     tile of an item always does) makes the warps agree on new maxima (exact per-row tile
//     maxima) and, if O holds earlier tiles, rescale their O^T columns in TMEM.  Each thread
//     writes its key's part of the P row (bf16, MN-major, swizzled: the B operand of the PV
//     product) and keeps its share of every row sum;
//   * warps 8-11 (epilogue) add the row-sum shares, read O^T from TMEM and write the normalised
//     output or, for a split item, the (O, m, l) partials; the last chunk of a split
//     (request, head, row group) to finish merges all its chunks.  This runs while the softmax
//     warps are already on the next item.
// Every mbarrier wait is bounded in time; an expired wait records WISP_DEV_TIMEOUT and the CTA
// drains.  No named barrier is used: a warp that gives up cannot leave the others blocked, and the
// TMEM is freed once every warp has arrived on a final mbarrier.
#include "attn.cuh"
#include "sm100_ptx.cuh"

#include <cudaTypedefs.h>
#include <cstring>
#include <mutex>
#include <type_traits>

namespace wisp {

namespace {

constexpr int kBT = 128;            // KV tokens per tile (the M of S^T)
constexpr int kNR = kTcRowsPerItem; // query rows per item at most (64: the planner cuts larger sets)
constexpr int kThreads = 512;       // warp 0 K producer, warp 1 MMA, warps 2-5 softmax (rows 0-31), warp 6
                                    // item loader, warp 7 V producer, warps 8-11 epilogue, warps 12-15
                                    // softmax (rows 32-63)
constexpr int kSoftmaxWarps = 8;
constexpr uint32_t kTmemCols = 256; // S^T[2] at columns 0 / 64, O^T[2] at 128 / 192
constexpr long long kWaitCycles = 4000000000LL;  // about two seconds: a wait that long is a failure
constexpr float kTau = 8.0f;        // lazy rescale threshold (log2 units)
constexpr float kExpTau = 256.0f;   // 2^kTau
static_assert(kNR == 64, "TMEM and shared-memory layout assume 64 rows per item");

template <int D>
struct Cfg {
  static constexpr int HALVES = D / 64;
  static constexpr int HALF = kBT * 128;        // one 64-wide half of a K / V tile: [128 tokens][128 B]
  static constexpr int KV_TILE = HALVES * HALF; // K (or V) of one tile
  static constexpr int QHALF = kNR * 128;       // one half of a Q buffer: [64 rows][128 B]
  static constexpr int Q_BYTES = HALVES * QHALF;
  static constexpr int P_BYTES = kBT * kNR * 2; // P^T: [128 tokens][64 rows] bf16
  static constexpr int NSK = D == 128 ? 2 : 4;  // K ring stages
  static constexpr int NSV = D == 128 ? 2 : 4;  // V ring stages
  static constexpr int NQ = 2;                  // Q buffers: item li's rows in buffer li % NQ
  static constexpr int NP = 2;                  // P buffers: P(n) in buffer n % NP
  static constexpr int RING = 4;                // slots of the item ring
  static constexpr int OFF_Q = 0;
  static constexpr int OFF_K = OFF_Q + NQ * Q_BYTES;
  static constexpr int OFF_V = OFF_K + NSK * KV_TILE;
  static constexpr int OFF_P = OFF_V + NSV * KV_TILE;
  static constexpr int OFF_BAR = OFF_P + NP * P_BYTES;
  static constexpr int N_BAR = 2 * NSK + 2 * NSV + 8 + 2 * NP + 6 + 1 + 2 * RING + 5;
  static constexpr int OFF_MW = (OFF_BAR + N_BAR * 8 + 15) / 16 * 16;  // float [8][32] per-warp row maxima
  static constexpr int OFF_FW = OFF_MW + kSoftmaxWarps * 32 * 4;       // float [8][32] per-warp rescale factors
  static constexpr int OFF_RED = OFF_FW + kSoftmaxWarps * 32 * 4;      // float [4][64] tile maxima per quadrant
  static constexpr int OFF_FLAG = OFF_RED + 4 * kNR * 4;               // uint32 [2][8] exceed votes per warp
  static constexpr int OFF_HL = OFF_FLAG + 64;                         // float [2][4][64] row-sum shares per quadrant
  static constexpr int OFF_HM = OFF_HL + 2 * 4 * kNR * 4;              // float [2][64] row reference maxima
  static constexpr int OFF_EM = OFF_HM + 2 * kNR * 4;                  // float [2][64] merge: max, 1 / sum
  static constexpr int OFF_MISC = OFF_EM + 2 * kNR * 4;                // tmem base, flags
  static constexpr int OFF_RING = OFF_MISC + 64;                       // RING x (index, WorkItem)
  static constexpr int SMEM = OFF_RING + RING * 64 + 1024;             // + slack to align the base to 1024
  static_assert(SMEM <= 227 * 1024, "shared memory of one CTA on sm_103a");
  static_assert(OFF_K % 1024 == 0 && OFF_V % 1024 == 0 && OFF_P % 1024 == 0, "swizzled buffers need 1 KB alignment");
};

struct Bars {
  uint64_t *k_full, *k_empty, *v_full, *v_empty, *q_full, *q_empty, *s_full, *s_empty, *p_full, *o_full;
  uint64_t *o_empty, *o_done, *ep_full, *mma_done, *it_full, *it_empty, *egrp, *sm_sync, *sm_sync2, *fin, *claim;
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
  return w.r >= 0 && w.r < p.B && p.req_flag[w.r] == REQ_OK && w.t1 > w.t0 && w.rows > 0 && w.rows <= kNR &&
         w.row0 >= 0 && (w.nrg == 1 || w.nrg == 2) && w.rg >= 0 && w.rg < w.nrg;
}

__device__ __forceinline__ uint32_t pack_bf16(float a, float b) {
  __nv_bfloat162 v = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t *>(&v);
}

// Transposing reductions over the 32 lanes of a warp (v is consumed): on return lane i holds the
// sum (max) over all lanes of v[i].  31 shuffles for 32 values.
template <bool MAX>
__device__ __forceinline__ float warp_transpose_reduce(float (&v)[32], int lane) {
#pragma unroll
  for (int w = 16; w >= 1; w >>= 1) {
    const bool up = (lane & w) != 0;
#pragma unroll
    for (int i = 0; i < w; ++i) {
      const float keep = up ? v[i + w] : v[i];
      const float send = up ? v[i] : v[i + w];
      const float got = __shfl_xor_sync(0xffffffffu, send, w);
      v[i] = MAX ? fmaxf(keep, got) : keep + got;
    }
  }
  return v[0];
}

}  // namespace

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    attn_tc_kernel(const __grid_constant__ AttnParams p, const __grid_constant__ CUtensorMap tmk,
                   const __grid_constant__ CUtensorMap tmv, const __grid_constant__ CUtensorMap tmk8,
                   const __grid_constant__ CUtensorMap tmv8) {
  using C = Cfg<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t sbase = ptx::smem_u32(smem);
  uint64_t *bar = reinterpret_cast<uint64_t *>(smem + C::OFF_BAR);
  Bars B;
  B.k_full = bar;
  B.k_empty = B.k_full + C::NSK;
  B.v_full = B.k_empty + C::NSK;
  B.v_empty = B.v_full + C::NSV;
  B.q_full = B.v_empty + C::NSV;
  B.q_empty = B.q_full + 2;
  B.s_full = B.q_empty + 2;
  B.s_empty = B.s_full + 2;
  B.p_full = B.s_empty + 2;     // [NP] per P buffer
  B.o_full = B.p_full + C::NP;  // [NP] per P buffer: PV of tiles n with n % NP == b
  B.o_empty = B.o_full + C::NP; // [2] per O buffer: its epilogue is done
  B.o_done = B.o_empty + 2;     // [2] per O buffer: the item's last PV is done
  B.ep_full = B.o_done + 2;     // [2] per O buffer: the softmax warps handed the item over
  B.mma_done = B.ep_full + 2;
  B.it_full = B.mma_done + 1;
  B.it_empty = B.it_full + C::RING;
  B.egrp = B.it_empty + C::RING;
  B.sm_sync = B.egrp + 1;       // the softmax warps, once per tile
  B.sm_sync2 = B.sm_sync + 1;   // the softmax warps, once per tile that moves a reference max
  B.fin = B.sm_sync2 + 1;       // every warp, once: its last access to TMEM is done
  B.claim = B.fin + 1;          // the K producer, once per item, a few tiles before the item's end
  static_assert(2 * C::NSK + 2 * C::NSV + 8 + 2 * C::NP + 6 + 1 + 2 * C::RING + 5 <= C::N_BAR, "barrier count");
  float *s_mw = reinterpret_cast<float *>(smem + C::OFF_MW);
  float *s_fw = reinterpret_cast<float *>(smem + C::OFF_FW);
  float *s_red = reinterpret_cast<float *>(smem + C::OFF_RED);
  volatile uint32_t *s_flag = reinterpret_cast<volatile uint32_t *>(smem + C::OFF_FLAG);
  float *s_em = reinterpret_cast<float *>(smem + C::OFF_EM);
  float *s_hl = reinterpret_cast<float *>(smem + C::OFF_HL);
  float *s_hm = reinterpret_cast<float *>(smem + C::OFF_HM);
  uint32_t *s_tmem = reinterpret_cast<uint32_t *>(smem + C::OFF_MISC);
  volatile int *s_abort = reinterpret_cast<volatile int *>(smem + C::OFF_MISC + 4);
  volatile int *s_last = reinterpret_cast<volatile int *>(smem + C::OFF_MISC + 8);
  struct RingSlot {
    int it;
    int pad[3];
    WorkItem w;
  };
  static_assert(sizeof(RingSlot) <= 64, "item ring slot");
  RingSlot *s_ring = reinterpret_cast<RingSlot *>(smem + C::OFF_RING);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < C::NSK; ++s) {
      ptx::mbar_init(B.k_full + s, 1);
      ptx::mbar_init(B.k_empty + s, 1);
    }
    for (int s = 0; s < C::NSV; ++s) {
      ptx::mbar_init(B.v_full + s, 1);
      ptx::mbar_init(B.v_empty + s, 1);
    }
    for (int b = 0; b < 2; ++b) {
      ptx::mbar_init(B.q_full + b, 1);
      ptx::mbar_init(B.q_empty + b, 1);
      ptx::mbar_init(B.s_full + b, 1);
      ptx::mbar_init(B.s_empty + b, kSoftmaxWarps);
    }
    for (int b = 0; b < C::NP; ++b) {
      ptx::mbar_init(B.p_full + b, kSoftmaxWarps);
      ptx::mbar_init(B.o_full + b, 1);
    }
    for (int b = 0; b < 2; ++b) {
      ptx::mbar_init(B.o_empty + b, 4);  // the four epilogue warps
      ptx::mbar_init(B.o_done + b, 1);
      ptx::mbar_init(B.ep_full + b, kSoftmaxWarps);
    }
    ptx::mbar_init(B.mma_done, 1);
    for (int i = 0; i < C::RING; ++i) {
      ptx::mbar_init(B.it_full + i, 1);
      ptx::mbar_init(B.it_empty + i, 3 + kSoftmaxWarps + 4);  // KV producers, MMA, softmax and epilogue warps
    }
    ptx::mbar_init(B.egrp, 4);      // the four epilogue warps
    ptx::mbar_init(B.sm_sync, kSoftmaxWarps);
    ptx::mbar_init(B.sm_sync2, kSoftmaxWarps);
    ptx::mbar_init(B.fin, kThreads / 32);
    ptx::mbar_init(B.claim, 1);
    *s_abort = 0;
    ptx::fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    ptx::prefetch_tmap(&tmk);
    ptx::prefetch_tmap(&tmv);
    ptx::prefetch_tmap(&tmk8);
    ptx::prefetch_tmap(&tmv8);
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

  // everything above may overlap the planner (programmatic dependent launch); the plan is read
  // only once the planner's grid has completed and its writes are visible
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int n_items = p.header->n_items;
  if ((int)blockIdx.x >= p.header->attn_ctas) {
    // the planner leaves this SM to the acceptance pass of the same step: nothing was issued yet
    if (warp == 1) ptx::tmem_dealloc(tmem, kTmemCols);
    return;
  }
  const int g = p.Hq / p.Hkv;

  if (warp == 0 || warp == 7) {
    // ------------------------------------------------------------------ K / V producers
    // K and V have rings of their own: a K stage is free again once S^T of its tile is done, a V
    // stage once PV is, so each tensor is fetched about as many tiles ahead of its use as its ring
    // has stages.
    const bool is_k = warp == 0;
    const uint32_t ns = is_k ? C::NSK : C::NSV;
    const CUtensorMap *tm1 = is_k ? &tmk : &tmv;
    const CUtensorMap *tm8 = is_k ? &tmk8 : &tmv8;
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
      int cur = fetch(0), nxt = fetch(32);  // block ids of tiles t..t+3 and t+4..t+7
      const int ntiles = (w.t1 - w.t0 + kBT - 1) / kBT;
      const int t_claim = ntiles > 3 ? ntiles - 3 : 0;
      for (int t = 0; t < ntiles; ++t, ++tile_n) {
        // a few tiles before this item's end the loader may take the next one (items are taken
        // just in time, so the work counter balances the CTAs to the end)
        if (is_k && t == t_claim && lane == 0) ptx::mbar_arrive(B.claim);
        if (t > 0 && (t & 3) == 0) {
          cur = nxt;
          nxt = fetch(32 * ((t >> 2) + 1));
        }
        const int s = (int)(tile_n % ns);
        const uint32_t round = tile_n / ns;
        if (!wait_bar(empty + s, (round & 1) ^ 1, s_abort)) { ok = false; break; }
        if (lane == 0) ptx::mbar_arrive_expect_tx(full + s, C::KV_TILE);
        __syncwarp();
        const int bi = lane & 7;  // block of the tile this lane looks after
        int bid = __shfl_sync(0xffffffffu, cur, (8 * t + bi) & 31);
        const int rel = 8 * t + bi;
        bool valid = rel < nblk && bid >= 0 && bid < p.num_blocks;
        if (is_k && lane < 8 && rel < nblk && !valid) report(p.status, WISP_DEV_BAD_BLOCK, p.request_ids, w.r);
        const int b0 = __shfl_sync(0xffffffffu, bid, 0);
        // eight consecutive valid blocks: one 16 KB box per (tensor, half) with the 8-block maps
        const unsigned contig = __ballot_sync(0xffffffffu, lane < 8 && valid && bid == b0 + lane);
        if (contig == 0xFFu) {
          if (lane == 0) {
#pragma unroll
            for (int hf = 0; hf < C::HALVES; ++hf) {
              ptx::tma_load_4d(off_t + s * C::KV_TILE + hf * C::HALF, tm8, full + s, hf * 64, 0, w.h, b0);
            }
          }
        } else if (lane < 8) {
          if (!valid) bid = p.num_blocks;  // past the item (or invalid): out-of-range box, reads zeros
#pragma unroll
          for (int hf = 0; hf < C::HALVES; ++hf) {
            const uint32_t off = s * C::KV_TILE + hf * C::HALF + lane * (16 * 128);
            ptx::tma_load_4d(off_t + off, tm1, full + s, hf * 64, 0, w.h, bid);
          }
        }
      }
    }
    if (!ok && lane == 0) report(p.status, WISP_DEV_TIMEOUT, p.request_ids, 0);
    // drain: every stage issued must land before the CTA's shared memory goes away
    if (lane == 0) {
      for (uint32_t k = 0; k < ns && k < tile_n; ++k) {
        const uint32_t n = tile_n - 1 - k;
        const long long t0 = clock64();
        while (!ptx::mbar_try_wait(full + n % ns, (n / ns) & 1) && clock64() - t0 < kWaitCycles) {
        }
      }
    }
  } else if (warp == 6) {
    // ------------------------------------------------------------------ item loader
    int li = 0;
    bool ok = true;
    for (uint32_t j = 0; ok; ++j) {
      // next valid work item: publish it to the other warps, then load its query rows.  Item j is
      // taken once the K producer is near the end of item j - 1 (the claim barrier completes once
      // per item, and the producer cannot pass item j - 1 before item j is published: the parity
      // is exact).
      const int slot = j % C::RING;
      if (j > 0 && !wait_bar(B.claim, (j - 1) & 1, s_abort)) { ok = false; break; }
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
      if (it < 0) {
        // no item left for this CTA: a kernel launched after this one as a programmatic
        // dependent (the acceptance walk) may be scheduled; it still waits for this grid to finish
        asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
        break;
      }
      const WorkItem w = p.items[it];
      const int qb = li % C::NQ;
      if (!wait_bar(B.q_empty + qb, ((li / C::NQ) & 1) ^ 1, s_abort)) { ok = false; break; }
      ++li;
      // the item's query rows -> Q[qb], row rho (query row row0 + rho = j*g + hh) at MMA row rho.
      // Loads are issued QBATCH at a time per lane before any store.  Rows past `rows` up to the
      // MMA's N only feed S^T columns that the softmax masks.
      const uint16_t *qg = static_cast<const uint16_t *>(p.q);
      uint8_t *qs = smem + C::OFF_Q + qb * C::Q_BYTES;
      constexpr int CPR = D / 8;  // 16-byte chunks per row
      constexpr int QBATCH = 8;
      const int nchunks = w.rows * CPR;
      for (int base = 0; base < nchunks; base += 32 * QBATCH) {
        uint4 v[QBATCH];
#pragma unroll
        for (int u = 0; u < QBATCH; ++u) {
          const int c = base + u * 32 + lane;
          if (c < nchunks) {
            const int row = c / CPR, cc = c % CPR;
            const int rj = w.row0 + row;
            const int jj = rj / g, hh = rj % g;
            v[u] = __ldg(reinterpret_cast<const uint4 *>(qg + ((int64_t)(w.q0 + jj) * p.Hq + w.h * g + hh) * D) + cc);
          }
        }
#pragma unroll
        for (int u = 0; u < QBATCH; ++u) {
          const int c = base + u * 32 + lane;
          if (c < nchunks) {
            const int row = c / CPR, cc = c % CPR;
            *reinterpret_cast<uint4 *>(qs + (cc >> 3) * C::QHALF + row * 128 + (((cc & 7) ^ (row & 7)) << 4)) = v[u];
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
    // One thread polls two queues: S^T(n) is issued as soon as tile n's K has landed, its Q is
    // loaded and its TMEM buffer has been read; PV(m) as soon as P(m) is published and V(m) has
    // landed (and, for an item's first tile, the previous item's O has been read).  S^T therefore
    // runs ahead of PV instead of waiting behind it.
    if (lane == 0) {
      uint32_t n_s = 0, n_pv = 0, j = 0;
      int li = 0, s_t = 0, s_nt = 0, s_qb = 0, s_li = 0;
      uint32_t s_idesc = 0, s_pvdesc = 0;
      bool s_have = false, items_done = false, ok = true;
      uint8_t tflag[4];     // per issued S^T tile: bit 0 first tile of its item, bit 1 its last
      int tli[4];           // item number of the tile (O buffer, o_empty parity)
      uint32_t tpv[4];      // instruction descriptor of the tile's PV product
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
              const int nrow = (w.rows + 15) / 16 * 16;  // the MMA's N: rows rounded up to 16
              s_idesc = ptx::idesc_bf16_f32(kBT, nrow, false, false);
              s_pvdesc = ptx::idesc_bf16_f32(128, nrow, true, true);
              s_have = true;
              s_t = 0;
              s_nt = (w.t1 - w.t0 + kBT - 1) / kBT;
              s_qb = li % C::NQ;
              s_li = li;
              ++li;
            }
            prog = true;
          }
        }
        if (s_have && n_s < n_pv + 4) {
          const int st = (int)(n_s % C::NSK), sb = n_s & 1;
          if ((s_t > 0 || ptx::mbar_test_wait(B.q_full + s_qb, (s_li / C::NQ) & 1)) &&
              ptx::mbar_test_wait(B.k_full + st, (n_s / C::NSK) & 1) &&
              ptx::mbar_test_wait(B.s_empty + sb, ((n_s >> 1) & 1) ^ 1)) {
            ptx::tc_fence_after();
            const uint32_t qa = sbase + C::OFF_Q + s_qb * C::Q_BYTES;
            const uint32_t ka = sbase + C::OFF_K + st * C::KV_TILE;
#pragma unroll
            for (int ks = 0; ks < D / 16; ++ks) {
              const uint32_t koff = (ks >> 2) * C::HALF + (ks & 3) * 32;
              const uint32_t qoff = (ks >> 2) * C::QHALF + (ks & 3) * 32;
              ptx::umma_f16(tmem + sb * kNR, ptx::sdesc_sw128(ka + koff, 16, 1024),
                            ptx::sdesc_sw128(qa + qoff, 16, 1024), s_idesc, ks > 0);
            }
            ptx::umma_commit(B.s_full + sb);
            ptx::umma_commit(B.k_empty + st);
            if (s_t == s_nt - 1) ptx::umma_commit(B.q_empty + s_qb);
            tflag[n_s & 3] = (s_t == 0 ? 1 : 0) | (s_t == s_nt - 1 ? 2 : 0);
            tli[n_s & 3] = s_li;
            tpv[n_s & 3] = s_pvdesc;
            ++n_s;
            if (++s_t == s_nt) s_have = false;
            prog = true;
          }
        }
        if (n_pv < n_s) {
          const int pb = (int)(n_pv % C::NP);
          const bool first = tflag[n_pv & 3] & 1, last = tflag[n_pv & 3] & 2;
          const int tl = tli[n_pv & 3], ob = tl & 1;  // the item's O buffer
          const int st = (int)(n_pv % C::NSV);
          if (ptx::mbar_test_wait(B.p_full + pb, (n_pv / C::NP) & 1) &&
              ptx::mbar_test_wait(B.v_full + st, (n_pv / C::NSV) & 1) &&
              (!first || ptx::mbar_test_wait(B.o_empty + ob, ((tl >> 1) & 1) ^ 1))) {
            ptx::tc_fence_after();
            const uint32_t pa = sbase + C::OFF_P + pb * C::P_BYTES;
            const uint32_t va = sbase + C::OFF_V + st * C::KV_TILE;
            // A = V^T, MN-major: the head dim's 64-wide halves are HALF apart (for D = 64 both MMA
            // halves read the same half, so O^T lanes 64..127 repeat lanes 0..63 and are not used)
            constexpr uint32_t lbo_v = D == 128 ? C::HALF : 0;
#pragma unroll
            for (int ks = 0; ks < kBT / 16; ++ks) {
              const uint64_t a = ptx::sdesc_sw128(va + ks * 16 * 128, lbo_v, 1024);
              const uint64_t b = ptx::sdesc_sw128(pa + ks * 16 * 128, C::P_BYTES, 1024);
              ptx::umma_f16(tmem + 128 + ob * kNR, a, b, tpv[n_pv & 3], (!first || ks > 0) ? 1u : 0u);
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
  } else if (warp >= 8 && warp < 12) {
    // ------------------------------------------------------------------ epilogue warps
    // One warp per TMEM lane quadrant: thread d (lane d of O^T) owns head-dim index d of every row.
    // Item li's O^T (buffer li & 1) is read once the softmax warps have handed the item over and
    // its last PV is done; the output (or, for a split item, the partial O, m, l) is written, the
    // buffer released, and the last chunk of a split (request, head, row group) to finish merges
    // all of its chunks.
    const int qd = warp & 3;
    const int d = qd * 32 + lane;
    const bool dval = d < D;  // for D = 64 the upper two quadrants hold copies
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
      const int ob = li & 1;
      const uint32_t o_col = 128 + ob * kNR;
      // the softmax warps' hand-over and the item's last PV
      if (!wait_bar(B.ep_full + ob, (li >> 1) & 1, s_abort)) { ok = false; break; }
      if (!wait_bar(B.o_done + ob, (li >> 1) & 1, s_abort)) { ok = false; break; }
      ++li;
      ptx::tc_fence_after();
      const int nc = (w.rows + 31) / 32;
      for (int c = 0; c < nc; ++c) {
        uint32_t x[32];  // O^T[d][rows 32c..]
        ptx::tmem_ld32(tmem + lane_addr + o_col + 32 * c, x);
        ptx::tmem_wait_ld();
        // lane i: row 32c + i's sum (the four softmax warps' shares)
        const int jl = 32 * c + lane;
        const float *hl = s_hl + ob * 4 * kNR;
        const float lsum = hl[jl] + hl[kNR + jl] + hl[2 * kNR + jl] + hl[3 * kNR + jl];
        if (w.poff < 0) {
          const float linv = 1.0f / lsum;
          uint16_t *og = static_cast<uint16_t *>(p.out);
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const int jr = 32 * c + i;
            const float inv = __shfl_sync(0xffffffffu, linv, i);
            if (jr < w.rows && dval) {
              const int rj = w.row0 + jr, jq = rj / g, hh = rj % g;
              const float o = __uint_as_float(x[i]) * inv;
              og[((int64_t)(w.q0 + jq) * p.Hq + w.h * g + hh) * D + d] = __bfloat16_as_ushort(__float2bfloat16_rn(o));
            }
          }
        } else {
          float *part = p.partials + w.poff;
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const int jr = 32 * c + i;
            if (jr < w.rows && dval) __stcg(part + (int64_t)jr * D + d, __uint_as_float(x[i]));
          }
          if (qd == 0 && jl < w.rows) {
            __stcg(part + w.rows * D + jl, s_hm[ob * kNR + jl]);
            __stcg(part + w.rows * D + w.rows + jl, lsum);
          }
        }
      }
      ptx::tc_fence_before();
      __syncwarp();
      if (lane == 0) ptx::mbar_arrive(B.o_empty + ob);

      // ---- split item: the last chunk of this (request, head, row group) to finish merges all ----
      if (w.poff >= 0) {
        __threadfence();
        if (!group_sync()) { ok = false; break; }
        if (warp == 8 && lane == 0) {
          const int chunks = p.req_chunks[w.r];
          const int done = atomicAdd(p.pair_done + ((int64_t)w.r * p.Hkv + w.h) * 2 + w.rg, 1);
          *s_last = done == chunks - 1 ? chunks : 0;
          __threadfence();
        }
        if (!group_sync()) { ok = false; break; }
        const int chunks = *s_last;
        if (chunks > 0) {
          const WorkItem *ci = p.items + p.req_item_begin[w.r] + (w.h * w.nrg + w.rg) * chunks;
          // thread jr < rows: row jr's overall max and 1 / sum over the chunks
          if (d < w.rows) {
            float mstar = -INFINITY;
            for (int c = 0; c < chunks; ++c) mstar = fmaxf(mstar, __ldcg(p.partials + ci[c].poff + w.rows * D + d));
            float den = 0.0f;
            for (int c = 0; c < chunks; ++c) {
              const float *part = p.partials + ci[c].poff;
              const float mc = __ldcg(part + w.rows * D + d);
              if (mc != -INFINITY) den = fmaf(__ldcg(part + w.rows * D + w.rows + d), ptx::ex2(mc - mstar), den);
            }
            s_em[d] = mstar;
            s_em[kNR + d] = 1.0f / den;
          }
          if (!group_sync()) { ok = false; break; }
          // thread d: column d of every row, eight rows at a time (independent loads in flight)
          if (dval) {
            uint16_t *og = static_cast<uint16_t *>(p.out);
            for (int j0 = 0; j0 < w.rows; j0 += 8) {
              float acc[8];
#pragma unroll
              for (int q = 0; q < 8; ++q) acc[q] = 0.0f;
#pragma unroll 4
              for (int c = 0; c < chunks; ++c) {
                const float *part = p.partials + ci[c].poff;
#pragma unroll
                for (int q = 0; q < 8; ++q) {
                  const int jr = j0 + q;
                  if (jr < w.rows) {
                    const float mc = __ldcg(part + w.rows * D + jr);
                    const float ov = __ldcg(part + (int64_t)jr * D + d);
                    if (mc != -INFINITY) acc[q] = fmaf(ov, ptx::ex2(mc - s_em[jr]), acc[q]);
                  }
                }
              }
#pragma unroll
              for (int q = 0; q < 8; ++q) {
                const int jr = j0 + q;
                if (jr < w.rows) {
                  const int rj = w.row0 + jr, jq = rj / g, hh = rj % g;
                  og[((int64_t)(w.q0 + jq) * p.Hq + w.h * g + hh) * D + d] =
                      __bfloat16_as_ushort(__float2bfloat16_rn(acc[q] * s_em[kNR + jr]));
                }
              }
            }
          }
          // s_em is read above until every warp is past this point
          if (!group_sync()) { ok = false; break; }
        }
      }
    }
    if (!ok && lane == 0) report(p.status, WISP_DEV_TIMEOUT, p.request_ids, 0);
  } else {
    // ------------------------------------------------------------------ softmax warps
    // Two groups of four: warps 2-5 take rows 0-31 of every item, warps 12-15 rows 32-63 (and only
    // keep in step for items of at most 32 rows).  Within a group, one warp per TMEM lane quadrant,
    // i.e. 32 keys of each tile: a thread holds one key's scores for the group's 32 rows.
    const int qd = warp & 3;                  // TMEM lane quadrant: keys 32*qd .. 32*qd + 31 of a tile
    const int grp = warp >= 12 ? 1 : 0;       // row chunk: rows 32*grp .. 32*grp + 31
    const int sw8 = grp * 4 + qd;             // index of this warp among the eight
    const uint32_t lane_addr = (uint32_t)(qd * 32) << 16;
    const float scale_log2 = 1.4426950408889634f / sqrtf((float)D);
    float *mw = s_mw + sw8 * 32;              // this warp's copy of its rows' reference maxima
    float *fw = s_fw + sw8 * 32;              // this warp's copy of its rows' rescale factors
    const int r0 = 32 * grp;                  // first row of the chunk
    uint32_t n = 0, nf = 0;                   // tiles so far; tiles that moved a reference max
    int li = 0;                               // items so far: item li accumulates into O buffer li & 1
    bool ok = true;
    for (uint32_t j = 0; ok; ++j) {
      const int slot = j % C::RING;
      if (!wait_bar(B.it_full + slot, (j / C::RING) & 1, s_abort)) { ok = false; break; }
      const int it = s_ring[slot].it;
      const WorkItem w = s_ring[slot].w;
      __syncwarp();
      if (lane == 0) ptx::mbar_arrive(B.it_empty + slot);
      if (it < 0) break;
      const int ob = li & 1;
      const uint32_t o_col = 128 + ob * kNR;
      const int ntiles = (w.t1 - w.t0 + kBT - 1) / kBT;
      // 8-row units of this chunk that the MMA reads (its N / 8 minus the chunk's offset)
      const int nu = min(4, max(0, (w.rows + 15) / 16 * 2 - 4 * grp));
      const bool active = nu > 0;
      const int jmax = w.rows - r0;          // rows of the item in this chunk (may be <= 0)
      mw[lane] = -INFINITY;
      __syncwarp();
      float lp[32];  // this thread's (key's) share of every row sum of the chunk
#pragma unroll
      for (int i = 0; i < 32; ++i) lp[i] = 0.0f;
      for (int t = 0; t < ntiles && ok; ++t, ++n) {
        const int sb = n & 1;
        if (!wait_bar(B.s_full + sb, (n >> 1) & 1, s_abort)) { ok = false; break; }
        ptx::tc_fence_after();
        const int pbuf = (int)(n % C::NP);
        uint8_t *prow = smem + C::OFF_P + pbuf * C::P_BYTES + (qd * 32 + lane) * 128;
        const int sw = lane & 7;
        // causal mask: key tok is visible to row jr iff tok <= ctx + (row0 + jr) / g, i.e.
        // row0 + jr >= g * (tok - ctx); keys past the item and rows past `rows` are masked too
        const int tok = w.t0 + t * kBT + qd * 32 + lane;
        const int jmin = (tok >= w.t1 ? kNR : max(0, g * (tok - w.ctx) - w.row0)) - r0;
        float emax = 0.0f;
        if (active) {
          // P buffer n % NP is free again once PV(n - NP) is done: the other group's wait or this
          // warp's own one covered PV(n - 2NP), and PV(n) needs the P(n) about to be published,
          // so the parity is exact
          if (n >= (uint32_t)C::NP && !wait_bar(B.o_full + pbuf, ((n - C::NP) / C::NP) & 1, s_abort)) {
            ok = false;
            break;
          }
          // P = 2^(s - m) against the current reference maxima (masked: 0), written straight to the
          // P buffer and added to the row-sum shares; the vote asks whether any P exceeds 2^kTau
          // (then the tile is redone below with new references)
          uint32_t x[32];
          ptx::tmem_ld32(tmem + lane_addr + sb * kNR + r0, x);
          ptx::tmem_wait_ld();
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            if (u < nu) {
              uint32_t pk[4];
#pragma unroll
              for (int h = 0; h < 2; ++h) {
                const int i0 = 8 * u + 4 * h;
                const float4 m4 = reinterpret_cast<const float4 *>(mw + i0)[0];
                const float mm[4] = {m4.x, m4.y, m4.z, m4.w};
                float e[4];
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                  const int jr = i0 + q;
                  const float v = ptx::ex2(fmaf(__uint_as_float(x[i0 + q]), scale_log2, -mm[q]));
                  e[q] = (jr >= jmin && jr < jmax) ? v : 0.0f;
                  emax = fmaxf(emax, e[q]);
                  lp[i0 + q] += e[q];
                }
                pk[2 * h] = pack_bf16(e[0], e[1]);
                pk[2 * h + 1] = pack_bf16(e[2], e[3]);
              }
              *reinterpret_cast<uint4 *>(prow + (((4 * grp + u) ^ sw) << 4)) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
            }
          }
        }
        // the eight warps' votes, double-buffered by tile parity (NaN never wins fmaxf, and a
        // visible key of a row without a reference yet gives +inf)
        const uint32_t vote = __ballot_sync(0xffffffffu, !(emax <= kExpTau));
        if (lane == 0) {
          s_flag[(n & 1) * 8 + sw8] = vote;
          ptx::mbar_arrive(B.sm_sync);
        }
        if (!wait_bar(B.sm_sync, n & 1, s_abort)) { ok = false; break; }
        uint32_t anyv = 0;
#pragma unroll
        for (int k8 = 0; k8 < 8; ++k8) anyv |= s_flag[(n & 1) * 8 + k8];
        if (anyv != 0) {
          // new references: exact tile maxima per row (over this warp's 32 keys, then over the
          // group's four quadrants), from the scores read again
          if (active) {
            uint32_t x[32];
            ptx::tmem_ld32(tmem + lane_addr + sb * kNR + r0, x);
            ptx::tmem_wait_ld();
            float sv[32];
#pragma unroll
            for (int i = 0; i < 32; ++i)
              sv[i] = (i >= jmin && i < jmax) ? __uint_as_float(x[i]) * scale_log2 : -INFINITY;  // scale > 0
            s_red[qd * kNR + r0 + lane] = warp_transpose_reduce<true>(sv, lane);
          }
          __syncwarp();
          if (lane == 0) ptx::mbar_arrive(B.sm_sync2);
          if (!wait_bar(B.sm_sync2, nf & 1, s_abort)) { ok = false; break; }
          ++nf;
          if (active) {
            // this tile's P leaves the shares (a row without a reference had nothing yet)
            {
              uint32_t x[32];
              ptx::tmem_ld32(tmem + lane_addr + sb * kNR + r0, x);
              ptx::tmem_wait_ld();
#pragma unroll
              for (int i = 0; i < 32; ++i) {
                const float mo = mw[i];
                const float v = ptx::ex2(fmaf(__uint_as_float(x[i]), scale_log2, -mo));
                const float eo = (i >= jmin && i < jmax) ? v : 0.0f;
                lp[i] = mo == -INFINITY ? 0.0f : lp[i] - eo;
              }
            }
            __syncwarp();
            // every warp of the group derives the same new maxima and factors from the same values
            const int jl = r0 + lane;
            const float tmax = fmaxf(fmaxf(s_red[jl], s_red[kNR + jl]), fmaxf(s_red[2 * kNR + jl], s_red[3 * kNR + jl]));
            const float mo = mw[lane];
            const float mn = tmax > mo + kTau ? tmax : mo;
            fw[lane] = mn == mo ? 1.0f : (mo == -INFINITY ? 0.0f : ptx::ex2(mo - mn));
            const bool moved = mn != mo && mo != -INFINITY;
            mw[lane] = mn;
            __syncwarp();
            // P again against the new references: shares rescaled, P rewritten
            {
              uint32_t x[32];
              ptx::tmem_ld32(tmem + lane_addr + sb * kNR + r0, x);
              ptx::tmem_wait_ld();
#pragma unroll
              for (int u = 0; u < 4; ++u) {
                uint32_t pk[4];
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                  float e[4];
#pragma unroll
                  for (int q = 0; q < 4; ++q) {
                    const int i = 8 * u + 4 * h + q;
                    const float v = ptx::ex2(fmaf(__uint_as_float(x[i]), scale_log2, -mw[i]));
                    e[q] = (i >= jmin && i < jmax) ? v : 0.0f;
                    lp[i] = fmaf(lp[i], fw[i], e[q]);
                  }
                  pk[2 * h] = pack_bf16(e[0], e[1]);
                  pk[2 * h + 1] = pack_bf16(e[2], e[3]);
                }
                if (u < nu)
                  *reinterpret_cast<uint4 *>(prow + (((4 * grp + u) ^ sw) << 4)) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
              }
            }
            // this chunk's O^T columns, if they hold earlier tiles of the item, move to the new
            // references; the rescale needs PV(n-1) complete and precedes PV(n)
            if (t > 0 && __any_sync(0xffffffffu, moved)) {
              // PV(m) completes barrier o_full[m % NP] for the (m / NP)-th time; PV(n-1-NP) was
              // waited for (by this warp or, through the tile votes, by the other group) and
              // PV(n-1+NP) needs P(n-1+NP), so the parity names PV(n-1)
              if (!wait_bar(B.o_full + (n - 1) % C::NP, ((n - 1) / C::NP) & 1, s_abort)) { ok = false; break; }
              ptx::tc_fence_after();
#pragma unroll
              for (int c = 0; c < 2; ++c) {
                uint32_t y[16];
                ptx::tmem_ld16(tmem + lane_addr + o_col + r0 + 16 * c, y);
                ptx::tmem_wait_ld();
#pragma unroll
                for (int i = 0; i < 16; ++i) y[i] = __float_as_uint(__uint_as_float(y[i]) * fw[16 * c + i]);
                ptx::tmem_st16(tmem + lane_addr + o_col + r0 + 16 * c, y);
              }
              ptx::tmem_wait_st();
            }
          }
        }
        // S^T(n) has been read: its TMEM buffer may be overwritten by S^T(n+2); P(n) is published
        ptx::tc_fence_before();
        ptx::fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          ptx::mbar_arrive(B.s_empty + sb);
          ptx::mbar_arrive(B.p_full + pbuf);
        }
      }
      if (!ok) break;
      // ---- hand the item over to the epilogue warps: this quadrant's share of each row sum of
      // the chunk, and the reference maxima.  The epilogue of item li - 2 (same buffers) must be
      // done with them.
      const float lsh = warp_transpose_reduce<false>(lp, lane);
      if (!wait_bar(B.o_empty + ob, ((li >> 1) & 1) ^ 1, s_abort)) { ok = false; break; }
      s_hl[(ob * 4 + qd) * kNR + r0 + lane] = lsh;
      if (qd == 0) s_hm[ob * kNR + r0 + lane] = mw[lane];
      __syncwarp();
      if (lane == 0) ptx::mbar_arrive(B.ep_full + ob);
      ++li;
    }
    if (!ok && lane == 0) report(p.status, WISP_DEV_TIMEOUT, p.request_ids, 0);
  }

  // Teardown: every warp reports on an mbarrier that it is done with TMEM, and warp 1 frees the
  // TMEM once all have (a bounded wait; the warps' shared memory stays until the last one exits).
  __syncwarp();
  ptx::tc_fence_before();
  if (lane == 0) ptx::mbar_arrive(B.fin);
  if (warp == 1) {
    const long long t0 = clock64();
    while (!ptx::mbar_try_wait(B.fin, 0) && clock64() - t0 < kWaitCycles) {
    }
    __syncwarp();
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
// consecutive blocks (1, or 8 for a whole 128-token tile of consecutive blocks).
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

namespace {

// The four tensor maps of a (K pool, V pool, D, Hkv, num_blocks) are the same from step to step:
// the last few sets are kept, so that a launch does not encode them again.
struct PoolMaps {
  const void *k = nullptr, *v = nullptr;
  int D = 0, Hkv = 0, num_blocks = 0;
  alignas(64) CUtensorMap tk, tv, tk8, tv8;
};
constexpr int kMapCache = 8;
PoolMaps g_maps[kMapCache];
int g_maps_next = 0;
std::mutex g_maps_mu;

cudaError_t pool_maps(const AttnParams &p, PoolMaps *out) {
  std::lock_guard<std::mutex> lk(g_maps_mu);
  for (const PoolMaps &m : g_maps) {
    if (m.k == p.k_cache && m.v == p.v_cache && m.D == p.D && m.Hkv == p.Hkv && m.num_blocks == p.num_blocks) {
      *out = m;
      return cudaSuccess;
    }
  }
  PoolMaps m;
  m.k = p.k_cache;
  m.v = p.v_cache;
  m.D = p.D;
  m.Hkv = p.Hkv;
  m.num_blocks = p.num_blocks;
  cudaError_t e = encode_pool(&m.tk, p.k_cache, p.D, p.Hkv, p.num_blocks, 1);
  if (e == cudaSuccess) e = encode_pool(&m.tv, p.v_cache, p.D, p.Hkv, p.num_blocks, 1);
  if (e == cudaSuccess) e = encode_pool(&m.tk8, p.k_cache, p.D, p.Hkv, p.num_blocks, 8);
  if (e == cudaSuccess) e = encode_pool(&m.tv8, p.v_cache, p.D, p.Hkv, p.num_blocks, 8);
  if (e != cudaSuccess) return e;
  g_maps[g_maps_next] = m;
  g_maps_next = (g_maps_next + 1) % kMapCache;
  *out = m;
  return cudaSuccess;
}

}  // namespace

cudaError_t attn_tc_launch(const AttnParams &p, int grid, cudaStream_t s, bool pdl) {
  PoolMaps m;
  const cudaError_t e = pool_maps(p, &m);
  if (e != cudaSuccess) return e;
  const CUtensorMap &tk = m.tk, &tv = m.tv, &tk8 = m.tk8, &tv8 = m.tv8;
  // programmatic dependent launch: the CTAs' set-up overlaps the kernel before this one (the
  // planner), which the kernel waits for before it reads the plan
  cudaLaunchConfig_t cfg;
  std::memset(&cfg, 0, sizeof cfg);
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.gridDim = dim3((unsigned)grid);
  cfg.blockDim = dim3(kThreads);
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  if (p.D == 128) {
    cfg.dynamicSmemBytes = Cfg<128>::SMEM;
    return cudaLaunchKernelEx(&cfg, attn_tc_kernel<128>, p, tk, tv, tk8, tv8);
  }
  cfg.dynamicSmemBytes = Cfg<64>::SMEM;
  return cudaLaunchKernelEx(&cfg, attn_tc_kernel<64>, p, tk, tv, tk8, tv8);
}

}  // namespace wisp
