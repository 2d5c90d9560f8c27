// attn_tc.cu -- tensor-core paged GQA attention for the verification forward (bf16 KV).
//
// Same contract as attn_simt.cu (Sec. 4.4-4.5: request r's k+1 new queries over its
// L_total = L_cached + L_new paged keys, query j seeing keys 0..c_r + j), built for sm_103a:
//
//   * persistent CTAs, one per SM, walking the planner's work items round-robin;
//   * warp 0 (producer): copies the item's g*(k+1) query rows into shared memory in the
//     128-byte-swizzled K-major layout, then streams K and V tiles of 64 tokens with TMA
//     tiled loads, one 2 KB box per (16-token block, 64-wide half of the head dim), block
//     ids read from the block table; blocks past the item read as zeros (out-of-range box);
//   * warp 1 (one thread): issues tcgen05.mma -- S = Q K^T (M=128 query rows, N=64 tokens,
//     K=D) into a double-buffered TMEM tile, and O_tile = P V (M=128, N=D, K=64) into TMEM;
//   * warps 2-5 (softmax): thread i owns query row i (its TMEM lane); it reads S with
//     tcgen05.ld, applies the causal / chunk mask and the online softmax in base 2,
//     writes P (bf16, swizzled) for the PV product, and folds each O_tile into its fp32
//     registers (O = O * 2^(m_old - m_new) + O_tile);
//   * mbarriers hand every buffer between roles; every wait is bounded in time and an
//     expired wait sets a device status (WISP_DEV_TIMEOUT) and drains the CTA.
// Rows past g*(k+1) are padding: they are computed from stale data and never written.
#include "attn.cuh"
#include "sm100_ptx.cuh"

#include <cudaTypedefs.h>

namespace wisp {

namespace {

constexpr int kBN = 64;             // KV tokens per tile
constexpr int kM = 128;             // MMA rows
constexpr int kThreads = 192;       // warp 0 producer, warp 1 MMA, warps 2-5 softmax
constexpr uint32_t kTmemCols = 256; // S[2] at columns 0 / 64, O at column 128
constexpr long long kWaitCycles = 4000000000LL;  // about two seconds: a wait that long is a failure

template <int D>
struct Cfg {
  static constexpr int HALVES = D / 64;
  static constexpr int Q_BYTES = kM * D * 2;
  static constexpr int KV_TILE = kBN * D * 2;  // K (or V) of one tile
  static constexpr int NSTAGE = D == 128 ? 4 : 6;
  static constexpr int P_BYTES = kM * kBN * 2;
  static constexpr int OFF_Q = 0;
  static constexpr int OFF_K = OFF_Q + 2 * Q_BYTES;
  static constexpr int OFF_V = OFF_K + NSTAGE * KV_TILE;
  static constexpr int OFF_P = OFF_V + NSTAGE * KV_TILE;
  static constexpr int OFF_BAR = OFF_P + 2 * P_BYTES;
  static constexpr int N_BAR = 2 * NSTAGE + 13;
  static constexpr int OFF_MISC = OFF_BAR + N_BAR * 8;
  static constexpr int SMEM = OFF_MISC + 64 + 1024;  // + slack to align the base to 1024
};

constexpr uint32_t IDESC_S = ptx::idesc_bf16_f32(kM, kBN, false);

struct Bars {
  uint64_t *kv_full, *kv_empty, *q_full, *q_empty, *s_full, *s_empty, *p_full, *o_full, *o_empty, *mma_done;
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
  uint32_t *s_tmem = reinterpret_cast<uint32_t *>(smem + C::OFF_MISC);
  volatile int *s_abort = reinterpret_cast<volatile int *>(smem + C::OFF_MISC + 4);

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
    for (int it = blockIdx.x; it < n_items && ok; it += gridDim.x) {
      const WorkItem w = p.items[it];
      if (!item_ok(p, w)) continue;
      const int qb = li & 1;
      if (!wait_bar(B.q_empty + qb, ((li >> 1) & 1) ^ 1, s_abort)) { ok = false; break; }
      ++li;
      // query rows of this KV head -> Q[qb], row rho = j*g + hh, 128B-swizzled K-major halves
      const uint16_t *qg = static_cast<const uint16_t *>(p.q);
      uint8_t *qs = smem + C::OFF_Q + qb * C::Q_BYTES;
      constexpr int CPR = D / 8;  // 16-byte chunks per row
      for (int c = lane; c < w.rows * CPR; c += 32) {
        const int row = c / CPR, cc = c % CPR;
        const int j = row / g, hh = row % g;
        const uint4 v = __ldg(reinterpret_cast<const uint4 *>(
                                  qg + ((int64_t)(w.q0 + j) * p.Hq + w.h * g + hh) * D) + cc);
        *reinterpret_cast<uint4 *>(qs + (cc >> 3) * (kM * 128) + row * 128 + (((cc & 7) ^ (row & 7)) << 4)) = v;
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
      auto issue_pv = [&](uint32_t m) -> bool {
        const int pb = m & 1;
        if (!wait_bar(B.p_full + pb, (m >> 1) & 1, s_abort)) return false;
        if (!wait_bar(B.o_empty, (m & 1) ^ 1, s_abort)) return false;
        ptx::tc_fence_after();
        const int st = (int)(m % C::NSTAGE);
        const uint32_t pa = sbase + C::OFF_P + pb * C::P_BYTES;
        const uint32_t va = sbase + C::OFF_V + st * C::KV_TILE;
#pragma unroll
        for (int ks = 0; ks < kBN / 16; ++ks) {
          const uint64_t a = ptx::sdesc_sw128(pa + ks * 32, 16, 1024);
          const uint64_t b = ptx::sdesc_sw128(va + ks * 16 * 128, kBN * 128, 1024);
          ptx::umma_f16(tmem + 128, a, b, IDESC_PV, ks > 0);
        }
        ptx::umma_commit(B.o_full);
        ptx::umma_commit(B.kv_empty + st);
        return true;
      };
      for (int it = blockIdx.x; it < n_items && ok; it += gridDim.x) {
        const WorkItem w = p.items[it];
        if (!item_ok(p, w)) continue;
        const int qb = li & 1;
        if (!wait_bar(B.q_full + qb, (li >> 1) & 1, s_abort)) { ok = false; break; }
        ++li;
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
          if (t > 0 && !issue_pv(n - 1)) { ok = false; break; }
        }
        if (ok && !issue_pv(n - 1)) ok = false;
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
    const int qd = warp & 3;
    const int row = qd * 32 + lane;
    const uint32_t lane_addr = (uint32_t)(qd * 32) << 16;
    const float scale_log2 = 1.4426950408889634f / sqrtf((float)D);
    uint32_t n = 0;
    bool ok = true;
    for (int it = blockIdx.x; it < n_items && ok; it += gridDim.x) {
      const WorkItem w = p.items[it];
      if (!item_ok(p, w)) continue;
      const bool wact = qd * 32 < w.rows;
      const bool ract = row < w.rows;
      const int jq = row / g;
      const int vis = w.ctx + jq;  // last key position this row may see
      float O[D];
#pragma unroll
      for (int d = 0; d < D; ++d) O[d] = 0.0f;
      float m = -INFINITY, l = 0.0f, a_prev = 0.0f;

      auto consume_o = [&](uint32_t mi, float alpha) -> bool {
        if (!wait_bar(B.o_full, mi & 1, s_abort)) return false;
        ptx::tc_fence_after();
        if (wact) {
#pragma unroll
          for (int c = 0; c < D / 32; ++c) {
            uint32_t x[32];
            ptx::tmem_ld32(tmem + lane_addr + 128 + c * 32, x);
            ptx::tmem_wait_ld();
#pragma unroll
            for (int i = 0; i < 32; ++i) O[c * 32 + i] = fmaf(O[c * 32 + i], alpha, __uint_as_float(x[i]));
          }
        }
        ptx::tc_fence_before();
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive(B.o_empty);
        return true;
      };

      const int ntiles = (w.t1 - w.t0 + kBN - 1) / kBN;
      for (int t = 0; t < ntiles; ++t, ++n) {
        const int sb = n & 1;
        if (!wait_bar(B.s_full + sb, (n >> 1) & 1, s_abort)) { ok = false; break; }
        ptx::tc_fence_after();
        float sv[kBN];
        if (wact) {
          uint32_t x[32];
          ptx::tmem_ld32(tmem + lane_addr + sb * 64, x);
          ptx::tmem_wait_ld();
#pragma unroll
          for (int i = 0; i < 32; ++i) sv[i] = __uint_as_float(x[i]);
          ptx::tmem_ld32(tmem + lane_addr + sb * 64 + 32, x);
          ptx::tmem_wait_ld();
#pragma unroll
          for (int i = 0; i < 32; ++i) sv[32 + i] = __uint_as_float(x[i]);
        }
        ptx::tc_fence_before();
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive(B.s_empty + sb);
        float a = 0.0f;
        if (wact) {
          const int tok0 = w.t0 + t * kBN;
          float mx = -INFINITY;
#pragma unroll
          for (int i = 0; i < kBN; ++i) {
            const int tok = tok0 + i;
            const bool valid = tok < w.t1 && tok <= vis;
            sv[i] = valid ? sv[i] * scale_log2 : -INFINITY;
            mx = fmaxf(mx, sv[i]);
          }
          const float m_new = fmaxf(m, mx);
          const float m_use = m_new == -INFINITY ? 0.0f : m_new;
          a = ptx::ex2(m - m_use);
          float sum = 0.0f;
          uint8_t *prow = smem + C::OFF_P + sb * C::P_BYTES + row * 128;
#pragma unroll
          for (int c = 0; c < kBN / 8; ++c) {
            float e[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) {
              e[i] = ptx::ex2(sv[c * 8 + i] - m_use);
              sum += e[i];
            }
            uint4 v;
            v.x = pack_bf16(e[0], e[1]);
            v.y = pack_bf16(e[2], e[3]);
            v.z = pack_bf16(e[4], e[5]);
            v.w = pack_bf16(e[6], e[7]);
            *reinterpret_cast<uint4 *>(prow + ((c ^ (row & 7)) << 4)) = v;
          }
          l = l * a + sum;
          m = m_new;
        }
        ptx::fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive(B.p_full + sb);
        if (t > 0 && !consume_o(n - 1, a_prev)) { ok = false; break; }
        a_prev = a;
      }
      if (!ok || !consume_o(n - 1, a_prev)) { ok = false; break; }

      // epilogue: normalised bf16 output, or (acc, m, l) partials of a split item
      if (ract) {
        const int hh = row % g;
        if (w.poff < 0) {
          const float inv = 1.0f / l;
          uint16_t *og = static_cast<uint16_t *>(p.out) + ((int64_t)(w.q0 + jq) * p.Hq + w.h * g + hh) * D;
#pragma unroll
          for (int c = 0; c < D / 8; ++c) {
            uint4 v;
            v.x = pack_bf16(O[8 * c + 0] * inv, O[8 * c + 1] * inv);
            v.y = pack_bf16(O[8 * c + 2] * inv, O[8 * c + 3] * inv);
            v.z = pack_bf16(O[8 * c + 4] * inv, O[8 * c + 5] * inv);
            v.w = pack_bf16(O[8 * c + 6] * inv, O[8 * c + 7] * inv);
            reinterpret_cast<uint4 *>(og)[c] = v;
          }
        } else {
          float *part = p.partials + w.poff;
#pragma unroll
          for (int c = 0; c < D / 4; ++c) {
            reinterpret_cast<float4 *>(part + (int64_t)row * D)[c] =
                make_float4(O[4 * c], O[4 * c + 1], O[4 * c + 2], O[4 * c + 3]);
          }
          part[w.rows * D + row] = m;
          part[w.rows * D + w.rows + row] = l;
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
