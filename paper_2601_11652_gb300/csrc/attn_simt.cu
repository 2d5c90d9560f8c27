// attn_simt.cu -- CUDA-core (FFMA) paged GQA attention for the verification forward.
//
// Computes, for one work item (request r, KV head h, keys [t0, t1)), the attention of
// the g * (k_r + 1) query rows that read KV head h (Sec. 4.4-4.5: k+1 new queries over
// L_total = L_cached + L_new keys, query j sees keys 0..c_r + j).  fp32 accumulation
// and an online (running max / running sum) softmax in base 2.  Items that cover a
// whole sequence write the normalised output; split items write (acc, m, l) partials
// that attn_combine_kernel merges.  This kernel serves fp32 inputs (where tensor cores
// would round operands) and D = 64; bf16 D = 128 uses the tcgen05 kernel.
#include "attn.cuh"

namespace wisp {

namespace {

constexpr int kTile = 32;
constexpr int kWarps = 4;

template <typename T>
__device__ __forceinline__ float ld(const T *p, int64_t i);
template <>
__device__ __forceinline__ float ld<float>(const float *p, int64_t i) { return __ldg(p + i); }
template <>
__device__ __forceinline__ float ld<uint16_t>(const uint16_t *p, int64_t i) {
  return bf16_bits_to_float(__ldg(p + i));
}

template <typename T>
__device__ __forceinline__ void st(T *p, int64_t i, float v);
template <>
__device__ __forceinline__ void st<float>(float *p, int64_t i, float v) { p[i] = v; }
template <>
__device__ __forceinline__ void st<uint16_t>(uint16_t *p, int64_t i, float v) {
  __nv_bfloat16 b = __float2bfloat16_rn(v);
  p[i] = *reinterpret_cast<uint16_t *>(&b);
}

}  // namespace

template <typename T, int D>
__global__ void __launch_bounds__(kWarps * 32) attn_simt_kernel(const AttnParams p) {
  extern __shared__ float smem[];
  const PlanHeader *hdr = p.header;
  const int item_idx = blockIdx.x;
  if (item_idx >= hdr->n_items) return;
  const WorkItem it = p.items[item_idx];
  if (it.r < 0 || it.r >= p.B || p.req_flag[it.r] != REQ_OK) return;
  const int g = p.Hq / p.Hkv;
  const int R = it.rows;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;

  float *Qs = smem;                       // [R][D]
  float *Acc = Qs + R * D;                // [R][D]
  float *Ms = Acc + R * D;                // [R]
  float *Ls = Ms + R;                     // [R]
  float *Ks = Ls + R;                     // [kTile][D+1]
  float *Vs = Ks + kTile * (D + 1);       // [kTile][D]
  __shared__ int s_bad;

  const T *q = static_cast<const T *>(p.q);
  const T *kc = static_cast<const T *>(p.k_cache);
  const T *vc = static_cast<const T *>(p.v_cache);
  if (threadIdx.x == 0) s_bad = 0;
  for (int i = threadIdx.x; i < R * D; i += blockDim.x) {
    const int rho = i / D, d = i % D;
    const int j = rho / g, hh = rho % g;
    Qs[i] = ld<T>(q, ((int64_t)(it.q0 + j) * p.Hq + it.h * g + hh) * D + d);
    Acc[i] = 0.0f;
  }
  for (int i = threadIdx.x; i < R; i += blockDim.x) {
    Ms[i] = -INFINITY;
    Ls[i] = 0.0f;
  }
  const float scale_log2 = 1.4426950408889634f / sqrtf((float)D);
  const int32_t *bt = p.block_tables + (int64_t)it.r * p.max_blocks_per_seq;

  for (int ts = it.t0; ts < it.t1; ts += kTile) {
    __syncthreads();
    // stage K/V of tokens ts .. ts + kTile - 1 (fp32) through the block table
    for (int i = threadIdx.x; i < kTile * D; i += blockDim.x) {
      const int tt = i / D, d = i % D;
      const int t = ts + tt;
      float kv = 0.0f, vv = 0.0f;
      if (t < it.t1) {
        const int32_t blk = bt[t / 16];
        if (blk < 0 || blk >= p.num_blocks) {
          s_bad = 1;
        } else {
          const int64_t src = (((int64_t)blk * p.Hkv + it.h) * 16 + (t % 16)) * D + d;
          kv = ld<T>(kc, src);
          vv = ld<T>(vc, src);
        }
      }
      Ks[tt * (D + 1) + d] = kv;
      Vs[tt * D + d] = vv;
    }
    __syncthreads();
    if (s_bad) break;
    const int t = ts + lane;
    for (int rho = warp; rho < R; rho += kWarps) {
      const int j = rho / g;
      const bool valid = t < it.t1 && t <= it.ctx + j;
      float s = -INFINITY;
      if (valid) {
        float a = 0.0f;
        const float *qr = Qs + rho * D;
        const float *kr = Ks + lane * (D + 1);
#pragma unroll 16
        for (int d = 0; d < D; ++d) a = fmaf(qr[d], kr[d], a);
        s = a * scale_log2;
      }
      float mx = s;
      for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
      const float m_old = Ms[rho];
      const float m_new = fmaxf(m_old, mx);
      if (m_new == -INFINITY) continue;  // no visible key yet for this row
      const float pe = valid ? exp2f(s - m_new) : 0.0f;
      const float alpha = exp2f(m_old - m_new);
      float sum = pe;
      for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
      float acc[D / 32];
#pragma unroll
      for (int dd = 0; dd < D / 32; ++dd) acc[dd] = Acc[rho * D + lane + 32 * dd] * alpha;
#pragma unroll 4
      for (int tt = 0; tt < kTile; ++tt) {
        const float pt = __shfl_sync(0xffffffffu, pe, tt);
#pragma unroll
        for (int dd = 0; dd < D / 32; ++dd) acc[dd] = fmaf(pt, Vs[tt * D + lane + 32 * dd], acc[dd]);
      }
#pragma unroll
      for (int dd = 0; dd < D / 32; ++dd) Acc[rho * D + lane + 32 * dd] = acc[dd];
      __syncwarp();
      if (lane == 0) {
        Ls[rho] = Ls[rho] * alpha + sum;
        Ms[rho] = m_new;
      }
      __syncwarp();
    }
  }
  __syncthreads();
  if (s_bad) {
    if (threadIdx.x == 0) report(p.status, WISP_DEV_BAD_BLOCK, p.request_ids, it.r);
    return;
  }
  if (it.poff < 0) {
    T *out = static_cast<T *>(p.out);
    for (int i = threadIdx.x; i < R * D; i += blockDim.x) {
      const int rho = i / D, d = i % D;
      const int j = rho / g, hh = rho % g;
      st<T>(out, ((int64_t)(it.q0 + j) * p.Hq + it.h * g + hh) * D + d, Acc[i] / Ls[rho]);
    }
  } else {
    float *part = p.partials + it.poff;  // [R][D] acc, then [R] m, then [R] l
    for (int i = threadIdx.x; i < R * D; i += blockDim.x) part[i] = Acc[i];
    for (int i = threadIdx.x; i < R; i += blockDim.x) {
      part[R * D + i] = Ms[i];
      part[R * D + R + i] = Ls[i];
    }
  }
}

static size_t attn_simt_smem_bytes(int R, int D) {
  return sizeof(float) * ((size_t)2 * R * D + 2 * R + kTile * (D + 1) + kTile * D);
}

// Merge the split partials of one (request, KV head): O = sum_c acc_c 2^(m_c - m) / sum_c l_c 2^(m_c - m).
// One warp per query row: the chunk weights are formed once per row, each lane owns D/32
// consecutive output elements and reads the chunk accumulators as 8- or 16-byte vectors.
template <typename T, int D>
__global__ void __launch_bounds__(128) attn_combine_kernel(const AttnParams p) {
  constexpr int PER = D / 32;  // 2 or 4 floats per lane
  const int pair = blockIdx.x;
  const int r = pair / p.Hkv, h = pair % p.Hkv;
  if (r >= p.B || p.req_flag[r] != REQ_OK) return;
  const int chunks = p.req_chunks[r];
  if (chunks <= 1) return;
  const WorkItem *items = p.items + p.req_item_begin[r] + h * chunks;
  const int R = items[0].rows;
  const int q0 = items[0].q0;
  const int g = p.Hq / p.Hkv;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  T *out = static_cast<T *>(p.out);
  for (int rho = warp; rho < R; rho += 4) {
    float m = -INFINITY;
    for (int c = lane; c < chunks; c += 32) m = fmaxf(m, p.partials[items[c].poff + R * D + rho]);
    for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
    float acc[PER];
#pragma unroll
    for (int i = 0; i < PER; ++i) acc[i] = 0.0f;
    float den = 0.0f;
    for (int c = 0; c < chunks; ++c) {
      const float *part = p.partials + items[c].poff;
      const float mc = part[R * D + rho];
      if (mc == -INFINITY) continue;
      const float w = exp2f(mc - m);
      den = fmaf(part[R * D + R + rho], w, den);
      const float *src = part + (int64_t)rho * D + lane * PER;
      if (PER == 4) {
        const float4 v = *reinterpret_cast<const float4 *>(src);
        acc[0] = fmaf(v.x, w, acc[0]);
        acc[1] = fmaf(v.y, w, acc[1]);
        acc[2] = fmaf(v.z, w, acc[2]);
        acc[3] = fmaf(v.w, w, acc[3]);
      } else {
        const float2 v = *reinterpret_cast<const float2 *>(src);
        acc[0] = fmaf(v.x, w, acc[0]);
        acc[1] = fmaf(v.y, w, acc[1]);
      }
    }
    const float inv = 1.0f / den;
    const int j = rho / g, hh = rho % g;
    const int64_t o0 = ((int64_t)(q0 + j) * p.Hq + h * g + hh) * D + lane * PER;
#pragma unroll
    for (int i = 0; i < PER; ++i) st<T>(out, o0 + i, acc[i] * inv);
  }
}

template <typename T, int D>
static cudaError_t simt_attr() {
  return cudaFuncSetAttribute(attn_simt_kernel<T, D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)attn_simt_smem_bytes(kMaxRowsPerHead, D));
}

cudaError_t attn_simt_setup() {
  cudaError_t e = simt_attr<float, 64>();
  if (e == cudaSuccess) e = simt_attr<float, 128>();
  if (e == cudaSuccess) e = simt_attr<uint16_t, 64>();
  if (e == cudaSuccess) e = simt_attr<uint16_t, 128>();
  return e;
}

cudaError_t attn_simt_launch(const AttnParams &p, bool bf16, int grid, cudaStream_t s) {
  const size_t smem = attn_simt_smem_bytes(kMaxRowsPerHead, p.D);
  if (p.D == 64) {
    if (bf16) attn_simt_kernel<uint16_t, 64><<<grid, kWarps * 32, smem, s>>>(p);
    else attn_simt_kernel<float, 64><<<grid, kWarps * 32, smem, s>>>(p);
  } else {
    if (bf16) attn_simt_kernel<uint16_t, 128><<<grid, kWarps * 32, smem, s>>>(p);
    else attn_simt_kernel<float, 128><<<grid, kWarps * 32, smem, s>>>(p);
  }
  return cudaGetLastError();
}

cudaError_t attn_combine_launch(const AttnParams &p, bool bf16, cudaStream_t s) {
  const unsigned grid = (unsigned)((int64_t)p.B * p.Hkv);
  if (p.D == 64) {
    if (bf16) attn_combine_kernel<uint16_t, 64><<<grid, 128, 0, s>>>(p);
    else attn_combine_kernel<float, 64><<<grid, 128, 0, s>>>(p);
  } else {
    if (bf16) attn_combine_kernel<uint16_t, 128><<<grid, 128, 0, s>>>(p);
    else attn_combine_kernel<float, 128><<<grid, 128, 0, s>>>(p);
  }
  return cudaGetLastError();
}

}  // namespace wisp
