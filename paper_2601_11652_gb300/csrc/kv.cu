// kv.cu -- paged KV-cache maintenance around the verification step (include/wisp_kv.h).
//
// Sec. 4.5: per-session KV lives in fixed-size pages (PageAttention) and a prefix cache that is
// updated in place, so a verification forwards only the new block.  Three kernels:
//   kv_reserve_kernel (one CTA): validates the lengths, counts each request's missing pages among
//     those covering tokens 0 .. c + k, serves requests in order from the top of the device-side
//     free stack (block-wide scans, so the assignment is deterministic), and maps every new K/V row
//     to its (request, position);
//   kv_append_kernel: one warp per (new row, KV head) copies the row into its page slot;
//   kv_commit_kernel (one CTA): c <- c + 1 + L (Eq. 2's L), and the pages past the new length
//     among those the step could use go back on the free stack in table order.
#include "common.cuh"

#include <cstring>

#include "wisp_kv.h"

namespace wisp {

namespace {

constexpr int kThreads = 1024;
constexpr int kPage = 16;

struct KvParams {
  int B, Hkv, D, max_blocks, num_blocks, total_rows, esize;
  const int64_t *request_ids;
  const int32_t *draft_lens;
  int32_t *context_lens, *block_tables, *free_blocks, *free_count;
  char *k_cache, *v_cache;
  const char *k_new, *v_new;
  const int32_t *accepted_len;
  DeviceStatus *status;
  int32_t *row_req, *row_pos;  // [total_rows]: request of a new row (-1: skipped) and its position
};

__device__ __forceinline__ int64_t min64(int64_t a, int64_t b) { return a < b ? a : b; }

// Exclusive block-wide prefix sum; *total receives the block's sum.
__device__ int64_t scan_excl(int64_t v, int64_t *s_warp, int64_t *total) {
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  int64_t x = v;
  for (int d = 1; d < 32; d <<= 1) {
    const int64_t o = __shfl_up_sync(0xffffffffu, x, d);
    if (lane >= d) x += o;
  }
  if (lane == 31) s_warp[w] = x;
  __syncthreads();
  if (w == 0) {
    int64_t t = s_warp[lane];
    for (int d = 1; d < 32; d <<= 1) {
      const int64_t o = __shfl_up_sync(0xffffffffu, t, d);
      if (lane >= d) t += o;
    }
    s_warp[lane] = t;
  }
  __syncthreads();
  const int64_t incl = x + (w > 0 ? s_warp[w - 1] : 0);
  *total = s_warp[31];
  __syncthreads();
  return incl - v;
}

// Block-wide maximum.
__device__ int64_t block_max(int64_t v, int64_t *s_warp) {
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  for (int d = 16; d > 0; d >>= 1) v = max(v, __shfl_xor_sync(0xffffffffu, v, d));
  if (lane == 0) s_warp[w] = v;
  __syncthreads();
  int64_t m = s_warp[0];
  for (int i = 1; i < 32; ++i) m = max(m, s_warp[i]);
  __syncthreads();
  return m;
}

__global__ void __launch_bounds__(kThreads) kv_reserve_kernel(const KvParams p) {
  __shared__ int64_t s_warp[32];
  int64_t F = *p.free_count;
  if (F < 0 || F > p.num_blocks) {  // inconsistent pool: serve nobody
    if (threadIdx.x == 0) report(p.status, WISP_DEV_BAD_BLOCK, p.request_ids, -1);
    F = 0;
  }
  const int64_t cap = (int64_t)p.max_blocks * kPage;
  int64_t carry_need = 0, carry_rows = 0, taken = 0;
  for (int base = 0; base < p.B; base += kThreads) {
    const int r = base + threadIdx.x;
    int64_t k = 0, c = 0, need = 0;
    int bad = 0;
    if (r < p.B) {
      k = p.draft_lens[r];
      c = p.context_lens[r];
      if (k < 0) { bad = WISP_DEV_BAD_LENGTH; k = 0; }
      if (!bad && (c < 0 || c + k + 1 > cap)) bad = WISP_DEV_BAD_LENGTH;
      if (!bad) {
        const int32_t *row = p.block_tables + (int64_t)r * p.max_blocks;
        const int64_t nb = (c + k + 1 + kPage - 1) / kPage;
        for (int64_t b = 0; b < nb; ++b) {
          const int32_t id = row[b];
          if (id < 0) ++need;
          else if (id >= p.num_blocks) bad = WISP_DEV_BAD_BLOCK;
        }
      }
      if (bad) need = 0;
    }
    int64_t tot_need, tot_rows;
    const int64_t before = carry_need + scan_excl(need, s_warp, &tot_need);
    const int64_t q0 = carry_rows + scan_excl(r < p.B ? k + 1 : 0, s_warp, &tot_rows);
    // served requests form a prefix of the valid ones: `before + need` only grows with r
    const bool served = r < p.B && !bad && before + need <= F;
    if (r < p.B) {
      if (bad) report(p.status, bad, p.request_ids, r);
      else if (!served) report(p.status, WISP_DEV_NO_BLOCKS, p.request_ids, r);
      if (served) {
        // pop from the top of the stack: this request's missing pages, in table order, take
        // entries F-1-before, F-2-before, ...
        int32_t *row = p.block_tables + (int64_t)r * p.max_blocks;
        const int64_t nb = (c + k + 1 + kPage - 1) / kPage;
        int64_t t = 0;
        for (int64_t b = 0; b < nb; ++b)
          if (row[b] < 0) row[b] = p.free_blocks[F - 1 - before - t++];
      }
      for (int64_t j = 0; j <= k && q0 + j < p.total_rows; ++j) {
        p.row_req[q0 + j] = served ? r : -1;
        p.row_pos[q0 + j] = (int32_t)(c + j);
      }
    }
    taken = max(taken, block_max(served ? before + need : 0, s_warp));
    carry_need += tot_need;
    carry_rows += tot_rows;
  }
  if (threadIdx.x == 0) {
    *p.free_count = (int32_t)(F - taken);
    if (carry_rows != p.total_rows) atomicCAS(&p.status->code, 0, (int32_t)WISP_DEV_BAD_LENGTH);
  }
}

// One warp per (new row, KV head): the row's D values into their page slot (16-byte vectors).
__global__ void __launch_bounds__(256) kv_append_kernel(const KvParams p) {
  const int lane = threadIdx.x & 31;
  const int64_t nwarps = (int64_t)gridDim.x * (blockDim.x >> 5);
  const int nvec = p.D * p.esize / 16;
  for (int64_t wi = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); wi < (int64_t)p.total_rows * p.Hkv;
       wi += nwarps) {
    const int64_t row = wi / p.Hkv;
    const int h = (int)(wi % p.Hkv);
    const int r = p.row_req[row];
    if (r < 0) continue;
    const int pos = p.row_pos[row];
    const int32_t page = p.block_tables[(int64_t)r * p.max_blocks + pos / kPage];
    if (page < 0 || page >= p.num_blocks) {  // a page id from the free stack outside the pool
      if (lane == 0) report(p.status, WISP_DEV_BAD_BLOCK, p.request_ids, r);
      continue;
    }
    const int64_t dst = ((((int64_t)page * p.Hkv + h) * kPage) + pos % kPage) * p.D * p.esize;
    const int64_t src = (row * p.Hkv + h) * (int64_t)p.D * p.esize;
    for (int v = lane; v < nvec; v += 32) {
      reinterpret_cast<uint4 *>(p.k_cache + dst)[v] = __ldg(reinterpret_cast<const uint4 *>(p.k_new + src) + v);
      reinterpret_cast<uint4 *>(p.v_cache + dst)[v] = __ldg(reinterpret_cast<const uint4 *>(p.v_new + src) + v);
    }
  }
}

__global__ void __launch_bounds__(kThreads) kv_commit_kernel(const KvParams p) {
  __shared__ int64_t s_warp[32];
  const int64_t F = *p.free_count;
  if (F < 0 || F > p.num_blocks) {  // inconsistent pool: release nothing
    if (threadIdx.x == 0) report(p.status, WISP_DEV_BAD_BLOCK, p.request_ids, -1);
    return;
  }
  int64_t carry = 0;
  for (int base = 0; base < p.B; base += kThreads) {
    const int r = base + threadIdx.x;
    int64_t rel = 0, keep = 0, used = 0, cnew = 0;
    int bad = 0;
    if (r < p.B) {
      const int64_t k = p.draft_lens[r], c = p.context_lens[r], L = p.accepted_len[r];
      if (k < 0 || c < 0 || L < 0 || L > k || c + k + 1 > (int64_t)p.max_blocks * kPage) bad = WISP_DEV_BAD_LENGTH;
      if (!bad) {
        cnew = c + 1 + L;
        keep = (cnew + kPage - 1) / kPage;
        used = (c + k + 1 + kPage - 1) / kPage;
        const int32_t *row = p.block_tables + (int64_t)r * p.max_blocks;
        for (int64_t b = keep; b < used; ++b) rel += row[b] >= 0 ? 1 : 0;
      } else {
        report(p.status, bad, p.request_ids, r);
      }
    }
    int64_t tot;
    const int64_t at = F + carry + scan_excl(rel, s_warp, &tot);
    if (r < p.B && !bad) {
      int32_t *row = p.block_tables + (int64_t)r * p.max_blocks;
      int64_t t = 0;
      for (int64_t b = keep; b < used; ++b) {
        if (row[b] >= 0) {
          if (at + t >= p.num_blocks) {  // more pages than the pool holds: the caller's state is broken
            report(p.status, WISP_DEV_BAD_BLOCK, p.request_ids, r);
            break;
          }
          p.free_blocks[at + t++] = row[b];
          row[b] = -1;
        }
      }
      p.context_lens[r] = (int32_t)cnew;
    }
    carry += tot;
  }
  if (threadIdx.x == 0) *p.free_count = (int32_t)min64(F + carry, p.num_blocks);
}

struct KvLayout {
  size_t status = 0, row_req = 0, row_pos = 0, total = 0;
};

KvLayout kv_layout(const wisp_kv_args *a) {
  KvLayout L;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t at = off;
    off = (off + bytes + 255) & ~(size_t)255;
    return at;
  };
  L.status = take(sizeof(DeviceStatus));
  L.row_req = take(sizeof(int32_t) * (size_t)a->total_q_rows);
  L.row_pos = take(sizeof(int32_t) * (size_t)a->total_q_rows);
  L.total = off;
  return L;
}

bool al16(const void *p) { return ((uintptr_t)p & 15) == 0; }

wisp_status kv_check(const wisp_kv_args *a, bool need_new, bool need_accepted) {
  if (!a) return WISP_ERR_INVALID_ARG;
  if (a->B < 0 || a->Hkv <= 0 || a->total_q_rows < a->B || a->num_blocks <= 0 || a->max_blocks_per_seq <= 0)
    return WISP_ERR_INVALID_ARG;
  if (a->D != 64 && a->D != 128) return WISP_ERR_UNSUPPORTED;
  if (a->block_size != kPage) return WISP_ERR_UNSUPPORTED;
  if (a->kv_dtype != WISP_F32 && a->kv_dtype != WISP_BF16) return WISP_ERR_INVALID_ARG;
  if (a->B == 0) return WISP_OK;
  if (!a->draft_lens || !a->context_lens || !a->block_tables || !a->free_blocks || !a->free_count)
    return WISP_ERR_INVALID_ARG;
  if (need_new && (!a->k_cache || !a->v_cache || !a->k_new || !a->v_new)) return WISP_ERR_INVALID_ARG;
  if (need_new && (!al16(a->k_cache) || !al16(a->v_cache) || !al16(a->k_new) || !al16(a->v_new)))
    return WISP_ERR_INVALID_ARG;
  if (need_accepted && !a->accepted_len) return WISP_ERR_INVALID_ARG;
  if ((int64_t)a->max_blocks_per_seq * kPage > INT32_MAX / 2) return WISP_ERR_UNSUPPORTED;
  return WISP_OK;
}

KvParams kv_params(const wisp_kv_args *a, void *ws, const KvLayout &L) {
  KvParams p;
  std::memset(&p, 0, sizeof p);
  p.B = a->B;
  p.Hkv = a->Hkv;
  p.D = a->D;
  p.max_blocks = a->max_blocks_per_seq;
  p.num_blocks = a->num_blocks;
  p.total_rows = a->total_q_rows;
  p.esize = a->kv_dtype == WISP_BF16 ? 2 : 4;
  p.request_ids = a->request_ids;
  p.draft_lens = a->draft_lens;
  p.context_lens = a->context_lens;
  p.block_tables = a->block_tables;
  p.free_blocks = a->free_blocks;
  p.free_count = a->free_count;
  p.k_cache = static_cast<char *>(a->k_cache);
  p.v_cache = static_cast<char *>(a->v_cache);
  p.k_new = static_cast<const char *>(a->k_new);
  p.v_new = static_cast<const char *>(a->v_new);
  p.accepted_len = a->accepted_len;
  p.status = reinterpret_cast<DeviceStatus *>(static_cast<char *>(ws) + L.status);
  p.row_req = reinterpret_cast<int32_t *>(static_cast<char *>(ws) + L.row_req);
  p.row_pos = reinterpret_cast<int32_t *>(static_cast<char *>(ws) + L.row_pos);
  return p;
}

wisp_status kv_ws_ok(void *ws, size_t bytes, const KvLayout &L) {
  return !ws || ((uintptr_t)ws & 255) != 0 || bytes < L.total ? WISP_ERR_WORKSPACE : WISP_OK;
}

}  // namespace

}  // namespace wisp

using namespace wisp;

extern "C" {

size_t wisp_kv_workspace_size(const wisp_kv_args *kv) {
  if (kv_check(kv, false, false) != WISP_OK) return 0;
  return kv_layout(kv).total;
}

wisp_status wisp_kv_reserve_append(const wisp_kv_args *kv, void *ws, size_t ws_bytes, void *stream) {
  wisp_status st = kv_check(kv, true, false);
  if (st != WISP_OK) return st;
  const KvLayout L = kv_layout(kv);
  if ((st = kv_ws_ok(ws, ws_bytes, L)) != WISP_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const KvParams p = kv_params(kv, ws, L);
  if (cudaMemsetAsync(p.status, 0, sizeof(DeviceStatus), s) != cudaSuccess) return WISP_ERR_CUDA;
  if (kv->B == 0) return WISP_OK;
  kv_reserve_kernel<<<1, kThreads, 0, s>>>(p);
  const int64_t warps = (int64_t)kv->total_q_rows * kv->Hkv;
  const int64_t blocks = (warps + 7) / 8;
  kv_append_kernel<<<(unsigned)(blocks < 4096 ? blocks : 4096), 256, 0, s>>>(p);
  return cudaGetLastError() == cudaSuccess ? WISP_OK : WISP_ERR_CUDA;
}

wisp_status wisp_kv_commit(const wisp_kv_args *kv, void *ws, size_t ws_bytes, void *stream) {
  wisp_status st = kv_check(kv, false, true);
  if (st != WISP_OK) return st;
  const KvLayout L = kv_layout(kv);
  if ((st = kv_ws_ok(ws, ws_bytes, L)) != WISP_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const KvParams p = kv_params(kv, ws, L);
  if (cudaMemsetAsync(p.status, 0, sizeof(DeviceStatus), s) != cudaSuccess) return WISP_ERR_CUDA;
  if (kv->B == 0) return WISP_OK;
  kv_commit_kernel<<<1, kThreads, 0, s>>>(p);
  return cudaGetLastError() == cudaSuccess ? WISP_OK : WISP_ERR_CUDA;
}

}  // extern "C"
