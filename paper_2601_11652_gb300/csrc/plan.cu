// plan.cu -- one-CTA planner: request offsets, length validation and the split-KV work list.
//
// The verification batch (Sec. 4.5) is ragged: request r contributes k_r + 1 query
// rows and c_r + k_r + 1 keys (L_total = L_cached + L_new, Sec. 4.4).  Lengths
// live on the device, so the planner runs there: it prefix-sums the row offsets,
// flags invalid requests, and cuts every (request, KV head) sequence into chunks
// of at most `chunk_len` keys so that the attention grid has about one item per
// SM (kItemsPerSM when there are fewer (request, head) pairs than SMs) whatever
// the length mix.
#include "plan.cuh"

namespace wisp {

namespace {

constexpr int kThreads = 1024;
constexpr int kOrderBuckets = 1024;  // tile-count buckets of the dispatch order
constexpr int kOrderTile = 64;       // tokens per KV tile of the attention kernels

__device__ __forceinline__ int64_t min64(int64_t a, int64_t b) { return a < b ? a : b; }
__device__ __forceinline__ int64_t max64(int64_t a, int64_t b) { return a > b ? a : b; }

// Inclusive block scan of one int64 per thread; returns the inclusive value, *total the block sum.
__device__ int64_t block_scan(int64_t v, int64_t *s_warp, int64_t *total) {
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  for (int d = 1; d < 32; d <<= 1) {
    int64_t o = __shfl_up_sync(0xffffffffu, v, d);
    if (lane >= d) v += o;
  }
  if (lane == 31) s_warp[w] = v;
  __syncthreads();
  if (w == 0) {
    int64_t t = s_warp[lane];
    for (int d = 1; d < 32; d <<= 1) {
      int64_t o = __shfl_up_sync(0xffffffffu, t, d);
      if (lane >= d) t += o;
    }
    s_warp[lane] = t;
  }
  __syncthreads();
  int64_t res = v + (w > 0 ? s_warp[w - 1] : 0);
  *total = s_warp[31];
  __syncthreads();
  return res;
}

// Inclusive block scans of N int64 per thread at once (one set of barriers for all N): v is replaced
// by its inclusive values, total[] receives the block sums.  s_w holds N x 32 values.
template <int N>
__device__ void block_scan_n(int64_t (&v)[N], int64_t (*s_w)[32], int64_t (&total)[N]) {
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  for (int d = 1; d < 32; d <<= 1) {
#pragma unroll
    for (int x = 0; x < N; ++x) {
      const int64_t o = __shfl_up_sync(0xffffffffu, v[x], d);
      if (lane >= d) v[x] += o;
    }
  }
  if (lane == 31) {
#pragma unroll
    for (int x = 0; x < N; ++x) s_w[x][w] = v[x];
  }
  __syncthreads();
  if (w == 0) {
#pragma unroll
    for (int x = 0; x < N; ++x) {
      int64_t t = s_w[x][lane];
      for (int d = 1; d < 32; d <<= 1) {
        const int64_t o = __shfl_up_sync(0xffffffffu, t, d);
        if (lane >= d) t += o;
      }
      s_w[x][lane] = t;
    }
  }
  __syncthreads();
#pragma unroll
  for (int x = 0; x < N; ++x) {
    v[x] += w > 0 ? s_w[x][w - 1] : 0;
    total[x] = s_w[x][31];
  }
  __syncthreads();
}

// The acceptance pass's dispatch order and state.  Rows are listed level-major: row index 0 of
// every valid request, then row index 1, ... (the requests of a level in decreasing draft length, so
// that request r holds the same position pos(r) in every level it reaches).  The decision of row i
// of a request is then usually known before its row i + 1 comes up, and the acceptance kernel skips
// rows past a rejection.  Also clears the per-row and per-request state of the launch and gives the
// requests this planner refused -1 outputs.
__device__ void plan_accept(const PlanParams &p, int64_t *s_warp) {
  constexpr int KB = kMaxDraft + 1;  // draft lengths 0..kMaxDraft
  __shared__ int32_t s_n[KB + 1];    // level sizes n_i = #{valid r : k_r >= i}, then cursors
  __shared__ int32_t s_ls[KB + 1];   // level starts
  const int tid = threadIdx.x;
  __syncthreads();  // pass 1's flags and offsets are visible to every thread
  for (int b = tid; b <= KB; b += kThreads) s_n[b] = 0;
  __syncthreads();
  int nv = 0;
  for (int r = tid; r < p.B; r += kThreads) {
    p.req_rej[r] = INT32_MAX;
    p.req_claim[r] = 0;
    p.req_dcnt[r] = 0;
    p.queue[r] = -1;
    if (p.req_flag[r] == REQ_OK) {
      atomicAdd(&s_n[p.draft_lens[r]], 1);  // histogram of k
      ++nv;
    } else {
      p.accepted_len[r] = -1;
      p.next_token[r] = -1;
    }
  }
  for (int64_t j = tid; j < p.total_q_rows; j += kThreads) {
    p.row_cnt[j] = 0;
    p.row_code[j] = 0;
  }
  // valid requests: a warp sum per warp, added into a shared counter
  __shared__ int32_t s_nvalid;
  if (tid == 0) s_nvalid = 0;
  __syncthreads();
  for (int o = 16; o > 0; o >>= 1) nv += __shfl_xor_sync(0xffffffffu, nv, o);
  if ((tid & 31) == 0 && nv) atomicAdd(&s_nvalid, nv);
  __syncthreads();
  const int64_t nvalid = s_nvalid;
  static_assert(KB + 1 <= 2 * kThreads, "two histogram buckets per thread");
  // n_i: suffix sums of the histogram (buckets in decreasing order, two per thread)
  {
    const int b0 = KB - 1 - 2 * tid, b1 = b0 - 1;
    const int64_t h0 = b0 >= 0 ? s_n[b0] : 0, h1 = b1 >= 0 ? s_n[b1] : 0;
    int64_t tot;
    const int64_t incl = block_scan(h0 + h1, s_warp, &tot);
    if (b0 >= 0) s_n[b0] = (int32_t)(incl - h1);
    if (b1 >= 0) s_n[b1] = (int32_t)incl;
  }
  if (tid == 0) s_n[KB] = 0;
  __syncthreads();
  // level starts: exclusive prefix sums of n_i (two per thread)
  int64_t rows_valid;
  {
    const int b0 = 2 * tid, b1 = b0 + 1;
    const int64_t c0 = b0 <= KB ? s_n[b0] : 0, c1 = b1 <= KB ? s_n[b1] : 0;
    const int64_t incl = block_scan(c0 + c1, s_warp, &rows_valid);
    if (b0 <= KB) s_ls[b0] = (int32_t)(incl - c0 - c1);
    if (b1 <= KB) s_ls[b1] = (int32_t)(incl - c1);
  }
  __syncthreads();
  // cursors: in every level, the requests with a larger k come first; bucket k starts at n_{k+1}
  int32_t nxt[2];
  for (int j = 0; j < 2; ++j) {
    const int b = j * kThreads + tid;
    nxt[j] = b < KB ? s_n[b + 1] : 0;
  }
  __syncthreads();
  for (int j = 0; j < 2; ++j) {
    const int b = j * kThreads + tid;
    if (b < KB) s_n[b] = nxt[j];
  }
  __syncthreads();
  for (int r = tid; r < p.B; r += kThreads) {
    if (p.req_flag[r] != REQ_OK) continue;
    const int k = p.draft_lens[r];
    const int pos = atomicAdd(&s_n[k], 1);
    for (int i = 0; i <= k; ++i) p.row_order[s_ls[i] + pos] = make_int2(r, i);
  }
  if (tid == 0) {
    p.acc_ctr->n_items = (int32_t)(rows_valid * p.sslices);
    p.acc_ctr->n_valid = (int32_t)nvalid;
    p.acc_ctr->q_reserve = 0;
    p.acc_ctr->q_head = 0;
    p.acc_ctr->n_claimed = 0;
    p.acc_ctr->stats_next = 0;
  }
  for (int j = tid; j < kTabCacheSlots; j += kThreads) {
    p.acc_ctr->tab_state[j] = 0;
    p.acc_ctr->tab_m[j] = 0;
  }
}

}  // namespace

__global__ void __launch_bounds__(kThreads) plan_kernel(const PlanParams p) {
  // a kernel launched after this one with programmatic stream serialization (the attention) may
  // start its own set-up now; it reads the plan only after waiting for this grid to complete
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  __shared__ int64_t s_warp[32];
  __shared__ int64_t s_warp4[4][32];
  const int tid = threadIdx.x;
  // the launch's status word starts clear (every kernel of the call reports into it)
  if (tid == 0) {
    p.status->code = 0;
    p.status->pad = 0;
    p.status->request_id = 0;
  }
  __syncthreads();
  const int g = p.Hq > 0 && p.Hkv > 0 ? p.Hq / p.Hkv : 1;
  const int64_t cap_tokens = (int64_t)p.max_blocks_per_seq * p.block_size;

  // pass 1: offsets (negative lengths count as 0) and validation
  int64_t carry_q = 0, carry_d = 0, carry_n = 0, carry_v = 0;
  // with at most kThreads requests, pass 3 reuses what this thread read and decided here
  int32_t my_k = 0, my_ctx = 0, my_q0 = 0;
  bool my_ok = false;
  for (int base = 0; base < p.B; base += kThreads) {
    const int r = base + tid;
    int64_t k = 0, n = 0;
    int bad = 0;
    if (r < p.B) {
      k = p.draft_lens[r];
      my_k = (int32_t)k;
      if (k < 0) { bad = WISP_DEV_BAD_LENGTH; k = 0; }
      if (!bad && k > kMaxDraft) bad = WISP_DEV_UNSUPPORTED;
      if (p.with_attention) {
        const int64_t c = p.context_lens[r];
        my_ctx = (int32_t)c;
        if (!bad && (c < 0 || c + k + 1 > cap_tokens)) bad = WISP_DEV_BAD_LENGTH;
        if (!bad && (int64_t)g * (k + 1) > kMaxRowsPerHead) bad = WISP_DEV_UNSUPPORTED;
        n = bad ? 0 : c + k + 1;
      }
    }
    int64_t sv[4] = {r < p.B ? k + 1 : 0, r < p.B ? k : 0, n, n > 0 ? 1 : 0}, st[4];
    block_scan_n<4>(sv, s_warp4, st);
    const int64_t iq = sv[0], id = sv[1], tq = st[0], td = st[1], tn = st[2], tv = st[3];
    if (r < p.B) {
      const int64_t q0 = carry_q + iq - (k + 1), d0 = carry_d + id - k;
      // a request whose rows fall outside the caller's buffers is never touched
      if (!bad && (q0 + k + 1 > p.total_q_rows || (p.total_draft >= 0 && d0 + k > p.total_draft)))
        bad = WISP_DEV_BAD_LENGTH;
      p.q_row_start[r] = (int32_t)min64(q0, INT32_MAX);
      p.draft_start[r] = (int32_t)min64(d0, INT32_MAX);
      p.req_flag[r] = bad ? REQ_BAD : REQ_OK;
      my_q0 = (int32_t)min64(q0, INT32_MAX);
      my_ok = !bad;
      if (bad) report(p.status, bad, p.request_ids, r);
    }
    carry_q += tq;
    carry_d += td;
    carry_n += tn;
    carry_v += tv;
  }
  if (tid == 0) {
    p.q_row_start[p.B] = (int32_t)min64(carry_q, INT32_MAX);
    p.draft_start[p.B] = (int32_t)min64(carry_d, INT32_MAX);
    if (carry_q != p.total_q_rows || (p.total_draft >= 0 && carry_d != p.total_draft)) {
      // the caller sized its buffers with other totals: flag it (requests that still fit run)
      atomicCAS(&p.status->code, 0, (int32_t)WISP_DEV_BAD_LENGTH);
    }
  }
  if (p.with_accept && !p.accept_apart) plan_accept(p, s_warp);
  if (!p.with_attention) return;
  __syncthreads();

  // pass 2: chunk length.  With at least as many (request, head) pairs as SMs, a longest-first
  // order balances whole sequences: only a sequence longer than 5/4 of the average work per SM
  // is cut (a split costs a merge of its chunks).  With fewer pairs than SMs, sequences are cut
  // into about kItemsPerSM items per SM.
  const int64_t work = carry_n * p.Hkv;
  const int64_t sms = max(1, p.target_items / kItemsPerSM);
  const bool many_pairs = carry_v * p.Hkv >= sms;
  const int64_t goal = many_pairs ? sms : (int64_t)p.target_items;
  int64_t chunk = (work + goal - 1) / goal;
  if (many_pairs) chunk += chunk / 4;
  chunk = max64(chunk, kMinChunk);
  chunk = (chunk + kChunkAlign - 1) / kChunkAlign * kChunkAlign;

  // pass 3: items and partial slots (request-major, then KV head, then row group, then chunk).
  // Per chunk of kThreads requests: one thread per request sizes its items (block scans), then the
  // chunk's items are written by consecutive threads (item i by thread i mod kThreads, its request
  // found by binary search over the chunk's first items), so that the stores coalesce.
  __shared__ int32_t s_first[kThreads + 1];  // the chunk's requests' first items, relative
  // per request of the chunk: query rows, chunks (0: no items), first partial, context, first
  // query row, keys
  __shared__ int32_t s_rows[kThreads], s_ch[kThreads], s_pf[kThreads], s_ctx[kThreads], s_q0[kThreads], s_nn[kThreads];
  int64_t item_carry = 0, poff_carry = 0;
  for (int base = 0; base < p.B; base += kThreads) {
    const int r = base + tid;
    int64_t n = 0, chunks = 0, rows = 0, nrg = 1, rows0 = 0;
    int32_t ctx_r = 0;
    const bool one = p.B <= kThreads;  // this thread's request of pass 1
    if (r < p.B && (one ? my_ok : p.req_flag[r] == REQ_OK)) {
      const int32_t k_r = one ? my_k : p.draft_lens[r];
      ctx_r = one ? my_ctx : p.context_lens[r];
      n = (int64_t)ctx_r + k_r + 1;
      chunks = (n + chunk - 1) / chunk;
      rows = (int64_t)g * (k_r + 1);
      nrg = rows > p.max_rows_item ? 2 : 1;
      rows0 = (rows + nrg - 1) / nrg;  // rows <= 2 * max_rows_item: both groups fit
    }
    const int64_t nitems = chunks * p.Hkv * nrg;
    // each split item's partials start on a 16-byte boundary (vector stores)
    const int64_t slot_a = (rows0 * (p.D + 2) + 3) / 4 * 4;
    const int64_t slot_b = nrg == 2 ? ((rows - rows0) * (p.D + 2) + 3) / 4 * 4 : 0;
    const int64_t pfl = chunks > 1 ? chunks * p.Hkv * (slot_a + slot_b) : 0;
    int64_t sv[2] = {nitems, pfl}, st[2];
    block_scan_n<2>(sv, s_warp4, st);
    const int64_t ii = sv[0], ip = sv[1], ti = st[0], tp = st[1];
    bool fits = false;
    if (r < p.B) {
      const int64_t first = item_carry + ii - nitems;
      const int64_t pfirst = poff_carry + ip - pfl;
      fits = first + nitems <= p.max_items && pfirst + pfl <= p.partial_cap;
      if (!fits && nitems > 0) {
        // cannot happen with the host's bounds; refuse the request rather than overflow
        p.req_flag[r] = REQ_BAD;
        report(p.status, WISP_DEV_UNSUPPORTED, p.request_ids, r);
      }
      p.req_item_begin[r] = (int32_t)first;
      p.req_chunks[r] = fits ? (int32_t)chunks : 0;
    }
    // the chunk's requests in shared memory: first item (relative), rows, chunks (0: no items)
    s_first[tid] = (int32_t)(ii - nitems);
    if (tid == kThreads - 1) s_first[kThreads] = (int32_t)ti;
    s_rows[tid] = (int32_t)rows;
    s_ch[tid] = fits ? (int32_t)chunks : 0;
    s_pf[tid] = (int32_t)min64(poff_carry + ip - pfl, INT32_MAX);
    s_ctx[tid] = ctx_r;
    s_q0[tid] = r < p.B ? (one ? my_q0 : p.q_row_start[r]) : 0;
    s_nn[tid] = (int32_t)n;
    // per (request, head, row group) finished-chunk counters of the chunk's requests: zeroed, coalesced
    const int64_t pd0 = (int64_t)base * p.Hkv * 2;
    const int64_t pd1 = (int64_t)min(p.B, base + kThreads) * p.Hkv * 2;
    for (int64_t x = pd0 + tid; x < pd1; x += kThreads) p.pair_done[x] = 0;
    __syncthreads();
    for (int64_t i = tid; i < ti; i += kThreads) {
      // the request of item i: the last one whose first item is <= i
      int lo = 0, hi = kThreads - 1;
      while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (s_first[mid] <= i) lo = mid;
        else hi = mid - 1;
      }
      const int rr = base + lo;
      const int ch = s_ch[lo];
      if (ch == 0 || rr >= p.B) continue;  // a refused request (its scan slot is empty)
      const int rws = s_rows[lo];
      const int ng = rws > p.max_rows_item ? 2 : 1;
      const int r0 = (rws + ng - 1) / ng;
      const int j = (int)(i - s_first[lo]);  // (head, row group, chunk) in that order
      const int hg = j / ch, c = j - hg * ch;
      const int h = ng == 2 ? hg >> 1 : hg, rg = ng == 2 ? hg & 1 : 0;
      const int sa = (r0 * (p.D + 2) + 3) / 4 * 4;
      const int sb = ng == 2 ? ((rws - r0) * (p.D + 2) + 3) / 4 * 4 : 0;
      WorkItem it;
      it.r = rr;
      it.h = h;
      it.t0 = (int32_t)(c * chunk);
      it.t1 = (int32_t)min64(s_nn[lo], (c + 1) * chunk);
      it.row0 = rg ? r0 : 0;
      it.rows = rg ? rws - r0 : r0;
      it.rg = rg;
      it.nrg = ng;
      it.poff = ch > 1 ? (int32_t)(s_pf[lo] + (int64_t)(h * ch + c) * (sa + sb) + (rg ? sa : 0)) : -1;
      it.q0 = s_q0[lo];
      it.ctx = s_ctx[lo];
      it.pad = 0;
      p.items[item_carry + i] = it;
    }
    item_carry += ti;
    poff_carry += tp;
    __syncthreads();  // s_first / s_rq are rewritten by the next chunk
  }
  // pass 4: dispatch order, longest items first (counting sort on the tile count), so that the
  // persistent kernel ends with its shortest items and its CTAs finish close together
  __shared__ int32_t s_hist[kOrderBuckets];
  const int64_t n_items = min64(item_carry, p.max_items);
  for (int b = tid; b < kOrderBuckets; b += kThreads) s_hist[b] = 0;
  __syncthreads();  // also makes pass 3's items visible to every thread of the block
  // an item's KV tiles: with one chunk of requests (B <= kThreads) from pass 3's shared arrays,
  // which still describe every request (no global read of the items just written), else from the
  // item itself
  const bool one_chunk = p.B <= kThreads;
  auto item_tiles = [&](int64_t i) -> int64_t {
    int64_t t0, t1;
    if (one_chunk) {
      int lo = 0, hi = kThreads - 1;
      while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (s_first[mid] <= i) lo = mid;
        else hi = mid - 1;
      }
      const int ch = max(1, s_ch[lo]);
      const int c = (int)(i - s_first[lo]) % ch;  // item = (head, row group) * ch + chunk
      t0 = (int64_t)c * chunk;
      t1 = min64(s_nn[lo], t0 + chunk);
    } else {
      const WorkItem &w = p.items[i];
      t0 = w.t0;
      t1 = w.t1;
    }
    return (t1 - t0 + kOrderTile - 1) / kOrderTile;
  };
  auto bucket_of = [&](int64_t tiles) -> int {
    return kOrderBuckets - 1 - (int)max64(0, min64(tiles, kOrderBuckets - 1));  // bucket 0: the longest
  };
  int64_t my_tiles = 0;  // KV tile passes of the attention (kOrderTile tokens), this thread's items
  for (int64_t i = tid; i < n_items; i += kThreads) {
    const int64_t t = item_tiles(i);
    atomicAdd(&s_hist[bucket_of(t)], 1);
    my_tiles += t;
  }
  __syncthreads();
  {
    static_assert(kOrderBuckets == kThreads, "one bucket per thread in the scan");
    int64_t tot;
    const int64_t incl = block_scan(s_hist[tid], s_warp, &tot);
    const int32_t excl = (int32_t)(incl - s_hist[tid]);
    __syncthreads();
    s_hist[tid] = excl;
    __syncthreads();
  }
  for (int64_t i = tid; i < n_items; i += kThreads) p.order[atomicAdd(&s_hist[bucket_of(item_tiles(i))], 1)] = (int32_t)i;
  int64_t tiles = 0;
  block_scan(my_tiles, s_warp, &tiles);

  if (tid == 0) {
    // SMs for the attention in a step whose acceptance pass runs beside it.  Both kernels are
    // persistent and each fills an SM's shared memory, so the acceptance CTAs start on the SMs the
    // attention leaves.  Measured on GB300 (bf16, D = 128): with few KV tiles per SM (under ~200
    // of 64 tokens) the attention is latency-bound and about half the SMs stream its keys as fast
    // as all of them (32 requests with 0.5-4K contexts: step 0.156 -> 0.129 ms with 80 attention
    // CTAs of 152); with more it is bound by each SM's streaming rate, and only a few SMs (an
    // eighth) pay off by starting the acceptance early (2-3% at 256-512 requests; a quarter or
    // more is slower).  When the acceptance has little vocabulary work per KV tile (under 50
    // elements: a few requests with long contexts) every SM stays with the attention.
    const int sms = p.target_items / kItemsPerSM;
    int na = sms;
    if (p.with_accept && p.split_sms && tiles > 0 && (int64_t)p.B * p.V >= 50 * tiles)
      na = tiles < (int64_t)200 * sms ? sms / 2 + 4 : sms - sms / 8;
    PlanHeader hd;
    hd.n_items = (int32_t)n_items;
    hd.chunk_len = (int32_t)chunk;
    hd.partial_floats = (int32_t)min64(poff_carry, p.partial_cap);
    hd.next_item = 0;
    hd.attn_ctas = na;
    for (int i = 0; i < 3; ++i) hd.pad[i] = 0;
    *p.header = hd;
  }
}

// The acceptance part of the plan on its own (a step: it runs on the acceptance pass's stream, so
// that the attention, which waits for the whole planner grid, does not wait for it).  Reads what
// plan_kernel's first pass wrote (flags and offsets).
__global__ void __launch_bounds__(kThreads) plan_accept_kernel(const PlanParams p) {
  __shared__ int64_t s_warp[32];
  plan_accept(p, s_warp);
}

}  // namespace wisp
