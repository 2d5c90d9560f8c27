// api.cu -- host side of the C ABI (include/wisp_verify.h): argument checks, workspace
// carving and kernel launches.  No allocation, no synchronisation on these paths.
#include <algorithm>
#include <cmath>
#include <cstring>
#include <mutex>

#include "accept.cuh"
#include "attn.cuh"

using namespace wisp;

namespace {

constexpr int kMaxDevices = 64;

// wisp_verify_step runs the acceptance pass on a side stream forked from and joined back into the
// caller's stream with two events.  Each caller stream gets its own side stream, so that steps
// issued on different streams do not wait for each other; past kMaxSides caller streams the slots
// are shared (correct, only serialised).
constexpr int kMaxSides = 32;
struct SideSlot {
  cudaStream_t caller = nullptr;
  cudaStream_t side = nullptr;
  cudaEvent_t ev_fork = nullptr, ev_join = nullptr;
};
struct DeviceInfo {
  int sms = 0;
  bool attrs_done = false;
  SideSlot sides[kMaxSides];
  int n_sides = 0;
  std::mutex step_mu;  // the slot table, and the fork / join of one call kept together
};
DeviceInfo g_dev[kMaxDevices];
std::mutex g_mu;

Exp2Table make_exp2_table() {
  Exp2Table t;
  for (int j = 0; j < 256; ++j) {
    const double v = std::exp2(j / 256.0);
    t.hi[j] = (float)v;
    t.lo[j] = (float)(v - (double)t.hi[j]);
  }
  return t;
}
const Exp2Table g_exp2 = make_exp2_table();

size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

// The side stream and events of caller stream `s` (created on its first step; under d.step_mu).
SideSlot *side_slot(DeviceInfo &d, cudaStream_t s) {
  for (int i = 0; i < d.n_sides; ++i)
    if (d.sides[i].caller == s) return &d.sides[i];
  if (d.n_sides == kMaxSides) return &d.sides[(uintptr_t)s % kMaxSides];
  SideSlot &n = d.sides[d.n_sides];
  if (cudaStreamCreateWithFlags(&n.side, cudaStreamNonBlocking) != cudaSuccess ||
      cudaEventCreateWithFlags(&n.ev_fork, cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&n.ev_join, cudaEventDisableTiming) != cudaSuccess)
    return nullptr;
  n.caller = s;
  ++d.n_sides;
  return &n;
}

wisp_status device_setup(int *dev_out, int *sms_out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return WISP_ERR_CUDA;
  std::lock_guard<std::mutex> lk(g_mu);
  DeviceInfo &d = g_dev[dev];
  if (!d.attrs_done) {
    int sms = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return WISP_ERR_CUDA;
    cudaError_t e = attn_simt_setup();
    if (e == cudaSuccess) e = attn_tc_setup();
    if (e == cudaSuccess) e = accept_setup();
    if (e != cudaSuccess) return WISP_ERR_CUDA;
    d.sms = sms;
    d.attrs_done = true;
  }
  *dev_out = dev;
  *sms_out = d.sms;
  return WISP_OK;
}

bool aligned16(const void *p) { return ((uintptr_t)p & 15) == 0; }

wisp_status check_attn(const wisp_attn_args *a) {
  if (!a) return WISP_ERR_INVALID_ARG;
  if (a->B < 0 || a->Hq <= 0 || a->Hkv <= 0 || a->Hq % a->Hkv != 0) return WISP_ERR_INVALID_ARG;
  if (a->D != 64 && a->D != 128) return WISP_ERR_UNSUPPORTED;
  if (a->block_size != 16) return WISP_ERR_UNSUPPORTED;
  if (a->qkv_dtype != WISP_F32 && a->qkv_dtype != WISP_BF16) return WISP_ERR_INVALID_ARG;
  if (a->B == 0) return WISP_OK;
  if (a->max_blocks_per_seq <= 0 || a->num_blocks <= 0 || a->total_q_rows < a->B) return WISP_ERR_INVALID_ARG;
  if (!a->draft_lens || !a->context_lens || !a->block_tables || !a->q || !a->k_cache || !a->v_cache || !a->out)
    return WISP_ERR_INVALID_ARG;
  if (!aligned16(a->q) || !aligned16(a->k_cache) || !aligned16(a->v_cache) || !aligned16(a->out))
    return WISP_ERR_INVALID_ARG;
  if ((int64_t)a->max_blocks_per_seq * a->block_size > INT32_MAX / 2) return WISP_ERR_UNSUPPORTED;
  return WISP_OK;
}

// Vocabulary slices per logit row for the row-statistics kernel (one warp each): enough warps to
// keep every SM streaming (48 per SM), slices of at least 256 vectors (4 KB), at most kMaxSlices.
void accept_slices(const wisp_accept_args *c, int sms, int *slices, int *vps) {
  const int E = c->logits_dtype == WISP_BF16 ? 8 : 4;
  const int64_t nvec = ((int64_t)c->V + E - 1) / E;
  const int64_t rows = c->total_q_rows > 0 ? c->total_q_rows : 1;
  int64_t S = ((int64_t)48 * sms + rows - 1) / rows;
  const int64_t by_size = (nvec + 255) / 256;
  if (S > by_size) S = by_size;
  if (S > kMaxSlices) S = kMaxSlices;
  if (S < 1) S = 1;
  const int64_t v = ((nvec + S - 1) / S + 31) / 32 * 32;
  *vps = (int)v;
  *slices = (int)((nvec + v - 1) / v);
}

// Work shape of the acceptance kernel: statistics slices per row (about two items per resident
// CTA over the batch's rows: more, smaller items cost more in per-item set-up and bookkeeping than
// they gain in balance; a slice is a whole number of 3-vector chunks per thread), draw tiles (64 vectors: one warp's share of a draw chunk; no tile records when they
// would exceed tile_budget bytes) and draw slices per row (one item per resident CTA over the batch
// when it is small, up to two per CTA as it grows; whole chunks of 256 vectors).
constexpr size_t kTileBudget = (size_t)256 << 20;
constexpr size_t kNoAllocTileBudget = (size_t)4 << 20;
struct AcceptShape {
  int sslices, svps, dslices, vpd, tile_vecs, ntiles;
};
AcceptShape accept_shape(const wisp_accept_args *c, int sms, size_t tile_budget) {
  const int E = c->logits_dtype == WISP_BF16 ? 8 : 4;
  const int64_t nvec = ((int64_t)c->V + E - 1) / E;
  const int64_t ctas = (int64_t)sms * kAcceptCtasPerSM;
  const int64_t B = c->B > 0 ? c->B : 1;
  auto cut = [&](int64_t want, int64_t units, int64_t min_vecs, int *n, int *per) {
    int64_t S = (want + units - 1) / units;
    const int64_t by_size = (nvec + min_vecs - 1) / min_vecs;
    if (S > by_size) S = by_size;
    if (S > 32) S = 32;
    if (S < 1) S = 1;
    // whole rounds of the CTA's loads per slice
    const int64_t v = ((nvec + S - 1) / S + min_vecs - 1) / min_vecs * min_vecs;
    *per = (int)v;
    *n = (int)((nvec + v - 1) / v);
  };
  AcceptShape sh;
  cut(2 * ctas, c->total_q_rows > 0 ? c->total_q_rows : 1, (int64_t)kAcceptThreads * kStatsChunkVecs, &sh.sslices,
      &sh.svps);
  // a tile is one warp's 64 vectors of a draw chunk; without room for the records, none
  const int64_t nt = (nvec + 63) / 64;
  const bool tiles = B * nt * (int64_t)sizeof(TileRec) <= (int64_t)tile_budget;
  sh.tile_vecs = tiles ? 64 : 0;
  sh.ntiles = tiles ? (int)nt : 0;
  // draw slices: one wave of items over the CTAs when the batch is small, up to two waves (and
  // about three slices per row) as it grows, and at least two per row (a slice keeps at most
  // kAmbPerSlice undecided elements; past that the bookkeeper weighs the slice exactly alone)
  cut(std::max<int64_t>(2 * B, std::max<int64_t>(ctas, std::min<int64_t>(2 * ctas, 3 * B))), B, kAcceptThreads,
      &sh.dslices, &sh.vpd);
  return sh;
}

// need_probs: the sampling rule reads the draft distributions and the uniforms; the greedy one does not
wisp_status check_accept(const wisp_accept_args *c, bool need_probs = true) {
  if (!c) return WISP_ERR_INVALID_ARG;
  if (c->B < 0 || c->V <= 0 || c->total_draft < 0) return WISP_ERR_INVALID_ARG;
  if (c->logits_dtype != WISP_F32 && c->logits_dtype != WISP_BF16) return WISP_ERR_INVALID_ARG;
  if (c->B == 0) return WISP_OK;
  if (c->total_q_rows < c->B) return WISP_ERR_INVALID_ARG;
  if (!c->draft_lens || !c->target_logits || !c->accepted_len || !c->next_token) return WISP_ERR_INVALID_ARG;
  if (need_probs && !c->sample_uniforms) return WISP_ERR_INVALID_ARG;
  if (c->total_draft > 0 && !c->draft_tokens) return WISP_ERR_INVALID_ARG;
  if (need_probs && c->total_draft > 0 && (!c->draft_probs || !c->accept_uniforms)) return WISP_ERR_INVALID_ARG;
  if (c->V > (1 << 24)) return WISP_ERR_UNSUPPORTED;  // vocabulary limit of the acceptance kernel
  if ((int64_t)c->B * 8 > INT32_MAX) return WISP_ERR_UNSUPPORTED;
  if ((int64_t)c->total_q_rows * kMaxSlices > INT32_MAX) return WISP_ERR_UNSUPPORTED;
  return WISP_OK;
}

Layout make_layout(const wisp_attn_args *a, const wisp_accept_args *c, int sms, size_t tile_budget = kTileBudget) {
  Layout L;
  const int B = a ? a->B : (c ? c->B : 0);
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t at = off;
    off = align256(off + bytes);
    return at;
  };
  L.status = take(sizeof(DeviceStatus));
  L.q_row_start = take(sizeof(int32_t) * (size_t)(B + 1));
  L.draft_start = take(sizeof(int32_t) * (size_t)(B + 1));
  L.req_flag = take(sizeof(int32_t) * (size_t)B);
  L.plan_header = take(sizeof(PlanHeader));
  if (a) {
    L.target_items = sms * kItemsPerSM;
    // the tensor-core kernel takes at most kTcRowsPerItem query rows per item: a (request, head)
    // with more is cut into two row groups, which at most doubles the item count
    const int64_t rg = a->qkv_dtype == WISP_BF16 ? 2 : 1;
    L.max_items = rg * ((int64_t)L.target_items + (int64_t)B * a->Hkv);
    L.partial_cap = (int64_t)2 * L.target_items * kMaxRowsPerHead * (a->D + 2);
    L.req_item_begin = take(sizeof(int32_t) * (size_t)B);
    L.req_chunks = take(sizeof(int32_t) * (size_t)B);
    L.pair_done = take(sizeof(int32_t) * (size_t)B * a->Hkv * 2);
    L.items = take(sizeof(WorkItem) * (size_t)L.max_items);
    L.order = take(sizeof(int32_t) * (size_t)L.max_items);
    L.partials = take(sizeof(float) * (size_t)L.partial_cap);
  }
  if (c && c->B > 0) {
    const AcceptShape sh = accept_shape(c, sms, tile_budget);
    const size_t T = (size_t)c->total_q_rows;
    L.acc_ctr = take(sizeof(AccCounters));
    L.row_order = take(sizeof(int2) * T);
    L.row_cnt = take(sizeof(int32_t) * T);
    L.row_code = take(sizeof(int32_t) * T);
    L.row_rec = take(sizeof(RowRec) * T);
    L.sparts = take(sizeof(SlicePart) * T * sh.sslices);
    L.req_state = take(sizeof(int32_t) * 5 * (size_t)c->B);
    L.dparts = take(sizeof(DrawPart) * (size_t)c->B * sh.dslices);
    L.tiles = take(sizeof(TileRec) * ((size_t)c->B * sh.ntiles + 1));
    L.tcache = c->logits_dtype == WISP_BF16 ? take((size_t)kTabCacheSlots * kExpTabBytes) : 0;
    // the greedy variant's argmax partials (8 bytes per row and warp slice) share the statistics'
    // space when they fit, else get their own
    int S = 1, vps = 0;
    accept_slices(c, sms, &S, &vps);
    const size_t gbytes = 8 * T * S;
    L.row_parts = gbytes <= sizeof(SlicePart) * T * sh.sslices ? L.sparts : take(gbytes);
  }
  L.total = off;
  return L;
}

template <typename T>
T *at(void *ws, size_t off) {
  return reinterpret_cast<T *>(static_cast<char *>(ws) + off);
}

wisp_status check_ws(void *ws, size_t bytes, const Layout &L) {
  if (!ws || ((uintptr_t)ws & 255) != 0 || bytes < L.total) return WISP_ERR_WORKSPACE;
  return WISP_OK;
}

PlanParams plan_params(const wisp_attn_args *a, const wisp_accept_args *c, void *ws, const Layout &L, int sms,
                       bool with_accept) {
  PlanParams pp;
  std::memset(&pp, 0, sizeof pp);
  pp.B = a ? a->B : c->B;
  pp.draft_lens = a ? a->draft_lens : c->draft_lens;
  pp.request_ids = a ? a->request_ids : c->request_ids;
  pp.total_q_rows = a ? a->total_q_rows : c->total_q_rows;
  pp.total_draft = c ? c->total_draft : -1;
  pp.status = at<DeviceStatus>(ws, L.status);
  pp.q_row_start = at<int32_t>(ws, L.q_row_start);
  pp.draft_start = at<int32_t>(ws, L.draft_start);
  pp.req_flag = at<int32_t>(ws, L.req_flag);
  pp.header = at<PlanHeader>(ws, L.plan_header);
  if (a) {
    pp.Hq = a->Hq;
    pp.Hkv = a->Hkv;
    pp.D = a->D;
    pp.max_blocks_per_seq = a->max_blocks_per_seq;
    pp.block_size = a->block_size;
    pp.context_lens = a->context_lens;
    pp.with_attention = 1;
    pp.target_items = L.target_items;
    pp.max_rows_item = a->qkv_dtype == WISP_BF16 ? kTcRowsPerItem : kMaxRowsPerHead;
    pp.max_items = L.max_items;
    pp.partial_cap = L.partial_cap;
    pp.req_item_begin = at<int32_t>(ws, L.req_item_begin);
    pp.req_chunks = at<int32_t>(ws, L.req_chunks);
    pp.pair_done = at<int32_t>(ws, L.pair_done);
    pp.items = at<WorkItem>(ws, L.items);
    pp.order = at<int32_t>(ws, L.order);
  } else {
    pp.Hq = pp.Hkv = 1;
  }
  if (c && c->B > 0 && with_accept) {
    pp.with_accept = 1;
    pp.split_sms = a != nullptr;
    pp.V = c->V;
    pp.sslices = accept_shape(c, sms, kTileBudget).sslices;  // (the statistics slices do not depend on the budget)
    pp.row_order = at<int2>(ws, L.row_order);
    pp.row_cnt = at<int32_t>(ws, L.row_cnt);
    pp.row_code = at<int32_t>(ws, L.row_code);
    int32_t *rs = at<int32_t>(ws, L.req_state);
    pp.req_rej = rs;
    pp.req_claim = rs + c->B;
    pp.req_dcnt = rs + 3 * (size_t)c->B;
    pp.queue = rs + 4 * (size_t)c->B;
    pp.acc_ctr = at<AccCounters>(ws, L.acc_ctr);
    pp.accepted_len = c->accepted_len;
    pp.next_token = c->next_token;
  }
  return pp;
}

wisp_status launch_attention(const wisp_attn_args *a, void *ws, const Layout &L, cudaStream_t s, bool pdl) {
  AttnParams ap;
  ap.B = a->B;
  ap.Hq = a->Hq;
  ap.Hkv = a->Hkv;
  ap.D = a->D;
  ap.max_blocks_per_seq = a->max_blocks_per_seq;
  ap.num_blocks = a->num_blocks;
  ap.request_ids = a->request_ids;
  ap.block_tables = a->block_tables;
  ap.q = a->q;
  ap.k_cache = a->k_cache;
  ap.v_cache = a->v_cache;
  ap.out = a->out;
  ap.status = at<DeviceStatus>(ws, L.status);
  ap.req_flag = at<int32_t>(ws, L.req_flag);
  ap.req_item_begin = at<int32_t>(ws, L.req_item_begin);
  ap.req_chunks = at<int32_t>(ws, L.req_chunks);
  ap.header = at<PlanHeader>(ws, L.plan_header);
  ap.header_mut = at<PlanHeader>(ws, L.plan_header);
  ap.items = at<WorkItem>(ws, L.items);
  ap.order = at<int32_t>(ws, L.order);
  ap.partials = at<float>(ws, L.partials);
  ap.pair_done = at<int32_t>(ws, L.pair_done);
  const bool bf = a->qkv_dtype == WISP_BF16;
  if (bf) {
    // persistent tensor-core kernel: one CTA per SM
    const int grid = (int)(L.max_items < L.target_items / kItemsPerSM ? L.max_items : L.target_items / kItemsPerSM);
    // the work counter lives in the plan header written by the planner on this stream
    // split items are merged inside the kernel by the last chunk to finish
    return attn_tc_launch(ap, grid, s, pdl) == cudaSuccess ? WISP_OK : WISP_ERR_CUDA;
  }
  if (attn_simt_launch(ap, bf, (int)L.max_items, s) != cudaSuccess) return WISP_ERR_CUDA;
  return attn_combine_launch(ap, bf, s) == cudaSuccess ? WISP_OK : WISP_ERR_CUDA;
}

AcceptParams accept_params(const wisp_accept_args *c, void *ws, const Layout &L, int sms,
                           size_t tile_budget = kTileBudget) {
  AcceptParams ap;
  std::memset(&ap, 0, sizeof ap);
  ap.B = c->B;
  ap.V = c->V;
  const bool bf = c->logits_dtype == WISP_BF16;
  const size_t esz = bf ? 2 : 4;
  ap.vec_z = ((uintptr_t)c->target_logits % 16 == 0) && ((size_t)c->V * esz % 16 == 0);
  ap.vec_q = c->draft_probs && ((uintptr_t)c->draft_probs % 16 == 0) && ((size_t)c->V * 4 % 16 == 0);
  const AcceptShape sh = accept_shape(c, sms, tile_budget);
  ap.sslices = sh.sslices;
  ap.svps = sh.svps;
  ap.dslices = sh.dslices;
  ap.vpd = sh.vpd;
  ap.tile_vecs = sh.tile_vecs;
  ap.ntiles = sh.ntiles;
  ap.tiles = at<TileRec>(ws, L.tiles);
  ap.total_rows = c->total_q_rows;
  accept_slices(c, sms, &ap.slices, &ap.vps);
  ap.parts = at<void>(ws, L.row_parts);
  ap.row_order = at<int2>(ws, L.row_order);
  ap.row_cnt = at<int32_t>(ws, L.row_cnt);
  ap.row_code = at<int32_t>(ws, L.row_code);
  ap.row_rec = at<RowRec>(ws, L.row_rec);
  ap.sparts = at<SlicePart>(ws, L.sparts);
  int32_t *rs = at<int32_t>(ws, L.req_state);
  ap.req_rej = rs;
  ap.req_claim = rs + c->B;
  ap.req_L = rs + 2 * (size_t)c->B;
  ap.req_dcnt = rs + 3 * (size_t)c->B;
  ap.queue = rs + 4 * (size_t)c->B;
  ap.dparts = at<DrawPart>(ws, L.dparts);
  ap.ctr = at<AccCounters>(ws, L.acc_ctr);
  ap.tcache = bf ? at<uint32_t>(ws, L.tcache) : nullptr;
  ap.request_ids = c->request_ids;
  ap.draft_lens = c->draft_lens;
  ap.logits = c->target_logits;
  ap.draft_tokens = c->draft_tokens;
  ap.draft_probs = c->draft_probs;
  ap.accept_u = c->accept_uniforms;
  ap.sample_u = c->sample_uniforms;
  ap.accepted_len = c->accepted_len;
  ap.next_token = c->next_token;
  ap.q_row_start = at<int32_t>(ws, L.q_row_start);
  ap.draft_start = at<int32_t>(ws, L.draft_start);
  ap.req_flag = at<int32_t>(ws, L.req_flag);
  ap.status = at<DeviceStatus>(ws, L.status);
  ap.tab = g_exp2;
  return ap;
}

// with_accept: the planner also lays out the sampling rule's dispatch order and clears its state
// accept_apart: the acceptance part is left to launch_plan_accept (on another stream).
wisp_status launch_plan(const wisp_attn_args *a, const wisp_accept_args *c, void *ws, const Layout &L, int sms,
                        bool with_accept, cudaStream_t s, bool accept_apart = false) {
  PlanParams pp = plan_params(a, c, ws, L, sms, with_accept);
  pp.accept_apart = accept_apart ? 1 : 0;
  plan_kernel<<<1, 1024, 0, s>>>(pp);
  return cudaGetLastError() == cudaSuccess ? WISP_OK : WISP_ERR_CUDA;
}
wisp_status launch_plan_accept(const wisp_attn_args *a, const wisp_accept_args *c, void *ws, const Layout &L,
                               int sms, cudaStream_t s) {
  const PlanParams pp = plan_params(a, c, ws, L, sms, true);
  plan_accept_kernel<<<1, 1024, 0, s>>>(pp);
  return cudaGetLastError() == cudaSuccess ? WISP_OK : WISP_ERR_CUDA;
}

// The planner, then the acceptance kernel as its programmatic dependent (its CTAs are placed while
// the planner runs and wait for it before reading anything).
wisp_status launch_accept(const wisp_accept_args *c, void *ws, const Layout &L, int sms, cudaStream_t s,
                          size_t tile_budget = kTileBudget) {
  wisp_status st = launch_plan(nullptr, c, ws, L, sms, true, s);
  if (st != WISP_OK || c->B == 0) return st;
  const AcceptParams ap = accept_params(c, ws, L, sms, tile_budget);
  return accept_launch(ap, c->logits_dtype == WISP_BF16, sms, s, true) == cudaSuccess ? WISP_OK : WISP_ERR_CUDA;
}

}  // namespace

// Workspace of wisp_verify_accept_noalloc: status word, per-request offsets, flags and state,
// planner header, the dispatch order and statistics of every logit row, the draw's slice totals.
// 16 MiB holds them for batches of up to kNoAllocMaxBatch requests and kNoAllocMaxRows logit rows.
constexpr size_t kNoAllocScratchBytes = 16 << 20;
constexpr int kNoAllocMaxBatch = 8192;
constexpr int kNoAllocMaxRows = 131072;
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

namespace {

void *g_noalloc_ptr[kMaxDevices];  // device address of g_noalloc_scratch, per device

// Address of the scratch array on the current device `dev`, looked up once (under g_mu).
wisp_status noalloc_scratch(int dev, void **out) {
  std::lock_guard<std::mutex> lk(g_mu);
  if (!g_noalloc_ptr[dev]) {
    void *ptr = nullptr;
    if (cudaGetSymbolAddress(&ptr, g_noalloc_scratch) != cudaSuccess || !ptr) return WISP_ERR_CUDA;
    g_noalloc_ptr[dev] = ptr;
  }
  *out = g_noalloc_ptr[dev];
  return WISP_OK;
}

}  // namespace

extern "C" {

size_t wisp_verify_workspace_size(const wisp_attn_args *attn, const wisp_accept_args *acc) {
  if (!attn && !acc) return 0;
  if (attn && check_attn(attn) != WISP_OK) return 0;
  if (acc && check_accept(acc, false) != WISP_OK) return 0;  // the size does not depend on the distributions
  if (attn && acc && attn->B != acc->B) return 0;
  int dev = 0, sms = 0;
  if (device_setup(&dev, &sms) != WISP_OK) return 0;
  return make_layout(attn, acc, sms).total;
}

wisp_status wisp_verify_attention(const wisp_attn_args *attn, void *ws, size_t ws_bytes, void *stream) {
  wisp_status st = check_attn(attn);
  if (st != WISP_OK) return st;
  int dev = 0, sms = 0;
  if ((st = device_setup(&dev, &sms)) != WISP_OK) return st;
  const Layout L = make_layout(attn, nullptr, sms);
  if ((st = check_ws(ws, ws_bytes, L)) != WISP_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if ((st = launch_plan(attn, nullptr, ws, L, sms, false, s)) != WISP_OK) return st;
  if (attn->B == 0) return WISP_OK;
  // alone on the stream after the planner: the attention CTAs set up while the planner runs
  return launch_attention(attn, ws, L, s, true);
}

wisp_status wisp_verify_accept(const wisp_accept_args *acc, void *ws, size_t ws_bytes, void *stream) {
  wisp_status st = check_accept(acc);
  if (st != WISP_OK) return st;
  int dev = 0, sms = 0;
  if ((st = device_setup(&dev, &sms)) != WISP_OK) return st;
  const Layout L = make_layout(nullptr, acc, sms);
  if ((st = check_ws(ws, ws_bytes, L)) != WISP_OK) return st;
  return launch_accept(acc, ws, L, sms, static_cast<cudaStream_t>(stream));
}

wisp_status wisp_verify_accept_greedy(const wisp_accept_args *acc, void *ws, size_t ws_bytes, void *stream) {
  wisp_status st = check_accept(acc, false);
  if (st != WISP_OK) return st;
  int dev = 0, sms = 0;
  if ((st = device_setup(&dev, &sms)) != WISP_OK) return st;
  const Layout L = make_layout(nullptr, acc, sms);
  if ((st = check_ws(ws, ws_bytes, L)) != WISP_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if ((st = launch_plan(nullptr, acc, ws, L, sms, false, s)) != WISP_OK) return st;
  if (acc->B == 0) return WISP_OK;
  const AcceptParams ap = accept_params(acc, ws, L, sms);
  return accept_greedy_launch(ap, acc->logits_dtype == WISP_BF16, s) == cudaSuccess ? WISP_OK : WISP_ERR_CUDA;
}

wisp_status wisp_verify_step(const wisp_attn_args *attn, const wisp_accept_args *acc, void *ws, size_t ws_bytes,
                             void *stream) {
  wisp_status st = check_attn(attn);
  if (st != WISP_OK) return st;
  if ((st = check_accept(acc)) != WISP_OK) return st;
  if (attn->B != acc->B || attn->total_q_rows != acc->total_q_rows) return WISP_ERR_INVALID_ARG;
  int dev = 0, sms = 0;
  if ((st = device_setup(&dev, &sms)) != WISP_OK) return st;
  const Layout L = make_layout(attn, acc, sms);
  if ((st = check_ws(ws, ws_bytes, L)) != WISP_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (attn->B == 0) return launch_plan(attn, acc, ws, L, sms, true, s);
  // One planner for both parts.  The attention follows it on `s` as its programmatic dependent
  // (persistent, one CTA per SM); the acceptance pass reads only the logits and the planner's
  // state, so it runs on the library's side stream, forked after the planner and joined back: its
  // CTAs take the SMs the attention's CTAs leave as they finish.
  DeviceInfo &d = g_dev[dev];
  std::lock_guard<std::mutex> lk(d.step_mu);
  SideSlot *sl = side_slot(d, s);
  if (!sl) return WISP_ERR_CUDA;
  if ((st = launch_plan(attn, acc, ws, L, sms, true, s, true)) != WISP_OK) return st;
  const AcceptParams ap = accept_params(acc, ws, L, sms);
  const bool bf = acc->logits_dtype == WISP_BF16;
  // the attention is enqueued first, so that its CTAs take the SMs first; the acceptance part of
  // the plan and the acceptance CTAs follow on the side stream, on the SMs the attention leaves
  bool ok = cudaEventRecord(sl->ev_fork, s) == cudaSuccess;
  ok = ok && launch_attention(attn, ws, L, s, true) == WISP_OK;
  const bool forked = ok && cudaStreamWaitEvent(sl->side, sl->ev_fork, 0) == cudaSuccess;
  ok = forked && launch_plan_accept(attn, acc, ws, L, sms, sl->side) == WISP_OK;
  ok = ok && accept_launch(ap, bf, sms, sl->side, false) == cudaSuccess;
  // join what was forked even after a failed launch, so that `s` never runs ahead of `side`
  const bool joined = !forked || (cudaEventRecord(sl->ev_join, sl->side) == cudaSuccess &&
                                  cudaStreamWaitEvent(s, sl->ev_join, 0) == cudaSuccess);
  return ok && joined ? WISP_OK : WISP_ERR_CUDA;
}

wisp_status wisp_verify_get_device_status(const void *ws, int32_t *code, int64_t *request_id) {
  if (!ws || !code || !request_id) return WISP_ERR_INVALID_ARG;
  DeviceStatus h;
  if (cudaMemcpy(&h, ws, sizeof h, cudaMemcpyDeviceToHost) != cudaSuccess) return WISP_ERR_CUDA;
  *code = h.code;
  *request_id = h.code ? h.request_id : -1;
  return WISP_OK;
}

// ---- acceptance pass without a caller workspace (no counterpart in the paper) -----------------
// Some callers cannot allocate device memory when they verify: a serving loop whose memory is
// owned by another allocator (a caching pool it must not bypass), or a latency path where
// cudaMalloc is off limits because it can synchronise the device.  This entry point runs the same
// planner and acceptance kernels as wisp_verify_accept, with their workspace carved from a fixed
// array in this library's device image instead of caller memory.  Nothing here allocates: the
// array exists once the module is loaded, and the first call on a device only looks up its
// address (cudaGetSymbolAddress) and sets kernel attributes.
wisp_status wisp_verify_accept_noalloc(const wisp_accept_args *acc, void *stream) {
  wisp_status st = check_accept(acc);
  if (st != WISP_OK) return st;
  if (acc->B > kNoAllocMaxBatch || acc->total_q_rows > kNoAllocMaxRows) return WISP_ERR_UNSUPPORTED;
  int dev = 0, sms = 0;
  if ((st = device_setup(&dev, &sms)) != WISP_OK) return st;
  const Layout L = make_layout(nullptr, acc, sms, kNoAllocTileBudget);
  if (L.total > kNoAllocScratchBytes) return WISP_ERR_UNSUPPORTED;
  void *ws = nullptr;
  if ((st = noalloc_scratch(dev, &ws)) != WISP_OK) return st;
  // the planner clears the status word and the launch's counters and per-row / per-request state
  // (everything that must start at zero) on `stream` first
  return launch_accept(acc, ws, L, sms, static_cast<cudaStream_t>(stream), kNoAllocTileBudget);
}

const char *wisp_verify_status_string(wisp_status s) {
  switch (s) {
    case WISP_OK: return "ok";
    case WISP_ERR_INVALID_ARG: return "invalid argument";
    case WISP_ERR_UNSUPPORTED: return "unsupported configuration";
    case WISP_ERR_CUDA: return "CUDA runtime error";
    case WISP_ERR_WORKSPACE: return "workspace missing, misaligned or too small";
  }
  return "unknown status";
}

const char *wisp_verify_device_code_string(int32_t code) {
  switch (code) {
    case WISP_DEV_OK: return "ok";
    case WISP_DEV_BAD_LENGTH: return "bad length";
    case WISP_DEV_BAD_BLOCK: return "block id out of range";
    case WISP_DEV_BAD_TOKEN: return "draft token out of range";
    case WISP_DEV_BAD_PROB: return "bad probability or logit row";
    case WISP_DEV_UNSUPPORTED: return "unsupported request shape";
    case WISP_DEV_TIMEOUT: return "device wait timed out";
    case WISP_DEV_NO_BLOCKS: return "no free KV pages";
  }
  return "unknown device code";
}

}  // extern "C"
