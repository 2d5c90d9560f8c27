/*
 * wisp_verify.h -- C ABI of the batched speculative-verification step.
 *
 * What the step is (arxiv 2601.11652, WISP):
 *   A verification batch B_k (Sec. 4.2-4.3) holds, per request, a draft block
 *   y_1..y_k proposed on an edge device with its draft distributions q, and the
 *   request's cached-prefix KV (PageAttention blocks + prefix cache, Sec. 4.5).
 *   The verification engine (Sec. 4.5, "batched one-step verification")
 *   forwards the new block over the cached prefix, applies the in-order
 *   acceptance rule (Eq. 1, a_i = min(1, p/q), A_i = 1[u_i <= a_i]), stops at
 *   the first rejection (Eq. 2, R and L = R - 1) and returns L and one extra
 *   token drawn at the stopping position (Eq. 3), which keeps the output
 *   distribution identical to target-only decoding (Sec. 4 opening).
 *
 *   This library implements the two parts of that step that move data:
 *     wisp_verify_attention  the attention of the forward over L_total =
 *                            L_cached + L_new keys (Sec. 4.4) for each
 *                            request's k+1 new query tokens, paged KV, GQA;
 *     wisp_verify_accept     the acceptance pass over the vocabulary (Eq. 1-3);
 *     wisp_verify_step       both, in one call.
 *   The linear layers that turn attention outputs into logits are outside this
 *   library: the target logits are an input of wisp_verify_accept.
 *
 * Conventions for every entry point:
 *   - Every pointer inside the argument structs is a DEVICE pointer owned by
 *     the caller, except where a field says otherwise.  The library never
 *     allocates, frees or synchronises in these calls; it only enqueues
 *     kernels on `stream` (a cudaStream_t; NULL = the legacy default stream).
 *   - All calls are asynchronous.  Argument errors that the host can see are
 *     returned before anything is enqueued (WISP_ERR_INVALID_ARG,
 *     WISP_ERR_UNSUPPORTED, WISP_ERR_WORKSPACE).
 *   - Errors in device data (a length, block id, token id or probability that
 *     is out of range) cannot be seen by the host.  The kernels record the
 *     first such error and its request id in a status word inside the
 *     workspace, skip that request (its outputs are left unspecified) and
 *     finish normally; they never trap.  Read the word with
 *     wisp_verify_get_device_status after synchronising the stream.  Each
 *     entry point clears the word when it starts.
 *   - The workspace is caller-owned device memory of at least
 *     wisp_verify_workspace_size() bytes, 256-byte aligned.  Calls that share a
 *     workspace must not overlap in time.
 *
 * Data layout (row-major, ids 0-based):
 *   request r owns k_r + 1 consecutive query/logit rows starting at
 *   Q0_r = sum_{r' < r} (k_r' + 1), and k_r consecutive draft rows starting at
 *   D0_r = sum_{r' < r} k_r'.  Logit row Q0_r + i is the target distribution
 *   for draft token i + 1 (i < k_r); row Q0_r + k_r is the bonus row.  Query
 *   row Q0_r + j (j = 0..k_r) sits at absolute position c_r + j and attends
 *   keys 0..c_r + j of its own sequence, whose token t lives in physical block
 *   block_tables[r][t / block_size], slot t % block_size.  The K/V of all
 *   c_r + k_r + 1 tokens must already be in the pool.
 */
#ifndef WISP_VERIFY_H
#define WISP_VERIFY_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  WISP_OK = 0,
  WISP_ERR_INVALID_ARG = 1,  /* a host-visible argument is invalid; nothing was enqueued */
  WISP_ERR_UNSUPPORTED = 2,  /* valid, but outside what the kernels implement; nothing enqueued */
  WISP_ERR_CUDA = 3,         /* a CUDA runtime call failed (launch, attribute, copy) */
  WISP_ERR_WORKSPACE = 4     /* workspace NULL, misaligned or smaller than required */
} wisp_status;

/* Codes of the device status word (see wisp_verify_get_device_status). */
typedef enum {
  WISP_DEV_OK = 0,
  WISP_DEV_BAD_LENGTH = 1,   /* k_r < 0, c_r < 0, c_r + k_r + 1 > max_blocks_per_seq * block_size,
                                or sum of lengths disagrees with total_q_rows / total_draft */
  WISP_DEV_BAD_BLOCK = 2,    /* a block id needed by the request is outside [0, num_blocks) */
  WISP_DEV_BAD_TOKEN = 3,    /* a draft token outside [0, V), anywhere in the draft */
  WISP_DEV_BAD_PROB = 4,     /* a draft probability q(y) that is negative or NaN at a decision the
                                walk takes, or a logit row it reads (rows 0..L) with no finite
                                maximum / no finite positive normaliser (a row without a softmax) */
  WISP_DEV_UNSUPPORTED = 5,  /* (Hq / Hkv) * (k_r + 1) > 128 query rows, or k_r > 1024 */
  WISP_DEV_TIMEOUT = 6,      /* a bounded device-side wait gave up (no kernel waits unboundedly) */
  WISP_DEV_NO_BLOCKS = 7     /* (wisp_kv.h) the free page pool could not serve the request */
} wisp_device_code;

typedef enum { WISP_F32 = 0, WISP_BF16 = 1 } wisp_dtype;

/*
 * Attention of the verification forward (Sec. 4.4-4.5).
 *   q        [total_q_rows, Hq, D]                 dtype qkv_dtype
 *   k_cache  [num_blocks, Hkv, block_size, D]      dtype qkv_dtype (v_cache likewise)
 *   out      [total_q_rows, Hq, D]                 dtype qkv_dtype
 *   out[row, h] = sum_t softmax_t(<q[row, h], K[t, h / (Hq/Hkv)]> / sqrt(D)) V[t, h / (Hq/Hkv)]
 *   over the keys t visible to the row (see the layout note above).
 * Supported: D in {64, 128}, block_size == 16, Hq % Hkv == 0.
 * Accumulation is fp32; bf16 outputs are rounded to nearest even.
 */
typedef struct {
  int32_t B, Hq, Hkv, D;
  int32_t block_size;            /* must be 16 */
  int32_t max_blocks_per_seq;    /* row stride of block_tables */
  int32_t num_blocks;            /* blocks in the pool; ids must lie in [0, num_blocks) */
  int32_t total_q_rows;          /* host copy of sum_r (k_r + 1) (sizes q/out; checked on device) */
  const int64_t *request_ids;    /* [B] echoed in the device status word; may be NULL */
  const int32_t *draft_lens;     /* [B] k_r >= 0 */
  const int32_t *context_lens;   /* [B] c_r >= 0: cached-prefix tokens, not counting the k_r + 1 new ones */
  const int32_t *block_tables;   /* [B, max_blocks_per_seq] */
  wisp_dtype qkv_dtype;
  const void *q;
  const void *k_cache;
  const void *v_cache;
  void *out;
} wisp_attn_args;

/*
 * Acceptance pass (Eq. 1-3).
 *   target_logits   [total_q_rows, V]  dtype logits_dtype; p = softmax of a row (temperature
 *                                      already applied by the caller)
 *   draft_tokens    [total_draft]      int32
 *   draft_probs     [total_draft, V]   fp32 draft distributions, used as given (not renormalised)
 *   accept_uniforms [total_draft]      fp32 in [0, 1): u_i of Eq. 1
 *   sample_uniforms [B]                fp32 in [0, 1): one draw per request for the extra token
 *   accepted_len    [B] out            L_r in [0, k_r]
 *   next_token      [B] out            the extra token of Eq. 3
 * Rule, per request: for i = 1..k_r in order, y = draft token i, a = 1 if q_i(y) == 0 else
 * min(1, p_{i-1}(y) / q_i(y)); accept iff u_i <= a; stop at the first rejection.  With L
 * accepted: if L < k_r the extra token is the inverse-CDF draw (ascending token ids, first t
 * whose cumulative mass is strictly greater than u * total) from max(0, p_L - q_{L+1}); if
 * that residual has no mass, or L == k_r, the draw is from p_L.
 * Supported: 1 <= V <= 2^24.
 * The kernel decides every comparison exactly up to about 1e-13 relative error: it computes
 * the row normaliser in fp32 with a certified error bound and recomputes it in double-float
 * arithmetic whenever a decision lies inside that bound; the extra-token draw sums the weights
 * exp(z - m) of row L as 2^-56 fixed-point integers (exact, order-free sums) and settles the
 * sign of p - q with the certified normaliser, weighing undecided elements exactly.
 * One call is one planner launch and one persistent acceptance kernel on `stream`.
 */
typedef struct {
  int32_t B, V;
  int32_t total_q_rows;          /* host copy of sum_r (k_r + 1) */
  int32_t total_draft;           /* host copy of sum_r k_r */
  const int64_t *request_ids;    /* [B] may be NULL */
  const int32_t *draft_lens;     /* [B] */
  wisp_dtype logits_dtype;
  const void *target_logits;
  const int32_t *draft_tokens;
  const float *draft_probs;
  const float *accept_uniforms;
  const float *sample_uniforms;
  int32_t *accepted_len;
  int32_t *next_token;
} wisp_accept_args;

/* Bytes of workspace needed by a call with these arguments (either pointer may be NULL).
 * Depends on the current device's SM count.  Returns 0 if the arguments are invalid. */
size_t wisp_verify_workspace_size(const wisp_attn_args *attn, const wisp_accept_args *acc);

/* Enqueue the attention (Sec. 4.4-4.5).  See wisp_attn_args. */
wisp_status wisp_verify_attention(const wisp_attn_args *attn, void *workspace, size_t workspace_bytes,
                                  void *stream);

/* Enqueue the acceptance pass (Eq. 1-3).  See wisp_accept_args. */
wisp_status wisp_verify_accept(const wisp_accept_args *acc, void *workspace, size_t workspace_bytes,
                               void *stream);

/* Greedy (temperature 0) variant of the acceptance pass: sampling at temperature 0 takes the most
 * likely token, so draft token i is accepted iff it is the argmax of logit row i-1 (the lowest token
 * id among equal maxima), the walk stops at the first mismatch (Eq. 2) and the extra token is the
 * argmax of row L.  draft_probs, accept_uniforms and sample_uniforms are not read (may be NULL).
 * NaN logits are never chosen; a row without a finite logit is flagged WISP_DEV_BAD_PROB. */
wisp_status wisp_verify_accept_greedy(const wisp_accept_args *acc, void *workspace, size_t workspace_bytes,
                                      void *stream);

/* Enqueue one whole verification step (Sec. 4.5): attention and acceptance.  The two parts
 * read disjoint inputs; draft_lens must describe the same batch in both structs.  One planner
 * serves both; the attention follows it on `stream`, and the acceptance pass (with the
 * acceptance part of the plan) runs on a side stream owned by the library, forked from and
 * joined back into `stream` with events, so work queued on `stream` afterwards sees the whole step
 * finished.  The planner sizes the attention from the batch: when the attention is small next to
 * the acceptance work, part of its CTAs exit at once and the acceptance pass starts on their SMs
 * (results are the same either way).  Each caller stream gets its own side stream (created on its
 * first step: make that first call before any stream capture), so steps on different streams,
 * with different workspaces, run independently. */
wisp_status wisp_verify_step(const wisp_attn_args *attn, const wisp_accept_args *acc, void *workspace,
                             size_t workspace_bytes, void *stream);

/* Acceptance pass (same rule, kernels and results as wisp_verify_accept) that needs no workspace
 * and allocates nothing.  No counterpart in the paper: it exists for callers that cannot allocate
 * device memory when they verify (memory owned by another allocator, or a latency path on which
 * cudaMalloc, which may synchronise the device, is not allowed).
 *   Scratch: a fixed 16 MiB array inside this library's device image, shared by every call in
 *   the process.  Calls that overlap in time (other streams, other host threads) race on it and
 *   corrupt each other's results: order them, e.g. on one stream.
 *   Limit: B <= 8192 requests and total_q_rows <= 131072; a larger batch returns
 *   WISP_ERR_UNSUPPORTED and enqueues nothing.
 *   Set-up: the first call on a device looks up the array's address and sets kernel attributes
 *   (host-side runtime calls, no allocation); make that first call before any stream capture.
 *   Device-data errors are recorded in the scratch's status word, which this entry point does not
 *   expose; a caller that must read them uses wisp_verify_accept with its own workspace. */
wisp_status wisp_verify_accept_noalloc(const wisp_accept_args *acc, void *stream);

/* Read the device status word of `workspace` (synchronous copy; synchronise the stream that
 * ran the step first).  *code receives a wisp_device_code, *request_id the request_ids entry
 * (or the batch index when request_ids was NULL) of the first failing request, or -1. */
wisp_status wisp_verify_get_device_status(const void *workspace, int32_t *code, int64_t *request_id);

const char *wisp_verify_status_string(wisp_status s);
const char *wisp_verify_device_code_string(int32_t code);

#ifdef __cplusplus
}
#endif
#endif /* WISP_VERIFY_H */
