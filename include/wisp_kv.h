/*
 * wisp_kv.h -- C ABI of the paged KV-cache maintenance around the verification step.
 *
 * WISP keeps each session's committed prefix in a PageAttention-style paged KV pool and a prefix
 * cache that is updated in place, so that a verification forwards only the newly drafted block
 * (Sec. 4.5, "Efficient consecutive verifications with PageAttention and prefix cache").  Around one
 * verification step (wisp_verify.h) that means:
 *   before: every request needs pages for its c_r cached tokens plus the k_r + 1 new ones, and the
 *           K/V of the new tokens (computed by the caller's projections) written at positions
 *           c_r .. c_r + k_r;                                   -> wisp_kv_reserve_append
 *   after:  the prefix grows by the last committed token and the L_r accepted drafts
 *           (c_r <- c_r + 1 + L_r, Eq. 2's L); the rejected drafts' K/V are dropped and pages past
 *           the new length go back to the pool.                  -> wisp_kv_commit
 *
 * Pool bookkeeping lives on the device: free_blocks is a stack of free page ids whose first
 * *free_count entries are valid; block_tables rows hold page ids, -1 for "no page".
 * Conventions as in wisp_verify.h: device pointers owned by the caller, asynchronous calls on
 * `stream`, host-visible argument errors returned before anything is enqueued, data errors recorded
 * in the workspace's status word (read with wisp_verify_get_device_status) with the request skipped.
 * Calls that share a pool (or a workspace) must not overlap in time.
 */
#ifndef WISP_KV_H
#define WISP_KV_H

#include "wisp_verify.h"

#ifdef __cplusplus
extern "C" {
#endif

typedef struct {
  int32_t B, Hkv, D;
  int32_t block_size;           /* must be 16 */
  int32_t max_blocks_per_seq;   /* row stride of block_tables */
  int32_t num_blocks;           /* pages in the pool (and capacity of free_blocks) */
  int32_t total_q_rows;         /* host copy of sum_r (k_r + 1): rows of k_new / v_new */
  const int64_t *request_ids;   /* [B] echoed in the device status word; may be NULL */
  const int32_t *draft_lens;    /* [B] k_r >= 0 */
  int32_t *context_lens;        /* [B] c_r; wisp_kv_commit advances it */
  int32_t *block_tables;        /* [B, max_blocks_per_seq] page ids, -1 = none */
  int32_t *free_blocks;         /* [num_blocks] stack of free page ids */
  int32_t *free_count;          /* [1] valid entries of free_blocks */
  wisp_dtype kv_dtype;          /* F32 or BF16 */
  void *k_cache, *v_cache;      /* [num_blocks, Hkv, block_size, D] */
  const void *k_new, *v_new;    /* [total_q_rows, Hkv, D], rows ordered as the queries of wisp_verify.h
                                   (request r's k_r + 1 rows start at sum_{r'<r} (k_r' + 1)); may be NULL
                                   for wisp_kv_commit */
  const int32_t *accepted_len;  /* [B] L_r in [0, k_r] (wisp_kv_commit); may be NULL for reserve_append */
} wisp_kv_args;

/* Bytes of workspace the KV calls need for these arguments; 0 if they are invalid. */
size_t wisp_kv_workspace_size(const wisp_kv_args *kv);

/* Give every request the pages for tokens 0 .. c_r + k_r (table entries that are -1 are filled from
 * the top of the free stack, requests served in order; a request the pool cannot serve entirely gets
 * no page and is flagged WISP_DEV_NO_BLOCKS, and so is every later one), then write request r's new
 * K/V rows j = 0..k_r at positions c_r + j.  Pages already in the table are kept. */
wisp_status wisp_kv_reserve_append(const wisp_kv_args *kv, void *workspace, size_t workspace_bytes, void *stream);

/* After acceptance (Eq. 2): c_r <- c_r + 1 + L_r; the pages of request r that covered tokens
 * 0 .. c_r + k_r (old c_r) but lie past the new length (table indices ceil(new c_r / block_size) ..
 * ceil((old c_r + k_r + 1) / block_size) - 1) are pushed back on the free stack (in table order,
 * requests in order) and their entries set to -1, which rolls back the rejected drafts.  A request
 * with L_r outside [0, k_r] is flagged WISP_DEV_BAD_LENGTH and left unchanged. */
wisp_status wisp_kv_commit(const wisp_kv_args *kv, void *workspace, size_t workspace_bytes, void *stream);

#ifdef __cplusplus
}
#endif
#endif /* WISP_KV_H */
