/*
 * oracle.c -- plain, slow fp64 CPU oracle of the WISP verification step.
 *
 * TEST INFRASTRUCTURE ONLY.  Only the tests, __graft_entry__.smoke() and the
 * cpu_baseline / reference legs of bench.py may load this file's library.  It
 * shares no code, header, table or helper with the CUDA library and never
 * reads anything that library produced.
 *
 * What it computes (arxiv 2601.11652):
 *   - oracle_attention: the attention of the verification engine's one-step
 *     forward (Sec. 4.5): every one of a request's k+1 new query tokens attends
 *     to L_total = L_cached + L_new keys (Sec. 4.4, definition of
 *     N_interactions), causal within the new block, read through the request's
 *     paged KV block table (PageAttention layout, Sec. 4.5).  Written as the
 *     plain definition: gather, scores, softmax with a two-pass max/sum, weighted
 *     sum of values.
 *   - oracle_accept: the in-order acceptance rule of Eq. 1 (a_i = min(1, p/q),
 *     A_i = 1[u_i <= a_i]), the stopping index of Eq. 2 (R = first rejection,
 *     L = R - 1) and the target token of Eq. 3 at the stopping position, read
 *     as the lossless residual draw norm(max(0, p - q)) when R <= K (the
 *     standard speculative sampling algorithm the paper states it follows,
 *     Sec. 4 opening) and as a draw from p when R = K + 1.
 * Readings where the paper is silent (all listed in the design notes):
 *   logits row i of a request scores draft token i+1, row k is the bonus row;
 *   u == a accepts; q(y) == 0 gives a = 1; draws use inverse CDF in ascending
 *   token order with a strict ">" against u * (total mass); no temperature.
 *
 * All arithmetic is IEEE double.  Inputs are exact float32 or bfloat16 values.
 * Functions return 0 on success, or a positive code naming the first invalid
 * input met (they never read out of bounds on invalid ids).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define OR_F32 0
#define OR_BF16 1

#define OR_OK 0
#define OR_BAD_ARG 1
#define OR_BAD_LENGTH 2
#define OR_BAD_BLOCK 3
#define OR_BAD_TOKEN 4
#define OR_BAD_PROB 5

static double bf16_value(uint16_t bits) {
    uint32_t u = ((uint32_t)bits) << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

static double elem(const void *base, int dtype, int64_t i) {
    if (dtype == OR_F32) return (double)((const float *)base)[i];
    return bf16_value(((const uint16_t *)base)[i]);
}

/* ------------------------------------------------------------------------ */
/* Attention                                                                */
/* ------------------------------------------------------------------------ */

/*
 * q      [T_q, Hq, D]              T_q = sum_r (k_r + 1)
 * k, v   [num_blocks, Hkv, bs, D]
 * block_tables [B, max_blocks]     physical block of logical block t / bs
 * out    [T_q, Hq, D] doubles
 * Request r's query j (0..k_r) sits at absolute position c_r + j and sees keys
 * 0 .. c_r + j.  Query head h reads KV head h / (Hq / Hkv).
 */
int oracle_attention(int B, int Hq, int Hkv, int D, int bs, int max_blocks, int num_blocks,
                     const int32_t *draft_lens, const int32_t *context_lens,
                     const int32_t *block_tables, int dtype, const void *q,
                     const void *kc, const void *vc, double *out, int nthreads) {
    if (B < 0 || Hq <= 0 || Hkv <= 0 || Hq % Hkv != 0 || D <= 0 || bs <= 0) return OR_BAD_ARG;
    int64_t *row0 = (int64_t *)malloc(sizeof(int64_t) * (size_t)(B + 1));
    if (!row0) return OR_BAD_ARG;
    row0[0] = 0;
    for (int r = 0; r < B; ++r) {
        if (draft_lens[r] < 0 || context_lens[r] < 0) { free(row0); return OR_BAD_LENGTH; }
        int64_t n = (int64_t)context_lens[r] + draft_lens[r] + 1;
        if (n > (int64_t)max_blocks * bs) { free(row0); return OR_BAD_LENGTH; }
        for (int64_t t = 0; t < n; t += bs) {
            int32_t blk = block_tables[(int64_t)r * max_blocks + t / bs];
            if (blk < 0 || blk >= num_blocks) { free(row0); return OR_BAD_BLOCK; }
        }
        row0[r + 1] = row0[r] + draft_lens[r] + 1;
    }
    const int g = Hq / Hkv;
    const double scale = 1.0 / sqrt((double)D);

    (void)nthreads;
#pragma omp parallel for schedule(dynamic, 1) num_threads(nthreads > 0 ? nthreads : 1)
    for (int64_t job = 0; job < (int64_t)B * Hq; ++job) {
        const int r = (int)(job / Hq), h = (int)(job % Hq), kvh = h / g;
        const int64_t n = (int64_t)context_lens[r] + draft_lens[r] + 1;
        double *kk = (double *)malloc(sizeof(double) * (size_t)(n * D));
        double *vv = (double *)malloc(sizeof(double) * (size_t)(n * D));
        double *s = (double *)malloc(sizeof(double) * (size_t)n);
        /* gather K_r, V_r through the block table */
        for (int64_t t = 0; t < n; ++t) {
            const int64_t blk = block_tables[(int64_t)r * max_blocks + t / bs];
            const int64_t base = ((blk * Hkv + kvh) * bs + t % bs) * (int64_t)D;
            for (int d = 0; d < D; ++d) {
                kk[t * D + d] = elem(kc, dtype, base + d);
                vv[t * D + d] = elem(vc, dtype, base + d);
            }
        }
        for (int j = 0; j <= draft_lens[r]; ++j) {
            const int64_t row = row0[r] + j;
            const int64_t visible = (int64_t)context_lens[r] + j + 1;
            const int64_t qbase = (row * Hq + h) * (int64_t)D;
            double mx = -INFINITY;
            for (int64_t t = 0; t < visible; ++t) {
                double acc = 0.0;
                for (int d = 0; d < D; ++d) acc += elem(q, dtype, qbase + d) * kk[t * D + d];
                s[t] = acc * scale;
                if (s[t] > mx) mx = s[t];
            }
            double denom = 0.0;
            for (int64_t t = 0; t < visible; ++t) {
                s[t] = exp(s[t] - mx);
                denom += s[t];
            }
            for (int d = 0; d < D; ++d) {
                double o = 0.0;
                for (int64_t t = 0; t < visible; ++t) o += s[t] * vv[t * D + d];
                out[qbase + d] = o / denom;
            }
        }
        free(kk);
        free(vv);
        free(s);
    }
    free(row0);
    return OR_OK;
}

/* ------------------------------------------------------------------------ */
/* Acceptance and the target token                                          */
/* ------------------------------------------------------------------------ */

/* p(v) = exp(z_v - max z) / sum_w exp(z_w - max z) for one logit row.  Returns 0 when the
 * softmax is undefined: no finite maximum (every logit -inf, or a +inf one) or a normaliser that
 * is not a finite positive number (a NaN logit); p is then not meaningful. */
static int row_softmax_checked(int V, int dtype, const void *row, double *p) {
    double mx = -INFINITY;
    for (int v = 0; v < V; ++v) {
        double z = elem(row, dtype, v);
        if (z > mx) mx = z;
    }
    double Z = 0.0;
    for (int v = 0; v < V; ++v) {
        p[v] = exp(elem(row, dtype, v) - mx);
        Z += p[v];
    }
    for (int v = 0; v < V; ++v) p[v] /= Z;
    return isfinite(mx) && Z > 0.0 && isfinite(Z);
}

void oracle_row_softmax(int V, int dtype, const void *row, double *p) {
    (void)row_softmax_checked(V, dtype, row, p);
}

/*
 * Inverse-CDF draw from the unnormalised non-negative weights w[0..V):
 * the smallest t with sum_{v<=t} w_v > u * S (S = sum w), or, if rounding
 * leaves no such t, the largest t with w_t > 0.  *margin receives the distance
 * from u*S to the nearer edge of t's interval, divided by S.  Returns -1 if
 * S <= 0.
 */
static int inverse_cdf(int V, const double *w, double u, double *margin) {
    double S = 0.0;
    for (int v = 0; v < V; ++v) S += w[v];
    if (!(S > 0.0)) return -1;
    const double thr = u * S;
    double below = 0.0;
    for (int v = 0; v < V; ++v) {
        const double above = below + w[v];
        if (above > thr) {
            const double m1 = thr - below, m2 = above - thr;
            *margin = (m1 < m2 ? m1 : m2) / S;
            return v;
        }
        below = above;
    }
    int last = V - 1;
    while (last > 0 && !(w[last] > 0.0)) --last;
    *margin = 0.0;
    return last;
}

/*
 * logits      [T_q, V]   k_r + 1 rows per request, request-major
 * draft_probs [T_d, V]   fp32, used exactly as given
 * draft_tokens, accept_u [T_d];  sample_u [B]
 * Outputs per request: accepted_len (L), next_token, accept_margin (smallest
 * |u_i - a_i| over the decisions taken, +inf if none), sample_margin
 * (normalised distance of u * S to the drawn token's interval edge), status.
 */
int oracle_accept(int B, int V, const int32_t *draft_lens, int dtype, const void *logits,
                  const int32_t *draft_tokens, const float *draft_probs,
                  const float *accept_u, const float *sample_u, int32_t *accepted_len,
                  int32_t *next_token, double *accept_margin, double *sample_margin,
                  int32_t *status, int nthreads) {
    if (B < 0 || V <= 0) return OR_BAD_ARG;
    int64_t *row0 = (int64_t *)malloc(sizeof(int64_t) * (size_t)(B + 1));
    int64_t *d0 = (int64_t *)malloc(sizeof(int64_t) * (size_t)(B + 1));
    if (!row0 || !d0) { free(row0); free(d0); return OR_BAD_ARG; }
    row0[0] = 0;
    d0[0] = 0;
    for (int r = 0; r < B; ++r) {
        if (draft_lens[r] < 0) { free(row0); free(d0); return OR_BAD_LENGTH; }
        row0[r + 1] = row0[r] + draft_lens[r] + 1;
        d0[r + 1] = d0[r] + draft_lens[r];
    }
    int first_err = OR_OK;
    const size_t esz = dtype == OR_F32 ? 4 : 2;

    (void)nthreads;
#pragma omp parallel for schedule(dynamic, 16) num_threads(nthreads > 0 ? nthreads : 1)
    for (int r = 0; r < B; ++r) {
        const int k = draft_lens[r];
        double *p = (double *)malloc(sizeof(double) * (size_t)V);
        double *w = (double *)malloc(sizeof(double) * (size_t)V);
        int st = OR_OK, L = k;
        double amargin = INFINITY;
        /* a draft token outside [0, V) anywhere in the draft makes the request invalid */
        for (int j = 0; j < k; ++j) {
            const int32_t y = draft_tokens[d0[r] + j];
            if (y < 0 || y >= V) { st = OR_BAD_TOKEN; break; }
        }
        /* Eq. 1-2: walk the draft in order, stop at the first rejection */
        for (int j = 1; j <= k && st == OR_OK; ++j) {
            const int64_t drow = d0[r] + j - 1;
            const int32_t y = draft_tokens[drow];
            if (y < 0 || y >= V) { st = OR_BAD_TOKEN; break; }
            const double qy = (double)draft_probs[drow * V + y];
            if (!(qy >= 0.0)) { st = OR_BAD_PROB; break; }
            if (!row_softmax_checked(V, dtype, (const char *)logits + (size_t)(row0[r] + j - 1) * V * esz, p)) {
                st = OR_BAD_PROB;
                break;
            }
            const double a = (qy == 0.0) ? 1.0 : fmin(1.0, p[y] / qy);
            const double u = (double)accept_u[drow];
            const double gap = fabs(u - a);
            if (gap < amargin) amargin = gap;
            if (!(u <= a)) { L = j - 1; break; }
        }
        int t = -1;
        double smargin = 0.0;
        if (st == OR_OK) {
            /* Eq. 3 at the stopping position: residual on rejection, p after a full accept */
            if (!row_softmax_checked(V, dtype, (const char *)logits + (size_t)(row0[r] + L) * V * esz, p))
                st = OR_BAD_PROB;
        }
        if (st == OR_OK) {
            if (L < k) {
                const float *qrow = draft_probs + (size_t)(d0[r] + L) * V;
                for (int v = 0; v < V; ++v) {
                    const double diff = p[v] - (double)qrow[v];
                    w[v] = diff > 0.0 ? diff : 0.0;
                }
                t = inverse_cdf(V, w, (double)sample_u[r], &smargin);
            }
            if (t < 0) t = inverse_cdf(V, p, (double)sample_u[r], &smargin);
            if (t < 0) st = OR_BAD_PROB;
        }
        accepted_len[r] = st == OR_OK ? L : -1;
        next_token[r] = st == OR_OK ? t : -1;
        accept_margin[r] = amargin;
        sample_margin[r] = smargin;
        status[r] = st;
        if (st != OR_OK) {
#pragma omp critical
            if (first_err == OR_OK) first_err = st;
        }
        free(p);
        free(w);
    }
    free(row0);
    free(d0);
    return first_err;
}
