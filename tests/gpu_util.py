"""Helpers shared by the GPU parity tests: tolerances and the oracle comparison."""
import numpy as np

# attention: max abs error of the output (bf16 KV + fp32 accumulate; fp32 inputs)
ATTN_TOL = {"bf16": 2e-2, "f32": 1e-4}
# acceptance decisions within this distance of their threshold are logged, not failed
ACCEPT_WINDOW = 1e-6
# the GPU draws the extra token with double-float weights and prefix sums (about 1e-12
# relative error against the fp64 oracle); draws within this normalised distance of a
# CDF edge are logged, not failed
SAMPLE_WINDOW = 1e-9


def compare_accept(batch, gpu_L, gpu_tok, ref):
    """Bit-exact comparison of accepted_len / next_token except logged near-threshold requests.

    Returns (n_compared, list of logged request indices)."""
    L, tok = ref["accepted_len"], ref["next_token"]
    near = (ref["accept_margin"] < ACCEPT_WINDOW) | (ref["sample_margin"] < SAMPLE_WINDOW)
    logged = [int(r) for r in np.nonzero(near)[0]]
    ok = ~near
    bad = np.nonzero(ok & ((gpu_L != L) | (gpu_tok != tok)))[0]
    assert len(bad) == 0, (
        f"{len(bad)} requests differ from the oracle, first {bad[:5]}: "
        f"gpu L={gpu_L[bad[:5]]} tok={gpu_tok[bad[:5]]} oracle L={L[bad[:5]]} tok={tok[bad[:5]]}")
    # logged ones must still be valid results
    for r in logged:
        assert 0 <= gpu_L[r] <= batch.draft_lens[r] and 0 <= gpu_tok[r] < batch.V
    return int(ok.sum()), logged


def attn_max_err(gpu_out, ref_out):
    return float(np.max(np.abs(gpu_out.astype(np.float64) - ref_out))) if ref_out.size else 0.0


def subset_rows(batch, reqs):
    qs = batch.q_row_start()
    return np.concatenate([np.arange(qs[r], qs[r + 1]) for r in reqs])


def request_groups(batch, max_row_keys=2e8):
    """Consecutive groups of requests whose oracle attention work (query rows x visible keys x
    heads) stays under max_row_keys each, so that every oracle call is bounded."""
    kv = batch.context_lens.astype(np.int64) + batch.draft_lens + 1
    work = (batch.draft_lens.astype(np.int64) + 1) * kv * batch.Hq
    groups, cur, acc = [], [], 0
    for r in range(batch.B):
        if cur and acc + work[r] > max_row_keys:
            groups.append(cur)
            cur, acc = [], 0
        cur.append(r)
        acc += int(work[r])
    if cur:
        groups.append(cur)
    return groups
