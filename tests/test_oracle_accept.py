"""Pins of the oracle's acceptance pass (Eq. 1-3 and the lossless target-token draw).

Pins used: hand-worked examples (tests/golden/accept_hand.json), invariants
the rule must satisfy (p == q accepts everything, 0 <= L <= k, monotone in u,
residual support), a special case that reduces to a library inverse CDF
(k = 0 is a plain draw from p), the exact output law by enumeration (k = 1),
and the lossless law checked statistically (chi-square over 10^6 trials,
plus the closed form of E[L]).
"""
import json
import os

import numpy as np
import pytest
from scipy.special import softmax
from scipy.stats import chisquare

from paper_2601_11652_gb300 import workload as wl

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


class _Batch:
    """Minimal acceptance-only batch (attributes the oracle reads)."""

    def __init__(self, logits, draft_lens, draft_tokens, draft_probs, accept_u, sample_u, dtype="f32"):
        self.logits = np.ascontiguousarray(logits, dtype=np.float32)
        self.V = self.logits.shape[1]
        self.draft_lens = np.asarray(draft_lens, np.int32)
        self.draft_tokens = np.asarray(draft_tokens, np.int32)
        self.draft_probs = np.ascontiguousarray(np.asarray(draft_probs, np.float32).reshape(-1, self.V))
        self.accept_uniforms = np.asarray(accept_u, np.float32)
        self.sample_uniforms = np.asarray(sample_u, np.float32)
        self.dtype = dtype


def test_hand_worked_examples(oracle_mod):
    with open(os.path.join(GOLDEN, "accept_hand.json")) as f:
        g = json.load(f)
    for req in g["requests"]:
        b = _Batch(req["logit_rows"], [len(req["draft_tokens"])], req["draft_tokens"],
                   np.asarray(req["draft_rows"], np.float32).reshape(-1, g["V"]), req["accept_u"], [req["sample_u"]])
        out = oracle_mod.accept(b)
        assert out["accepted_len"][0] == req["expected_accepted_len"], req["name"]
        assert out["next_token"][0] == req["expected_next_token"], req["name"]


def _random_rows(rng, n, V, sd=2.0):
    return (sd * rng.standard_normal((n, V))).astype(np.float32)


def test_p_equals_q_accepts_every_draft(oracle_mod):
    rng = np.random.default_rng(1)
    B, V = 200, 300
    k = rng.integers(0, 9, size=B)
    logits = _random_rows(rng, int(k.sum()) + B, V)
    qs = np.concatenate([[0], np.cumsum(k + 1)])
    probs, toks = [], []
    for r in range(B):
        for j in range(k[r]):
            p = softmax(logits[qs[r] + j].astype(np.float64)).astype(np.float32)
            probs.append(p)
            toks.append(rng.choice(V, p=p / p.sum()))
    # a = min(1, p/q) is within float32 rounding of 1; keep u below that band
    au = rng.uniform(0, 1 - 1e-6, size=int(k.sum()))
    b = _Batch(logits, k, toks, np.array(probs).reshape(-1, V), au, rng.random(B))
    out = oracle_mod.accept(b)
    np.testing.assert_array_equal(out["accepted_len"], k)


def test_ranges_and_residual_support(oracle_mod):
    b = wl.make_small_batch(3, B=60, Hq=2, Hkv=1, D=16, V=500, dtype="bf16", k_range=(0, 10), ctx_range=(0, 4))
    out = oracle_mod.accept(b)
    L, t = out["accepted_len"], out["next_token"]
    assert np.all((0 <= L) & (L <= b.draft_lens))
    assert np.all((0 <= t) & (t < b.V))
    qs, ds = b.q_row_start(), b.draft_start()
    z = wl.bf16_bits_to_f32(b.logits).astype(np.float64)
    rejected = 0
    for r in range(b.B):
        if L[r] < b.draft_lens[r]:
            rejected += 1
            p = softmax(z[qs[r] + L[r]])
            q = b.draft_probs[ds[r] + L[r]].astype(np.float64)
            assert p[t[r]] > q[t[r]], "a residual draw must land where p > q"
            # the rejected draft token itself had u > a
            y = b.draft_tokens[ds[r] + L[r]]
            assert b.accept_uniforms[ds[r] + L[r]] > min(1.0, p[y] / q[y])
    assert rejected > 10


def test_monotone_coupling_in_u(oracle_mod):
    b = wl.make_small_batch(4, B=80, Hq=2, Hkv=1, D=16, V=200, dtype="f32", k_range=(1, 8), ctx_range=(0, 4))
    base = oracle_mod.accept(b)["accepted_len"]
    rng = np.random.default_rng(7)
    for _ in range(5):
        lowered = wl.VerifyBatch(**{**b.__dict__,
                                    "accept_uniforms": (b.accept_uniforms * rng.uniform(0, 1, b.accept_uniforms.shape)).astype(np.float32)})
        assert np.all(oracle_mod.accept(lowered)["accepted_len"] >= base)
    zero = wl.VerifyBatch(**{**b.__dict__, "accept_uniforms": np.zeros_like(b.accept_uniforms)})
    np.testing.assert_array_equal(oracle_mod.accept(zero)["accepted_len"], b.draft_lens)  # u = 0 <= a always


def test_plain_decode_is_library_inverse_cdf(oracle_mod):
    # k = 0 for every request: next_token is the inverse-CDF draw from p (numpy searchsorted on the cumsum)
    rng = np.random.default_rng(11)
    B, V = 400, 1000
    logits = _random_rows(rng, B, V)
    su = rng.random(B).astype(np.float32)
    out = oracle_mod.accept(_Batch(logits, np.zeros(B), [], np.zeros((0, V)), [], su))
    assert np.all(out["accepted_len"] == 0)
    for r in range(B):
        cdf = np.cumsum(softmax(logits[r].astype(np.float64)))
        ref = int(np.searchsorted(cdf, float(su[r]) * cdf[-1], side="right"))
        if out["sample_margin"][r] > 1e-12:
            assert out["next_token"][r] == ref


def test_exact_law_by_enumeration_k1(oracle_mod):
    """k = 1, V = 5: P(first emitted token = t) must equal p_0(t) (losslessness, Sec. 4 opening).

    The law is assembled from the oracle's own decisions on fine midpoint grids of the two
    uniforms: P(token=t) = sum_y q(y) [P_u(accept | y) 1{t=y} + P_u(reject | y) P_us(draw=t | reject)].
    """
    V, N = 5, 4000
    z0 = np.array([0.3, -1.2, 2.0, 0.0, 0.9], np.float32)
    z1 = np.array([1.0, 0.0, -0.5, 0.2, 0.1], np.float32)
    q0 = np.array([0.05, 0.35, 0.2, 0.3, 0.1], np.float32)
    grid = ((np.arange(N) + 0.5) / N).astype(np.float32)
    p0 = softmax(z0.astype(np.float64))
    law = np.zeros(V)
    for y in range(V):
        acc = oracle_mod.accept(_Batch(np.tile(np.stack([z0, z1]), (N, 1)), np.ones(N), np.full(N, y),
                                       np.tile(q0, (N, 1)), grid, np.full(N, 0.5)))
        p_acc = float(np.mean(acc["accepted_len"] == 1))
        # residual draw law: force a rejection (u = 1 > a unless a == 1) and sweep the sample uniform
        rej = oracle_mod.accept(_Batch(np.tile(np.stack([z0, z1]), (N, 1)), np.ones(N), np.full(N, y),
                                       np.tile(q0, (N, 1)), np.ones(N), grid))
        if p_acc < 1.0:
            assert np.all(rej["accepted_len"] == 0)
            draw = np.bincount(rej["next_token"], minlength=V) / N
        else:
            draw = np.zeros(V)
        law += float(q0[y]) * (p_acc * np.eye(V)[y] + (1.0 - p_acc) * draw)
    law /= q0.astype(np.float64).sum()
    assert np.max(np.abs(law - p0)) < 3.0 / N


@pytest.mark.parametrize("seed", [0])
def test_lossless_chi_square_1e6(oracle_mod, seed):
    """V = 8, k = 3, 10^6 trials with y_j ~ q_j: first emitted token ~ p_0, second (given L >= 1) ~ p_1."""
    rng = np.random.default_rng(seed)
    V, k, N = 8, 3, 1_000_000
    z = (1.5 * rng.standard_normal((k + 1, V))).astype(np.float32)
    qrows = softmax(z[:k].astype(np.float64) + 0.8 * rng.standard_normal((k, V)), axis=1).astype(np.float32)
    p = softmax(z.astype(np.float64), axis=1)
    assert p.min() > 1e-3
    qn = qrows.astype(np.float64) / qrows.astype(np.float64).sum(axis=1, keepdims=True)
    toks = np.stack([rng.choice(V, size=N, p=qn[j]) for j in range(k)], axis=1).astype(np.int32)
    b = _Batch(np.tile(z, (N, 1)), np.full(N, k), toks.reshape(-1), np.tile(qrows, (N, 1)),
               rng.random(N * k), rng.random(N))
    out = oracle_mod.accept(b)
    L, t = out["accepted_len"], out["next_token"]
    first = np.where(L >= 1, toks[:, 0], t)
    assert chisquare(np.bincount(first, minlength=V), p[0] * N).pvalue > 0.01
    sel = L >= 1
    second = np.where(L[sel] >= 2, toks[sel, 1], t[sel])
    assert chisquare(np.bincount(second, minlength=V), p[1] * sel.sum()).pvalue > 0.01
    # E[L] = sum_j prod_{i<j} alpha_i with alpha_i = sum_v min(p_i, q_i) (rows independent here)
    alpha = np.minimum(p[:k], qrows.astype(np.float64)).sum(axis=1)
    expect = sum(np.prod(alpha[:j]) for j in range(1, k + 1))
    assert abs(L.mean() - expect) < 4 * L.std() / np.sqrt(N)


def test_rejects_out_of_range_token(oracle_mod):
    b = _Batch([[0, 0, 0, 0], [0, 0, 0, 0]], [1], [7], [[0.25] * 4], [0.5], [0.5])
    with pytest.raises(ValueError):
        oracle_mod.accept(b)
    out = oracle_mod.accept(b, check=False)
    assert out["status"][0] == 4 and out["accepted_len"][0] == -1


def test_undefined_softmax_rows_are_flagged(oracle_mod):
    """A logit row the rule reads must have a softmax: every logit -inf, a +inf or a NaN logit
    flags the request (status bad_prob = 5); a -inf entry among finite ones is an ordinary zero
    probability.  The other request of the batch is unaffected."""
    ninf, pinf, nan = -np.inf, np.inf, np.nan
    fine = [0.0, 1.0, -1.0, 0.5]
    for bad_row in ([ninf] * 4, [0.0, pinf, 1.0, 2.0], [0.0, nan, 1.0, 2.0]):
        # request 0: one draft token, rows 0 (decision) and 1; request 1: k = 0, one row
        b = _Batch([bad_row, fine, fine], [1, 0], [2], [[0.25] * 4], [0.1], [0.3, 0.6])
        out = oracle_mod.accept(b, check=False)
        assert out["status"].tolist() == [5, 0], bad_row
        assert out["accepted_len"][0] == -1 and out["next_token"][0] == -1
        ref = oracle_mod.accept(_Batch([fine], [0], [], [], [], [0.6]))
        assert out["next_token"][1] == ref["next_token"][0]
    # the draw row (row L) is read too: after a full acceptance the bonus row is all -inf
    b = _Batch([fine, [ninf] * 4], [1], [1], [[0.25] * 4], [0.0], [0.5])
    assert oracle_mod.accept(b, check=False)["status"][0] == 5
    # -inf among finite logits: p = 0 there, never drawn
    masked = [ninf, 1.0, ninf, 1.0]
    out = oracle_mod.accept(_Batch([masked], [0], [], [], [], [0.99]))
    assert out["status"][0] == 0 and out["next_token"][0] == 3


def test_out_of_range_token_anywhere_in_the_draft_is_flagged(oracle_mod):
    """The whole draft is validated, also a token after the first rejection (status bad_token = 4)."""
    rows = [[0.0, 0.0, 0.0, 0.0]] * 3
    # token 0 has p = 0.25 against q = 1.0: rejected with u = 0.9; token 1 is out of range
    b = _Batch(rows, [2], [0, 9], [[1.0, 0.0, 0.0, 0.0], [0.25] * 4], [0.9, 0.1], [0.5])
    out = oracle_mod.accept(b, check=False)
    assert out["status"][0] == 4 and out["accepted_len"][0] == -1
