"""GPU: the extra-token draw (Eq. 3) when u * S lies next to an edge of the residual's CDF.

The uniforms are placed about 1e-8 (relative) from an edge of the residual CDF: above the logging
window of the parity tests, far below what fp32 weights or an fp32 normaliser could resolve.  The
GPU's double-float weights and prefix sums must still give the fp64 oracle's token exactly.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2601_11652_gb300 import workload as wl
from tests.gpu_util import SAMPLE_WINDOW, compare_accept

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.fail("GPU tests need a CUDA device")
    from paper_2601_11652_gb300 import build
    build.build()


def _logit_row(batch, i):
    row = batch.logits[i]
    return row


def _edge_uniforms(batch, ref, rng):
    """For every request with a rejection, a float32 u next to an edge of its residual CDF."""
    qs, ds = batch.q_row_start(), batch.draft_start()
    out = {}
    for r in range(batch.B):
        L, k = int(ref["accepted_len"][r]), int(batch.draft_lens[r])
        if L < 0 or L >= k:
            continue
        p = oracle.row_softmax(_logit_row(batch, qs[r] + L), batch.dtype)
        q = batch.draft_probs[ds[r] + L].astype(np.float64)
        res = np.maximum(p - q, 0.0)
        tot = res.sum()
        if not tot > 0:
            continue
        cdf = np.cumsum(res) / tot
        # an edge in the middle of the mass, after an element of non-negligible weight
        cand = np.nonzero((cdf > rng.uniform(0.2, 0.8)) & (res / tot > 1e-5))[0]
        if len(cand) == 0:
            continue
        j = int(cand[0])
        out[r] = np.float32(cdf[j])
    return out


@pytest.mark.parametrize("seed,V", [(11, 40000), (12, 6000)])
def test_draw_next_to_a_cdf_edge_matches_the_oracle(seed, V):
    from paper_2601_11652_gb300.device_batch import DeviceBatch
    rng = np.random.default_rng(seed)
    b = wl.make_small_batch(seed, B=8, Hq=8, Hkv=2, D=128, V=V, dtype="bf16", k_range=(3, 8), ctx_range=(0, 300))
    ref = oracle.accept(b)
    edges = _edge_uniforms(b, ref, rng)
    assert len(edges) >= 3, "the seeds give requests with a rejection"
    for r, u in edges.items():
        b.sample_uniforms[r] = u
    ref = oracle.accept(b)
    # keep the edge requests whose margin is above the logging window (one float32 step off if not)
    for r in list(edges):
        if ref["sample_margin"][r] < SAMPLE_WINDOW:
            b.sample_uniforms[r] = np.nextafter(b.sample_uniforms[r], np.float32(1.0))
    ref = oracle.accept(b)
    near = [r for r in edges if SAMPLE_WINDOW <= ref["sample_margin"][r] < 1e-6]
    assert len(near) >= 3, [float(ref["sample_margin"][r]) for r in edges]
    db = DeviceBatch.from_host(b)
    db.step()
    torch.cuda.synchronize()
    code, rid = db.device_status()
    assert code == 0, (code, rid)
    got = db.results()
    for r in near:
        assert got["accepted_len"][r] == ref["accepted_len"][r]
        assert got["next_token"][r] == ref["next_token"][r], (r, float(ref["sample_margin"][r]))


@pytest.mark.parametrize("shift", [-40.0, 45.0, 75.0])
def test_draw_with_shifted_logits_matches_the_oracle(shift):
    """Row maxima far below 0, near 55 and above the exp table's range (|u| < 64): the table entries
    exp(u - m) reach the float underflow range, or most elements take the direct exp; all must give
    the oracle's tokens."""
    from paper_2601_11652_gb300.device_batch import DeviceBatch
    b = wl.make_small_batch(13, B=12, Hq=8, Hkv=2, D=128, V=40000, dtype="bf16", k_range=(2, 7), ctx_range=(0, 200))
    b.logits = wl.f32_to_bf16_bits(wl.bf16_bits_to_f32(b.logits) + np.float32(shift))
    ref = oracle.accept(b)
    assert np.any(ref["accepted_len"] < b.draft_lens), "some request draws from a residual"
    db = DeviceBatch.from_host(b)
    db.step()
    torch.cuda.synchronize()
    code, rid = db.device_status()
    assert code == 0, (code, rid)
    got = db.results()
    n, _ = compare_accept(b, got["accepted_len"], got["next_token"], ref)
    assert n >= b.B - 2


_SPECIAL = np.array([0x0000, 0x8000, 0x0001, 0x8001,   # +-0, +-smallest subnormal
                     0x3780, 0xB780, 0x377F, 0xB77F,   # +-2^-16 (the exp table's first value) and just below
                     0x3781, 0xB781, 0x427F, 0xC27F,   # just above; +-(64 - ulp) (its last)
                     0x4280, 0xC280, 0xFF80],          # +-64 (past the table), -inf (a masked token)
                    dtype=np.uint16)


@pytest.mark.parametrize("mode", ["near_zero", "large"])
def test_draw_rows_at_the_exp_table_bounds(oracle_mod, mode):
    """Draw rows (residual and bonus) whose logits sit on and next to the bounds of the draw's exp
    table: +-0 and subnormals, +-2^-16 and its neighbours, +-(64 - ulp), +-64, -inf.  Values
    outside the table take the direct exp (or weigh zero for -inf); all must give the oracle's
    tokens."""
    from paper_2601_11652_gb300.device_batch import DeviceBatch
    rng = np.random.default_rng(21 if mode == "near_zero" else 22)
    b = wl.make_small_batch(14, B=12, Hq=8, Hkv=2, D=128, V=6000, dtype="bf16", k_range=(1, 6), ctx_range=(0, 100))
    z = wl.bf16_bits_to_f32(b.logits).astype(np.float32)
    if mode == "near_zero":
        z = rng.normal(0.0, 1.0, size=z.shape).astype(np.float32)  # row maxima about 3-4: the specials carry mass
    else:
        z = rng.normal(62.0, 1.5, size=z.shape).astype(np.float32)  # maxima past 64
    bits = wl.f32_to_bf16_bits(z)
    pick = rng.random(bits.shape) < 0.3
    bits[pick] = rng.choice(_SPECIAL, size=int(pick.sum()))
    bits[:, 0] = wl.f32_to_bf16_bits(np.float32(4.0 if mode == "near_zero" else 66.0))  # a finite maximum
    b.logits = bits
    ref = oracle_mod.accept(b)
    assert np.any(ref["accepted_len"] < b.draft_lens) and np.any(ref["accepted_len"] == b.draft_lens), \
        "residual and bonus draws both occur"
    db = DeviceBatch.from_host(b)
    db.step()
    torch.cuda.synchronize()
    code, rid = db.device_status()
    assert code == 0, (code, rid)
    got = db.results()
    n, _ = compare_accept(b, got["accepted_len"], got["next_token"], ref)
    assert n >= b.B - 2
