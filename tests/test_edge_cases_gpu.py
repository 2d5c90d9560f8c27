"""GPU parity on the acceptance rule's edge cases and the extreme shapes (Eq. 1-3, Sec. 4.5).

Every case is compared with the fp64 oracle on the same inputs: accepted_len / next_token bit
for bit (outside the logged windows), attention within the dtype's tolerance.

  * a drafted token with q(y) = 0: Eq. 1 with a := 1, so it is accepted whatever u is;
  * logit rows with -inf entries among finite ones (a masked vocabulary), bf16 and fp32, on the
    rows the walk decides on and on the rows the extra token is drawn from, including a drafted
    token whose logit is -inf (p(y) = 0: rejected unless u = 0);
  * a drafted token far below the row maximum (p(y) below the float range) with a subnormal q(y);
  * a batch in which every request has k = 0 (plain decode only, no draft arrays);
  * B = 1 at a 131072-token context with the pages shuffled over the pool (the deepest split-KV
    path: 8 (request, KV head) pairs over all SMs);
  * fp32 logits over a 152064-token vocabulary;
  * a rejection whose residual max(0, p - q) has no mass (q = 2p, left unnormalised): the extra
    token is then drawn from p_L.
"""
import numpy as np
import pytest
import torch

from paper_2601_11652_gb300 import workload as wl
from tests.gpu_util import ATTN_TOL, attn_max_err, compare_accept

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.fail("GPU tests need a CUDA device")
    from paper_2601_11652_gb300 import build
    build.build()


def _run(batch, mode="step"):
    from paper_2601_11652_gb300.device_batch import DeviceBatch
    db = DeviceBatch.from_host(batch)
    getattr(db, mode)()
    torch.cuda.synchronize()
    code, rid = db.device_status()
    assert code == 0, f"device status {code} (request {rid})"
    return db.results()


def _z(batch):
    """Logits as float32 (a copy)."""
    return wl.bf16_bits_to_f32(batch.logits) if batch.dtype == "bf16" else batch.logits.astype(np.float32)


def _set_z(batch, z):
    batch.logits = wl.f32_to_bf16_bits(z) if batch.dtype == "bf16" else z.astype(np.float32)


def _check(oracle_mod, b, mode="step", with_attention=True):
    got = _run(b, mode)
    ref = oracle_mod.accept(b)
    n, logged = compare_accept(b, got["accepted_len"], got["next_token"], ref)
    assert n >= b.B - 1
    if with_attention:
        err = attn_max_err(got["out"], oracle_mod.attention(b))
        assert err <= ATTN_TOL[b.dtype], f"attention max abs error {err}"
    return got, ref


def test_zero_draft_probability_accepts(oracle_mod):
    b = wl.make_small_batch(31, B=8, Hq=8, Hkv=2, D=128, V=20000, dtype="bf16", k_range=(2, 6), ctx_range=(0, 300))
    ds = b.draft_start()
    b.draft_probs = b.draft_probs.copy()
    b.accept_uniforms = b.accept_uniforms.copy()
    for r in range(b.B):
        d = ds[r]  # the first decision of every request
        b.draft_probs[d, b.draft_tokens[d]] = 0.0
        b.accept_uniforms[d] = np.float32(0.9999)  # would reject for any a < 0.9999
    got, ref = _check(oracle_mod, b, "accept", with_attention=False)
    assert np.all(ref["accepted_len"] >= 1) and np.all(got["accepted_len"] >= 1)


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_masked_vocabulary_rows(oracle_mod, dtype):
    V = 30000 if dtype == "bf16" else 9000
    b = wl.make_small_batch(32, B=8, Hq=8, Hkv=2, D=128, V=V, dtype=dtype, k_range=(0, 7), ctx_range=(0, 400))
    rng = np.random.default_rng(32)
    z = _z(b)
    mask = rng.random(z.shape) < 0.3
    # keep every drafted token visible except in request 1, whose first drafted token is masked
    qs, ds = b.q_row_start(), b.draft_start()
    for r in range(b.B):
        for j in range(int(b.draft_lens[r])):
            mask[qs[r] + j, b.draft_tokens[ds[r] + j]] = (r == 1 and j == 0)
    z[mask] = -np.inf
    _set_z(b, z)
    got, ref = _check(oracle_mod, b, "step")
    if b.draft_lens[1] > 0:
        assert ref["accepted_len"][1] == 0  # p(y_1) = 0: rejected (u > 0)
    # the drawn tokens are never masked ones
    for r in range(b.B):
        assert not mask[qs[r] + got["accepted_len"][r], got["next_token"][r]]


def test_far_below_max_token_with_subnormal_q(oracle_mod):
    b = wl.make_small_batch(33, B=6, Hq=8, Hkv=2, D=128, V=20000, dtype="bf16", k_range=(2, 5), ctx_range=(0, 200))
    z = _z(b)
    qs, ds = b.q_row_start(), b.draft_start()
    b.draft_probs = b.draft_probs.copy()
    for r in range(b.B):
        y = b.draft_tokens[ds[r]]
        z[qs[r], y] = np.float32(z[qs[r]].max() - 95.0)            # p(y) about e^-95 / Z
        b.draft_probs[ds[r], y] = np.float32(1.4e-45)            # the smallest subnormal: p/q > 1
    _set_z(b, z)
    got, ref = _check(oracle_mod, b, "accept", with_attention=False)
    assert np.all(ref["accepted_len"] >= 1)


def test_all_plain_decode_batch(oracle_mod):
    B = 24
    b = wl.make_batch_from_lengths("decode_only", draft_lens=np.zeros(B, np.int32),
                                   context_lens=np.random.default_rng(34).integers(1, 3000, B), Hq=32, Hkv=8,
                                   D=128, V=128256, dtype="bf16", sigma=1.0, key=(134, 0))
    assert b.total_draft == 0
    got, ref = _check(oracle_mod, b, "step")
    assert np.all(got["accepted_len"] == 0)


def test_one_request_at_128k_context_shuffled_pages(oracle_mod):
    b = wl.make_batch_from_lengths("b1_128k", draft_lens=[7], context_lens=[131072], Hq=32, Hkv=8, D=128,
                                   V=128256, dtype="bf16", sigma=float(wl.sigma_for_alpha(0.7)), key=(135, 0),
                                   shuffle_blocks=True, extra_blocks=64)
    _check(oracle_mod, b, "step")


def test_fp32_logits_large_vocabulary(oracle_mod):
    b = wl.make_small_batch(36, B=6, Hq=8, Hkv=2, D=128, V=152064, dtype="f32", k_range=(0, 8), ctx_range=(0, 300))
    _check(oracle_mod, b, "step")


def test_residual_without_mass_draws_from_p(oracle_mod):
    b = wl.make_small_batch(37, B=6, Hq=8, Hkv=2, D=128, V=8000, dtype="bf16", k_range=(1, 5), ctx_range=(0, 200))
    qs, ds = b.q_row_start(), b.draft_start()
    b.draft_probs = b.draft_probs.copy()
    b.accept_uniforms = b.accept_uniforms.copy()
    for r in range(b.B):
        p = oracle_mod.row_softmax(b.logits[qs[r]], b.dtype)
        b.draft_probs[ds[r]] = (2.0 * p).astype(np.float32)  # q = 2p: a = 1/2, no residual mass
        b.accept_uniforms[ds[r]] = np.float32(0.9)
    got, ref = _check(oracle_mod, b, "accept", with_attention=False)
    assert np.all(ref["accepted_len"] == 0)


def test_batch_past_two_draw_waves(oracle_mod):
    """B = 700 requests (more than twice the 304 acceptance CTAs): statistics items are whole rows
    and the draw keeps two slices per row; every request matches the oracle."""
    b = wl.make_small_batch(31, B=700, Hq=8, Hkv=2, D=128, V=6000, dtype="bf16", k_range=(0, 4), ctx_range=(0, 64))
    got, ref = _check(oracle_mod, b)
    assert np.any(ref["accepted_len"] < b.draft_lens) and np.any(ref["accepted_len"] == b.draft_lens)
