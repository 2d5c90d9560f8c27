"""The seeded input generator: determinism, layout, bf16 rounding and the acceptance recipe."""
import numpy as np
import pytest
import torch
from scipy.special import softmax

from paper_2601_11652_gb300 import workload as wl


def test_bf16_rounding_matches_torch():
    x = np.random.default_rng(0).standard_normal(100_000).astype(np.float32) * 3
    x[:4] = [0.0, -0.0, 1e-30, 65504.0]
    ours = wl.f32_to_bf16_bits(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(ours, ref)
    np.testing.assert_array_equal(wl.bf16_bits_to_f32(ours), torch.from_numpy(x).to(torch.bfloat16).float().numpy())


def test_deterministic_and_shaped():
    a, b = wl.make_batch("tiny_f32"), wl.make_batch("tiny_f32")
    for f in ["q", "k_cache", "v_cache", "logits", "draft_probs", "draft_tokens", "accept_uniforms", "sample_uniforms"]:
        np.testing.assert_array_equal(getattr(a, f), getattr(b, f))
    assert a.q.shape == (14, 4, 64) and a.logits.shape == (14, 1000) and a.draft_probs.shape == (10, 1000)
    np.testing.assert_array_equal(a.draft_lens, [1, 2, 3, 4])
    np.testing.assert_array_equal(a.context_lens, [16, 40, 77, 128])
    c = wl.make_batch("tiny_f32", variant=1)
    assert not np.array_equal(a.q, c.q)


def test_block_tables_cover_each_request_once():
    b = wl.make_small_batch(2, B=6, shuffle_blocks=True)
    used = []
    for r in range(b.B):
        n = int(b.context_lens[r] + b.draft_lens[r] + 1)
        nb = (n + 15) // 16
        assert np.all(b.block_tables[r, :nb] >= 0) and np.all(b.block_tables[r, nb:] == -1)
        used += list(b.block_tables[r, :nb])
    assert len(set(used)) == len(used) and max(used) < b.num_blocks


def test_draft_tokens_drawn_from_stored_q():
    b = wl.make_small_batch(1, B=8, V=64, dtype="f32")
    assert np.all(b.draft_probs[np.arange(b.total_draft), b.draft_tokens] > 0)
    np.testing.assert_allclose(b.draft_probs.sum(axis=1), 1.0, atol=1e-5)


@pytest.mark.parametrize("alpha", [0.4, 0.7, 0.9])
def test_sigma_recipe_gives_target_acceptance(alpha):
    # realized sum_v min(p, q) on 128k-entry rows of N(0, 2) logits, bf16-rounded
    rng = np.random.default_rng(3)
    V = 128256
    z = wl.bf16_bits_to_f32(wl.f32_to_bf16_bits(2 * rng.standard_normal((4, V)).astype(np.float32))).astype(np.float64)
    s = float(wl.sigma_for_alpha(alpha))
    p = softmax(z, axis=1)
    q = softmax(z + s * rng.standard_normal(z.shape), axis=1)
    assert abs(np.minimum(p, q).sum(axis=1).mean() - alpha) < 0.02
    assert abs(float(wl.alpha_for_sigma(s)) - alpha) < 1e-12


def test_named_workload_lengths():
    # only the length draws (no tensors) of the large workloads
    for name in ["llama3_8b_b32", "fanin_b256", "longctx_b16", "hetero_b512"]:
        spec = wl.SPECS[name]
        rng = wl._rng(spec.config_id, 0, 0)
        k = wl._draw_lengths(spec, rng, spec.k_rule, spec.B)
        c = wl._draw_lengths(spec, rng, spec.ctx_rule, spec.B)
        assert len(k) == spec.B and len(c) == spec.B
        if spec.k_rule[0] == "uniform":
            assert k.min() >= spec.k_rule[1] and k.max() <= spec.k_rule[2]
        assert c.min() >= 1
