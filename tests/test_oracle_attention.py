"""Pins of the oracle's attention (Sec. 4.4-4.5: k+1 new queries over L_total keys).

Nothing here re-types the oracle's formula: the oracle is compared with a
library attention routine (torch scaled_dot_product_attention in float64),
with closed forms, with a hand-worked example and with invariances.
"""
import json
import os

import numpy as np
import pytest
import torch

from paper_2601_11652_gb300 import workload as wl

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _values(a, dtype):
    return wl.bf16_bits_to_f32(a).astype(np.float64) if dtype == "bf16" else np.asarray(a, np.float64)


def _library_attention(b):
    """Per request: gather contiguous K/V via the block table, then torch SDPA (float64, CPU)."""
    q = _values(b.q, b.dtype)
    kc = _values(b.k_cache, b.dtype)
    vc = _values(b.v_cache, b.dtype)
    g = b.Hq // b.Hkv
    out = np.zeros_like(q)
    qs = b.q_row_start()
    for r in range(b.B):
        c, k = int(b.context_lens[r]), int(b.draft_lens[r])
        n = c + k + 1
        blocks = b.block_tables[r, : (n + b.block_size - 1) // b.block_size]
        K = kc[blocks].transpose(1, 0, 2, 3).reshape(b.Hkv, -1, b.D)[:, :n]   # [Hkv, n, D]
        V = vc[blocks].transpose(1, 0, 2, 3).reshape(b.Hkv, -1, b.D)[:, :n]
        Q = q[qs[r]: qs[r + 1]].transpose(1, 0, 2)                           # [Hq, k+1, D]
        mask = np.arange(n)[None, :] <= (c + np.arange(k + 1))[:, None]     # query j sees keys <= c+j
        o = torch.nn.functional.scaled_dot_product_attention(
            torch.from_numpy(Q), torch.from_numpy(np.repeat(K, g, axis=0)),
            torch.from_numpy(np.repeat(V, g, axis=0)), attn_mask=torch.from_numpy(mask))
        out[qs[r]: qs[r + 1]] = o.numpy().transpose(1, 0, 2)
    return out


@pytest.mark.parametrize("seed,dtype,Hq,Hkv,D", [(0, "f32", 4, 4, 64), (1, "bf16", 8, 2, 128),
                                                  (2, "bf16", 28, 4, 128), (3, "f32", 6, 3, 16)])
def test_oracle_attention_vs_library(oracle_mod, seed, dtype, Hq, Hkv, D):
    b = wl.make_small_batch(seed, B=4, Hq=Hq, Hkv=Hkv, D=D, V=64, dtype=dtype,
                            k_range=(0, 6), ctx_range=(0, 90))
    got = oracle_mod.attention(b)
    ref = _library_attention(b)
    assert np.max(np.abs(got - ref)) < 1e-12


def test_oracle_attention_tiny_config_vs_library(oracle_mod):
    b = wl.make_batch("tiny_f32")
    np.testing.assert_allclose(oracle_mod.attention(b), _library_attention(b), rtol=0, atol=1e-12)


def _one_request(ctx, k, D=8, H=2, Hkv=1, seed=0, dtype="f32"):
    return wl.make_batch_from_lengths("t", draft_lens=[k], context_lens=[ctx], Hq=H, Hkv=Hkv, D=D, V=8,
                                      dtype=dtype, sigma=0.5, key=(900 + seed, 0))


def test_single_key_returns_its_value(oracle_mod):
    # ctx = 0, k = 0: the only visible key is the token itself, softmax weight 1 -> O = V_self
    b = _one_request(0, 0)
    out = oracle_mod.attention(b)
    blk = b.block_tables[0, 0]
    for h in range(b.Hq):
        np.testing.assert_array_equal(out[0, h], b.v_cache[blk, h // (b.Hq // b.Hkv), 0].astype(np.float64))


def test_identical_keys_average_visible_values(oracle_mod):
    # all keys equal -> uniform weights -> O_j = mean of the c+j+1 visible values
    b = _one_request(37, 5, D=16, H=3, Hkv=3, seed=1)
    b.k_cache[:] = b.k_cache[0, 0, 0]
    out = oracle_mod.attention(b)
    n = 37 + 5 + 1
    for h in range(3):
        vals = b.v_cache[b.block_tables[0, : (n + 15) // 16]][:, h].reshape(-1, 16)[:n].astype(np.float64)
        for j in range(6):
            np.testing.assert_allclose(out[j, h], vals[: 37 + j + 1].mean(axis=0), rtol=0, atol=1e-13)


def test_future_keys_are_invisible(oracle_mod):
    # changing K/V at positions > c+j must not change query j (causal within the draft)
    b = _one_request(20, 6, D=8, H=2, Hkv=2, seed=2)
    base = oracle_mod.attention(b)
    c = 20
    pos = c + 4  # visible only to queries j >= 4
    blk, slot = b.block_tables[0, pos // 16], pos % 16
    b.k_cache[blk, :, slot] += 3.0
    b.v_cache[blk, :, slot] -= 5.0
    after = oracle_mod.attention(b)
    np.testing.assert_array_equal(after[:4], base[:4])
    assert np.all(np.abs(after[4:] - base[4:]).max(axis=(1, 2)) > 0)


def test_gqa_equals_repeated_kv_heads(oracle_mod):
    # Hq = g * Hkv reads KV head h // g: identical to MHA with each KV head repeated g times
    b = wl.make_small_batch(5, B=3, Hq=8, Hkv=2, D=32, V=16, dtype="f32", k_range=(0, 4), ctx_range=(0, 50))
    gqa = oracle_mod.attention(b)
    mha = wl.VerifyBatch(**{**b.__dict__, "Hkv": 8, "k_cache": np.repeat(b.k_cache, 4, axis=1),
                            "v_cache": np.repeat(b.v_cache, 4, axis=1)})
    np.testing.assert_array_equal(gqa, oracle_mod.attention(mha))


def test_block_permutation_invariance(oracle_mod):
    b = wl.make_small_batch(6, B=3, Hq=4, Hkv=2, D=16, V=16, dtype="bf16", shuffle_blocks=False)
    base = oracle_mod.attention(b)
    perm = np.random.default_rng(0).permutation(b.num_blocks)
    inv = np.argsort(perm)
    bt = np.where(b.block_tables >= 0, inv[np.maximum(b.block_tables, 0)], -1).astype(np.int32)
    moved = wl.VerifyBatch(**{**b.__dict__, "block_tables": bt, "k_cache": b.k_cache[perm], "v_cache": b.v_cache[perm]})
    np.testing.assert_array_equal(oracle_mod.attention(moved), base)


def test_hand_worked_example(oracle_mod):
    """tests/golden/attention_hand.json: two keys whose scores differ by ln 3 -> weights 1/4, 3/4."""
    with open(os.path.join(GOLDEN, "attention_hand.json")) as f:
        g = json.load(f)
    D = g["D"]
    b = _one_request(g["context_len"], 0, D=D, H=1, Hkv=1)
    b.q[0, 0] = np.array(g["q"], np.float32)
    blk = b.block_tables[0, 0]
    b.k_cache[blk, 0, :2] = np.array(g["keys"], np.float32)
    b.v_cache[blk, 0, :2] = np.array(g["values"], np.float32)
    out = oracle_mod.attention(b)
    np.testing.assert_allclose(out[0, 0], g["expected_output"], rtol=0, atol=g["atol"])


def test_rejects_bad_block_id(oracle_mod):
    b = _one_request(40, 2)
    b.block_tables[0, 1] = b.num_blocks + 5
    with pytest.raises(ValueError):
        oracle_mod.attention(b)
