"""GPU parity: the sm_103a library (through its C ABI) against the fp64 oracle.

Small batches are compared element by element (attention within ATTN_TOL,
accepted_len / next_token bit-exact except logged near-threshold requests).
The full-size workloads run in the launch configuration the benchmark times;
their acceptance and attention outputs are compared for every request (the oracle's
attention in bounded groups of requests).
"""
import numpy as np
import pytest
import torch

from paper_2601_11652_gb300 import workload as wl
from tests.gpu_util import ATTN_TOL, attn_max_err, compare_accept, request_groups, subset_rows

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


SMALL_CASES = [
    # seed, dtype, Hq, Hkv, D, V, k_range, ctx_range
    (0, "bf16", 8, 2, 128, 4096, (0, 9), (0, 700)),
    (1, "bf16", 32, 8, 128, 32000, (1, 8), (100, 1500)),
    (2, "bf16", 28, 4, 128, 50000, (0, 12), (0, 3000)),
    (3, "f32", 4, 4, 64, 1000, (0, 6), (0, 300)),
    (4, "bf16", 16, 16, 64, 777, (0, 5), (0, 200)),
    (5, "f32", 8, 2, 128, 3001, (0, 4), (0, 400)),
    # 8 query heads per KV head and k up to 15: up to 128 rows per (request, head), cut into two
    # row groups of at most 64 by the planner, with split chunks
    (6, "bf16", 32, 4, 128, 2000, (8, 15), (0, 2500)),
    # two row groups at head dim 64 (16 query heads per KV head: 96-128 rows per (request, head))
    (9, "bf16", 32, 2, 64, 2000, (5, 7), (0, 1500)),
    # head dim 64 with 33-64 rows per (request, head): the second group of softmax warps at D = 64
    (7, "bf16", 16, 2, 64, 3000, (4, 7), (0, 2000)),
    # fp32 inputs (CUDA-core kernel) with up to 128 rows per (request, head)
    (8, "f32", 32, 2, 128, 1500, (6, 7), (0, 500)),
]


@pytest.mark.parametrize("case", SMALL_CASES, ids=[f"small{c[0]}-{c[1]}-g{c[2]//c[3]}-d{c[4]}-V{c[5]}" for c in SMALL_CASES])
def test_small_batches_elementwise(oracle_mod, case):
    seed, dtype, Hq, Hkv, D, V, kr, cr = case
    b = wl.make_small_batch(seed, B=7, Hq=Hq, Hkv=Hkv, D=D, V=V, dtype=dtype, k_range=kr, ctx_range=cr)
    got = _run(b)
    ref_attn = oracle_mod.attention(b)
    err = attn_max_err(got["out"], ref_attn)
    assert err <= ATTN_TOL[dtype], f"attention max abs error {err}"
    n, logged = compare_accept(b, got["accepted_len"], got["next_token"], oracle_mod.accept(b))
    assert n >= b.B - 1


def test_tiny_config_elementwise(oracle_mod):
    b = wl.make_batch("tiny_f32")
    got = _run(b)
    assert attn_max_err(got["out"], oracle_mod.attention(b)) <= ATTN_TOL["f32"]
    n, logged = compare_accept(b, got["accepted_len"], got["next_token"], oracle_mod.accept(b))
    assert n == b.B


def test_entry_points_agree_with_step(oracle_mod):
    b = wl.make_small_batch(7, B=5, V=5000)
    s = _run(b, "step")
    a = _run(b, "attention")
    c = _run(b, "accept")
    np.testing.assert_array_equal(s["out"], a["out"])
    np.testing.assert_array_equal(s["accepted_len"], c["accepted_len"])
    np.testing.assert_array_equal(s["next_token"], c["next_token"])


def test_deterministic_reruns():
    b = wl.make_small_batch(8, B=6, V=9000)
    from paper_2601_11652_gb300.device_batch import DeviceBatch
    db = DeviceBatch.from_host(b)
    db.step()
    first = db.results()
    for _ in range(3):
        db.step()
        again = db.results()
        for key in first:
            np.testing.assert_array_equal(first[key], again[key])


@pytest.mark.parametrize("name", ["llama3_8b_b32", "fanin_b256", "longctx_b16", "hetero_b512"])
def test_full_size_workloads(oracle_mod, name):
    b = wl.make_batch(name)
    got = _run(b)
    # acceptance: every request
    n, logged = compare_accept(b, got["accepted_len"], got["next_token"], oracle_mod.accept(b))
    assert n >= b.B - max(1, b.B // 100)
    # attention: every request, the oracle called on groups of requests so that each call stays
    # bounded (a few seconds of fp64 work on the host cores)
    assert np.all(np.isfinite(got["out"]))
    for reqs in request_groups(b, max_row_keys=2e8):
        ref = oracle_mod.attention(b.subset(reqs))
        err = attn_max_err(got["out"][subset_rows(b, reqs)], ref)
        assert err <= ATTN_TOL[b.dtype], f"attention max abs error {err} in requests {reqs[0]}..{reqs[-1]}"
