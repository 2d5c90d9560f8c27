"""GPU: verification steps on several caller streams, and steps fed from host memory.

  * two batches, each with its own workspace, stepped alternately on two torch streams (each
    caller stream gets its own side stream inside wisp_verify_step): both match the oracle;
  * the staged end-to-end path (one pinned staging buffer, one copy per step overlapped with the
    previous step, two device buffers in turn) returns the resident batch's results on every step.
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


def test_two_steps_on_two_streams(oracle_mod):
    from paper_2601_11652_gb300.device_batch import DeviceBatch
    b1 = wl.make_small_batch(41, B=12, Hq=8, Hkv=2, D=128, V=30000, dtype="bf16", k_range=(0, 7), ctx_range=(0, 900))
    b2 = wl.make_small_batch(42, B=20, Hq=8, Hkv=2, D=128, V=30000, dtype="bf16", k_range=(1, 8), ctx_range=(0, 500))
    d1, d2 = DeviceBatch.from_host(b1), DeviceBatch.from_host(b2)
    s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()
    torch.cuda.synchronize()
    for _ in range(4):  # interleaved on the host: each stream's steps only depend on that stream
        d1.step(s1)
        d2.step(s2)
    torch.cuda.synchronize()
    for b, d in ((b1, d1), (b2, d2)):
        code, rid = d.device_status()
        assert code == 0, f"device status {code} (request {rid})"
        got, ref = d.results(), oracle_mod.accept(b)
        n, _ = compare_accept(b, got["accepted_len"], got["next_token"], ref)
        assert n >= b.B - 1
        assert attn_max_err(got["out"], oracle_mod.attention(b)) <= ATTN_TOL["bf16"]


def test_staged_steps_match_resident_batch():
    from paper_2601_11652_gb300.device_batch import DeviceBatch, StagedSteps
    b = wl.make_small_batch(43, B=16, Hq=8, Hkv=2, D=128, V=20000, dtype="bf16", k_range=(0, 6), ctx_range=(0, 700))
    db = DeviceBatch.from_host(b)
    db.step()
    torch.cuda.synchronize()
    want = db.results()
    st = StagedSteps(b, pool=(db.t["k_cache"], db.t["v_cache"]))
    for _ in range(5):
        out = st.enqueue()
        torch.cuda.current_stream().synchronize()
        o = out.numpy()
        assert np.array_equal(o[0], want["accepted_len"]) and np.array_equal(o[1], want["next_token"])
    assert st.h2d_bytes >= b.logits.nbytes + b.draft_probs.nbytes
