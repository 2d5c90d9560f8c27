"""The allocation-free acceptance entry point against the workspace one (GPU).

wisp_verify_accept_noalloc runs the acceptance pass with its workspace carved from a fixed
array in the library's device image.  Two calls in a row must give the same accepted lengths
and extra tokens as wisp_verify_accept on the same inputs (same kernels, deterministic
results), and those agree with the oracle.  The file name sorts last, so that in a full run
the entry point is also exercised after every other GPU test has used the library.
"""
import numpy as np
import pytest
import torch

from paper_2601_11652_gb300 import workload as wl
from tests.gpu_util import compare_accept

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.fail("GPU tests need a CUDA device")
    from paper_2601_11652_gb300 import build
    build.build()


def _batches():
    yield "small-bf16", wl.make_small_batch(11, B=7, Hq=8, Hkv=2, D=128, V=32000, dtype="bf16",
                                            k_range=(0, 9), ctx_range=(0, 300))
    yield "small-f32", wl.make_small_batch(12, B=5, Hq=4, Hkv=4, D=64, V=1000, dtype="f32",
                                           k_range=(0, 6), ctx_range=(0, 100))
    yield "llama3_8b_b32", wl.make_batch("llama3_8b_b32")


@pytest.mark.parametrize("name", ["small-bf16", "small-f32", "llama3_8b_b32"])
def test_noalloc_matches_workspace_entry_point(oracle_mod, name):
    from paper_2601_11652_gb300 import binding as wb
    from paper_2601_11652_gb300.device_batch import DeviceBatch
    batch = dict(_batches())[name]
    db = DeviceBatch.from_host(batch)
    db.accept()
    torch.cuda.synchronize()
    assert db.device_status()[0] == 0
    ref_L = db.t["accepted_len"].cpu().numpy().copy()
    ref_tok = db.t["next_token"].cpu().numpy().copy()
    if name.startswith("small"):
        compare_accept(batch, ref_L, ref_tok, oracle_mod.accept(batch))
    for call in range(2):
        db.t["accepted_len"].fill_(-7)
        db.t["next_token"].fill_(-7)
        wb.wisp_verify_accept_noalloc(db.accept_args)
        torch.cuda.synchronize()
        L = db.t["accepted_len"].cpu().numpy()
        tok = db.t["next_token"].cpu().numpy()
        np.testing.assert_array_equal(L, ref_L, err_msg=f"accepted_len, call {call}")
        np.testing.assert_array_equal(tok, ref_tok, err_msg=f"next_token, call {call}")


def test_noalloc_bad_draft_token_refuses_only_that_request():
    """A draft token outside [0, V) in one request: this entry point does not expose its status
    word, so the documented error behaviour is visible only in the outputs -- that request gets
    -1 for accepted_len and next_token, every other request matches wisp_verify_accept."""
    from paper_2601_11652_gb300 import binding as wb
    from paper_2601_11652_gb300.device_batch import DeviceBatch
    b = wl.make_small_batch(11, B=7, Hq=8, Hkv=2, D=128, V=32000, dtype="bf16", k_range=(1, 9),
                            ctx_range=(0, 300))
    r = 3
    b.draft_tokens = b.draft_tokens.copy()
    b.draft_tokens[b.draft_start()[r] + b.draft_lens[r] - 1] = b.V + 11  # the request's last draft token
    db = DeviceBatch.from_host(b)
    db.accept()
    torch.cuda.synchronize()
    assert db.device_status() == (3, int(b.request_ids[r]))  # WISP_DEV_BAD_TOKEN
    ref_L = db.t["accepted_len"].cpu().numpy().copy()
    ref_tok = db.t["next_token"].cpu().numpy().copy()
    assert ref_L[r] == -1 and ref_tok[r] == -1
    for call in range(2):
        db.t["accepted_len"].fill_(-7)
        db.t["next_token"].fill_(-7)
        wb.wisp_verify_accept_noalloc(db.accept_args)
        torch.cuda.synchronize()
        L = db.t["accepted_len"].cpu().numpy()
        tok = db.t["next_token"].cpu().numpy()
        assert L[r] == -1 and tok[r] == -1, f"call {call}"
        np.testing.assert_array_equal(L, ref_L, err_msg=f"accepted_len, call {call}")
        np.testing.assert_array_equal(tok, ref_tok, err_msg=f"next_token, call {call}")
