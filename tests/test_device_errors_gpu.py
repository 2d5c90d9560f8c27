"""GPU: data errors found on the device (the C ABI's status word).

One bad input per call -- a block id outside the pool, a draft token outside [0, V), a negative
draft probability at a token the walk decides on, a logit row with no finite value, a context
longer than the request's block table.  Each must be reported in the workspace status word with
its code and the request's id, without a trap, and every other request of the batch must still
match the oracle.
"""
import numpy as np
import pytest
import torch

from paper_2601_11652_gb300 import workload as wl
from tests.gpu_util import ATTN_TOL, attn_max_err, subset_rows

pytestmark = pytest.mark.gpu

BAD_LENGTH, BAD_BLOCK, BAD_TOKEN, BAD_PROB = 1, 2, 3, 4   # WISP_DEV_* (include/wisp_verify.h)
ORACLE_STATUS = {BAD_TOKEN: 4, BAD_PROB: 5}               # the oracle's per-request codes


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.fail("GPU tests need a CUDA device")
    from paper_2601_11652_gb300 import build
    build.build()


def _batch(dtype):
    # every request drafts at least one token, so its first decision reads q(y_1) and row 0
    return wl.make_small_batch(21, B=6, Hq=8, Hkv=2, D=128, V=5000, dtype=dtype, k_range=(1, 6),
                               ctx_range=(20, 400), shuffle_blocks=False)


def _corrupt(b, kind, r):
    qs, ds = b.q_row_start(), b.draft_start()
    if kind == "block":
        b.block_tables = b.block_tables.copy()
        b.block_tables[r, 0] = b.num_blocks + 5
        return BAD_BLOCK
    if kind == "token":
        b.draft_tokens = b.draft_tokens.copy()
        b.draft_tokens[ds[r]] = b.V
        return BAD_TOKEN
    if kind == "prob":
        b.draft_probs = b.draft_probs.copy()
        b.draft_probs[ds[r], b.draft_tokens[ds[r]]] = -0.5
        return BAD_PROB
    if kind == "row":
        b.logits = b.logits.copy()
        ninf = np.float32(-np.inf)
        b.logits[qs[r]] = wl.f32_to_bf16_bits(np.full(b.V, ninf, np.float32)) if b.dtype == "bf16" else ninf
        return BAD_PROB
    if kind == "length":
        b.context_lens = b.context_lens.copy()
        b.context_lens[r] = b.block_tables.shape[1] * b.block_size  # c + k + 1 exceeds the table
        return BAD_LENGTH
    raise ValueError(kind)


@pytest.mark.parametrize("dtype,kind", [("bf16", "block"), ("f32", "block"), ("bf16", "token"),
                                        ("bf16", "prob"), ("bf16", "row"), ("f32", "row"),
                                        ("bf16", "length")])
def test_bad_input_is_reported_and_the_rest_is_exact(oracle_mod, dtype, kind):
    from paper_2601_11652_gb300.device_batch import DeviceBatch
    clean = _batch(dtype)
    ref_attn = oracle_mod.attention(clean)
    ref_acc = oracle_mod.accept(clean)
    r = 2
    b = _batch(dtype)
    code = _corrupt(b, kind, r)
    db = DeviceBatch.from_host(b)
    db.step()
    torch.cuda.synchronize()
    got_code, got_rid = db.device_status()
    assert (got_code, got_rid) == (code, int(b.request_ids[r]))
    got = db.results()
    others = [i for i in range(b.B) if i != r]
    rows = subset_rows(b, others)
    assert attn_max_err(got["out"][rows], ref_attn[rows]) <= ATTN_TOL[dtype]
    for i in others:
        assert got["accepted_len"][i] == ref_acc["accepted_len"][i], i
        assert got["next_token"][i] == ref_acc["next_token"][i], i
    if kind in ("token", "prob", "row"):
        # the acceptance pass refuses the request (outputs -1)
        assert got["accepted_len"][r] == -1 and got["next_token"][r] == -1
        # and the oracle flags it with the same reading
        assert oracle_mod.accept(b, check=False)["status"][r] == ORACLE_STATUS[code]


def test_too_many_query_rows_per_kv_head_is_reported(oracle_mod):
    """g (k + 1) = 4 x 33 = 132 query rows of one KV head, above the library's 128: the planner flags
    the request WISP_DEV_UNSUPPORTED and the step runs every other request exactly."""
    from paper_2601_11652_gb300.device_batch import DeviceBatch
    k = np.array([3, 2, 32, 4, 1], np.int32)
    c = np.array([100, 50, 80, 300, 10], np.int32)
    b = wl.make_batch_from_lengths("rows132", draft_lens=k, context_lens=c, Hq=8, Hkv=2, D=128, V=3000,
                                   dtype="bf16", sigma=float(wl.sigma_for_alpha(0.7)), key=(140, 0))
    ref_attn = oracle_mod.attention(b)
    ref_acc = oracle_mod.accept(b)
    db = DeviceBatch.from_host(b)
    db.step()
    torch.cuda.synchronize()
    assert db.device_status() == (5, int(b.request_ids[2]))  # WISP_DEV_UNSUPPORTED
    got = db.results()
    others = [0, 1, 3, 4]
    rows = subset_rows(b, others)
    assert attn_max_err(got["out"][rows], ref_attn[rows]) <= ATTN_TOL["bf16"]
    for i in others:
        assert got["accepted_len"][i] == ref_acc["accepted_len"][i], i
        assert got["next_token"][i] == ref_acc["next_token"][i], i


def test_empty_batch_is_a_no_op():
    """B = 0: every entry point accepts the empty batch (attention pointers may be NULL), enqueues
    only the planner, reports no error and writes no output."""
    from paper_2601_11652_gb300 import binding as wb
    dev = "cuda"
    lens = torch.zeros(1, dtype=torch.int32, device=dev)
    logits = torch.zeros((1, 1000), dtype=torch.bfloat16, device=dev)
    su = torch.zeros(1, dtype=torch.float32, device=dev)
    out_L = torch.full((1,), -7, dtype=torch.int32, device=dev)
    out_t = torch.full((1,), -7, dtype=torch.int32, device=dev)
    a = wb.wisp_attn_args()
    a.B, a.Hq, a.Hkv, a.D, a.block_size, a.qkv_dtype = 0, 8, 2, 128, 16, wb.WISP_BF16
    c = wb.wisp_accept_args()
    c.B, c.V, c.total_q_rows, c.total_draft, c.logits_dtype = 0, 1000, 0, 0, wb.WISP_BF16
    c.draft_lens, c.target_logits, c.sample_uniforms = lens.data_ptr(), logits.data_ptr(), su.data_ptr()
    c.accepted_len, c.next_token = out_L.data_ptr(), out_t.data_ptr()
    ws = wb.alloc_workspace(wb.wisp_verify_workspace_size(a, c), dev)
    wb.wisp_verify_step(a, c, ws)
    wb.wisp_verify_attention(a, ws)
    wb.wisp_verify_accept(c, ws)
    torch.cuda.synchronize()
    # no error: code 0 and request id -1, as include/wisp_verify.h documents
    assert wb.wisp_verify_get_device_status(ws) == (0, -1)
    assert out_L.item() == -7 and out_t.item() == -7
