"""The lossless law on the GPU path (Eq. 1-3): with draft tokens drawn from q, the tokens the
verification emits follow the target distribution p.

V = 8, k = 3, 10^6 seeded requests through wisp_verify_accept (fp32 and bf16 logits; bf16 takes
the acceptance kernel's table of exponentials): the first emitted token (y_1 if accepted, else
the extra token) against p_0 and the second (given L >= 1) against p_1 by chi-square, E[L]
against its closed form, and the first requests element by element against the oracle.
"""
import numpy as np
import pytest
import torch
from scipy.special import softmax
from scipy.stats import chisquare

from paper_2601_11652_gb300 import workload as wl
from tests.gpu_util import compare_accept

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.fail("GPU tests need a CUDA device")
    from paper_2601_11652_gb300 import build
    build.build()


class _Batch:
    """Acceptance-only batch in the layout the oracle reads."""

    def __init__(self, logits, draft_lens, draft_tokens, draft_probs, accept_u, sample_u, dtype):
        self.logits = logits
        self.V = logits.shape[1]
        self.draft_lens = draft_lens
        self.draft_tokens = draft_tokens
        self.draft_probs = draft_probs
        self.accept_uniforms = accept_u
        self.sample_uniforms = sample_u
        self.dtype = dtype
        self.B = len(draft_lens)


def _run_gpu(b: _Batch):
    from paper_2601_11652_gb300 import binding as wb
    dev = "cuda"
    if b.dtype == "bf16":
        logits = torch.from_numpy(b.logits.view(np.int16)).to(dev).view(torch.bfloat16)
    else:
        logits = torch.from_numpy(b.logits).to(dev)
    t = dict(draft_lens=torch.from_numpy(b.draft_lens).to(dev), target_logits=logits,
             draft_tokens=torch.from_numpy(b.draft_tokens).to(dev), draft_probs=torch.from_numpy(b.draft_probs).to(dev),
             accept_uniforms=torch.from_numpy(b.accept_uniforms).to(dev),
             sample_uniforms=torch.from_numpy(b.sample_uniforms).to(dev),
             accepted_len=torch.full((b.B,), -7, dtype=torch.int32, device=dev),
             next_token=torch.full((b.B,), -7, dtype=torch.int32, device=dev))
    args = wb.make_accept_args(**t)
    ws = wb.alloc_workspace(wb.wisp_verify_workspace_size(None, args))
    wb.wisp_verify_accept(args, ws)
    torch.cuda.synchronize()
    code, rid = wb.wisp_verify_get_device_status(ws)
    assert code == 0, (code, rid)
    return t["accepted_len"].cpu().numpy(), t["next_token"].cpu().numpy()


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_lossless_law_on_gpu(oracle_mod, dtype):
    rng = np.random.default_rng(20260112 + (dtype == "bf16"))
    V, k, N = 8, 3, 1_000_000
    z = (1.5 * rng.standard_normal((k + 1, V))).astype(np.float32)
    if dtype == "bf16":
        zb = wl.f32_to_bf16_bits(z)
        zval = wl.bf16_bits_to_f32(zb)
    else:
        zb, zval = z, z
    qrows = softmax(zval[:k].astype(np.float64) + 0.8 * rng.standard_normal((k, V)), axis=1).astype(np.float32)
    p = softmax(zval.astype(np.float64), axis=1)
    assert (p * N).min() > 50  # chi-square needs enough expected counts per cell
    qn = qrows.astype(np.float64) / qrows.astype(np.float64).sum(axis=1, keepdims=True)
    toks = np.stack([rng.choice(V, size=N, p=qn[j]) for j in range(k)], axis=1).astype(np.int32)
    b = _Batch(np.ascontiguousarray(np.tile(zb, (N, 1))), np.full(N, k, np.int32), np.ascontiguousarray(toks.reshape(-1)),
               np.ascontiguousarray(np.tile(qrows, (N, 1))), rng.random(N * k).astype(np.float32),
               rng.random(N).astype(np.float32), dtype)
    L, t = _run_gpu(b)
    assert L.min() >= 0 and L.max() <= k and t.min() >= 0 and t.max() < V
    first = np.where(L >= 1, toks[:, 0], t)
    assert chisquare(np.bincount(first, minlength=V), p[0] * N).pvalue > 0.01
    sel = L >= 1
    second = np.where(L[sel] >= 2, toks[sel, 1], t[sel])
    assert chisquare(np.bincount(second, minlength=V), p[1] * sel.sum()).pvalue > 0.01
    alpha = np.minimum(p[:k], qrows.astype(np.float64)).sum(axis=1)
    expect = sum(np.prod(alpha[:j]) for j in range(1, k + 1))
    assert abs(L.mean() - expect) < 4 * L.std() / np.sqrt(N)
    # the first requests, element by element against the oracle
    n = 20000
    sub = _Batch(np.ascontiguousarray(b.logits[: n * (k + 1)]), b.draft_lens[:n], b.draft_tokens[: n * k],
                 b.draft_probs[: n * k], b.accept_uniforms[: n * k], b.sample_uniforms[:n], dtype)
    compare_accept(sub, L[:n], t[:n], oracle_mod.accept(sub))
