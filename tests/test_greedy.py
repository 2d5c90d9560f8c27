"""Greedy (temperature 0) acceptance: the oracle's rule pinned on hand cases (CPU), and the GPU entry
point wisp_verify_accept_greedy against it on every request (GPU)."""
import numpy as np
import pytest
import torch

from paper_2601_11652_gb300 import workload as wl


class _Batch:
    def __init__(self, logits, draft_lens, draft_tokens, dtype="f32"):
        self.logits = np.ascontiguousarray(logits)
        self.V = self.logits.shape[1]
        self.draft_lens = np.asarray(draft_lens, np.int32)
        self.draft_tokens = np.asarray(draft_tokens, np.int32)
        self.dtype = dtype
        self.B = len(self.draft_lens)


def test_hand_cases(oracle_mod):
    z = np.array([[0.0, 3.0, 1.0, 3.0],    # argmax 1 (tie with 3: lowest index)
                  [5.0, 0.0, 0.0, 0.0],    # argmax 0
                  [0.0, 0.0, 0.0, 2.0],    # bonus row: argmax 3
                  [1.0, 2.0, 0.0, 0.0],    # request 2, row 0: argmax 1
                  [9.0, 9.0, 9.0, 9.0]],   # request 2, row 1 (all tied): argmax 0
                 dtype=np.float32)
    b = _Batch(z, [2, 1], [1, 0, 3])
    out = oracle_mod.accept_greedy(b)
    # request 0: y1 = 1 = argmax row 0, y2 = 0 = argmax row 1 -> L = 2, bonus argmax row 2 = 3
    # request 1: y1 = 3 != argmax row 3 (= 1) -> L = 0, token 1
    assert out["accepted_len"].tolist() == [2, 0] and out["next_token"].tolist() == [3, 1]
    b = _Batch(z[:1], [0], [])
    assert oracle_mod.accept_greedy(b)["next_token"].tolist() == [1]
    bad = _Batch(np.full((1, 4), -np.inf, np.float32), [0], [])
    assert oracle_mod.accept_greedy(bad)["status"].tolist() == [5]


def test_greedy_matches_rule_with_draft_equal_argmax(oracle_mod):
    # drafts that always take the argmax are always accepted
    rng = np.random.default_rng(3)
    z = rng.standard_normal((3 * 5, 50)).astype(np.float32)
    toks = [int(np.argmax(z[r * 5 + i])) for r in range(3) for i in range(4)]
    out = oracle_mod.accept_greedy(_Batch(z, [4, 4, 4], toks))
    assert out["accepted_len"].tolist() == [4, 4, 4]
    assert out["next_token"].tolist() == [int(np.argmax(z[r * 5 + 4])) for r in range(3)]


def _gpu_greedy(b):
    from paper_2601_11652_gb300 import binding as wb
    dev = "cuda"
    logits = (torch.from_numpy(b.logits.view(np.int16)).to(dev).view(torch.bfloat16) if b.dtype == "bf16"
              else torch.from_numpy(b.logits).to(dev))
    empty = torch.empty(0, dtype=torch.float32, device=dev)
    t = dict(draft_lens=torch.from_numpy(b.draft_lens).to(dev), target_logits=logits,
             draft_tokens=torch.from_numpy(b.draft_tokens).to(dev), draft_probs=empty, accept_uniforms=empty,
             sample_uniforms=empty, accepted_len=torch.full((b.B,), -7, dtype=torch.int32, device=dev),
             next_token=torch.full((b.B,), -7, dtype=torch.int32, device=dev))
    args = wb.make_accept_args(**t)
    args.sample_uniforms = None
    ws = wb.alloc_workspace(wb.wisp_verify_workspace_size(None, args))
    wb.wisp_verify_accept_greedy(args, ws)
    torch.cuda.synchronize()
    assert wb.wisp_verify_get_device_status(ws)[0] == 0
    return t["accepted_len"].cpu().numpy(), t["next_token"].cpu().numpy()


@pytest.mark.gpu
@pytest.mark.parametrize("name", ["small-f32", "small-bf16-ties", "llama3_8b_b32"])
def test_gpu_greedy_matches_oracle(oracle_mod, name):
    if not torch.cuda.is_available():
        pytest.fail("GPU tests need a CUDA device")
    from paper_2601_11652_gb300 import build
    build.build()
    rng = np.random.default_rng(11)
    if name == "llama3_8b_b32":
        wb_ = wl.make_batch(name)
        b = _Batch(wb_.logits, wb_.draft_lens, wb_.draft_tokens, wb_.dtype)
        # make half of the drafts follow the target so that the walks run past row 0
        z = wl.bf16_bits_to_f32(b.logits).reshape(-1, b.V)
        qs = np.concatenate([[0], np.cumsum(b.draft_lens + 1)])
        ds = np.concatenate([[0], np.cumsum(b.draft_lens)])
        toks = b.draft_tokens.copy()
        for r in range(0, b.B, 2):
            for i in range(b.draft_lens[r]):
                toks[ds[r] + i] = int(np.argmax(z[qs[r] + i]))
        b.draft_tokens = toks
    else:
        k = rng.integers(0, 6, size=9).astype(np.int32)
        V = 3001
        z = rng.standard_normal((int(k.sum()) + 9, V)).astype(np.float32)
        if name.endswith("ties"):
            z = np.round(z * 2) / 2        # coarse values: many ties at the maximum
        qs = np.concatenate([[0], np.cumsum(k + 1)])
        toks = []
        for r in range(9):
            for i in range(k[r]):
                a = int(np.argmax(z[qs[r] + i]))
                toks.append(a if rng.random() < 0.7 else int(rng.integers(V)))
        dt = "bf16" if "bf16" in name else "f32"
        b = _Batch(wl.f32_to_bf16_bits(z) if dt == "bf16" else z, k, toks, dt)
    L, tok = _gpu_greedy(b)
    ref = oracle_mod.accept_greedy(b)
    np.testing.assert_array_equal(L, ref["accepted_len"])
    np.testing.assert_array_equal(tok, ref["next_token"])
