"""The paged KV maintenance calls (include/wisp_kv.h) against the plain-Python model (oracle/kv.py):
tables, free stack, free count, context lengths and the page contents, bit for bit."""
import numpy as np
import pytest
import torch

from oracle import kv as model

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.fail("GPU tests need a CUDA device")
    from paper_2601_11652_gb300 import build
    build.build()


def _state(rng, nb, B, mb, ctx_hi):
    perm = rng.permutation(nb).tolist()
    tables = [[-1] * mb for _ in range(B)]
    ctx = rng.integers(0, ctx_hi, size=B).tolist()
    for r in range(B):
        for b in range((ctx[r] + 15) // 16):
            tables[r][b] = perm.pop()
    stack = perm + [-1] * (nb - len(perm))
    return tables, stack, len(perm), ctx


def _run(seed, dtype, D, nb=1000, B=37, mb=40, Hkv=4, ctx_hi=400, k_hi=9):
    from paper_2601_11652_gb300 import binding as wb
    rng = np.random.default_rng(seed)
    tables, stack, F, ctx = _state(rng, nb, B, mb, ctx_hi)
    draft = rng.integers(0, k_hi + 1, size=B).tolist()
    T = sum(draft) + B
    npdt = np.float32
    k_new = rng.standard_normal((T, Hkv, D)).astype(npdt)
    v_new = rng.standard_normal((T, Hkv, D)).astype(npdt)
    k_cache = rng.standard_normal((nb, Hkv, 16, D)).astype(npdt)
    v_cache = rng.standard_normal((nb, Hkv, 16, D)).astype(npdt)
    tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
    if dtype == "bf16":  # both sides see the same bf16 values
        k_new, v_new, k_cache, v_cache = (torch.from_numpy(a).to(tdt).float().numpy() for a in (k_new, v_new, k_cache, v_cache))
    dev = lambda a, dt=None: torch.tensor(np.asarray(a), dtype=dt, device="cuda")
    g = dict(draft_lens=dev(draft, torch.int32), context_lens=dev(ctx, torch.int32),
             block_tables=dev(tables, torch.int32), free_blocks=dev(stack, torch.int32),
             free_count=dev([F], torch.int32), k_cache=dev(k_cache).to(tdt), v_cache=dev(v_cache).to(tdt),
             k_new=dev(k_new).to(tdt), v_new=dev(v_new).to(tdt))
    args = wb.make_kv_args(**g)
    ws = wb.alloc_workspace(wb.wisp_kv_workspace_size(args))
    wb.wisp_kv_reserve_append(args, ws)
    torch.cuda.synchronize()
    code, _ = wb.wisp_verify_get_device_status(ws)
    # the model
    mt, ms = [row[:] for row in tables], stack[:]
    mk, mv = k_cache.copy(), v_cache.copy()
    F1, codes = model.reserve_append(mt, ms, F, ctx, draft, nb, k_new, v_new, mk, mv)
    errs = {c for c in codes if c != 0}
    assert (code == 0) == (not errs) and (not errs or code in errs), (code, errs)
    assert g["block_tables"].cpu().numpy().tolist() == mt
    assert int(g["free_count"].item()) == F1
    assert np.array_equal(g["k_cache"].float().cpu().numpy(), mk)
    assert np.array_equal(g["v_cache"].float().cpu().numpy(), mv)
    # commit with random accepted lengths (requests that were not served keep their state)
    acc = [int(rng.integers(0, d + 1)) for d in draft]
    kd = [d if c == 0 else -1 for d, c in zip(draft, codes)]   # flag unserved requests as bad lengths
    g["draft_lens"] = dev(kd, torch.int32)
    g["accepted_len"] = dev(acc, torch.int32)
    args = wb.make_kv_args(**g)
    wb.wisp_kv_commit(args, ws)
    torch.cuda.synchronize()
    mctx = ctx[:]
    F2, codes2 = model.commit(mt, ms, F1, mctx, kd, acc)
    assert g["block_tables"].cpu().numpy().tolist() == mt
    assert g["context_lens"].cpu().numpy().tolist() == mctx
    assert int(g["free_count"].item()) == F2
    assert g["free_blocks"].cpu().numpy()[:F2].tolist() == ms[:F2]
    return codes, codes2


@pytest.mark.parametrize("dtype,D", [("bf16", 128), ("f32", 64), ("bf16", 64)])
def test_reserve_append_commit_match_the_model(dtype, D):
    codes, _ = _run(1 + D, dtype, D)
    assert all(c == 0 for c in codes)


def test_pool_exhaustion_serves_a_prefix():
    # at most 1 cached page per request (12 in all), at least 8 free, about 2.5 new pages each
    codes, _ = _run(7, "bf16", 128, nb=20, B=12, ctx_hi=16, k_hi=40)
    assert model.NO_BLOCKS in codes and codes[0] == 0
