"""GPU: Algorithm 1 driving real verification steps over a shared paged KV pool (Sec. 4.3-4.5).

A short synthetic trace of sessions (edge devices) is served by `serve.serve_trace`: at every epoch
the scheduler forms a batch, and the server runs wisp_kv_reserve_append -> wisp_verify_step ->
wisp_kv_commit on it.  Every batch is replayed on the host against the oracles on the same inputs:
oracle/kv.py for the page tables, the free stack and the context lengths (bit for bit), the fp64
oracle for the attention output (within the bf16 tolerance) and for the accepted lengths and extra
tokens (bit for bit outside the logged windows).  The measured batch times are compared with the
estimator's predictions (MAPE, reported).
"""
import numpy as np
import pytest
import torch

from oracle import kv as kvm
from paper_2601_11652_gb300 import workload as wl
from tests.gpu_util import ATTN_TOL, attn_max_err, compare_accept

pytestmark = pytest.mark.gpu

Hq, Hkv, D, V = 8, 2, 128, 4096
NB, MB = 900, 96          # pool pages; table row length (1536 tokens per session at most)
N_SESS, ROUNDS = 6, 5


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.fail("GPU tests need a CUDA device")
    from paper_2601_11652_gb300 import build
    build.build()


def test_scheduler_drives_real_steps(oracle_mod):
    from paper_2601_11652_gb300 import serve
    from paper_2601_11652_gb300.scheduler import Request

    rng = np.random.default_rng(7)
    ks = rng.integers(1, 7, size=N_SESS)
    prefixes = rng.integers(40, 400, size=N_SESS)
    sess = serve.PagedSessions(N_SESS, Hkv, D, "bf16", NB, MB)
    firsts = [wl.make_round((7, s, 0), k=int(ks[s]), Hq=Hq, Hkv=Hkv, D=D, V=V, prefix=int(prefixes[s]))
              for s in range(N_SESS)]
    sess.prefill(list(range(N_SESS)), [f["prefix_k"] for f in firsts], [f["prefix_v"] for f in firsts])

    # the host mirror: tables, free stack, contexts and the pool, kept by the KV oracle
    tables = [[-1] * MB for _ in range(N_SESS)]
    stack, F = list(range(NB))[::-1], NB
    ctx = [0] * N_SESS
    kc = np.zeros((NB, Hkv, 16, D), np.uint16)
    vc = np.zeros_like(kc)
    F, codes = kvm.reserve_append(tables, stack, F, ctx, [int(p) - 1 for p in prefixes], NB,
                                  np.concatenate([f["prefix_k"] for f in firsts]),
                                  np.concatenate([f["prefix_v"] for f in firsts]), kc, vc)
    assert codes == [0] * N_SESS
    F, _ = kvm.commit(tables, stack, F, ctx, [int(p) - 1 for p in prefixes], [int(p) - 1 for p in prefixes])
    assert sess.tables.cpu().numpy().tolist() == tables and sess.ctx.cpu().numpy().tolist() == ctx

    def payload(r, n):
        d = firsts[r.device] if n == 0 else wl.make_round((7, r.device, n), k=r.k, Hq=Hq, Hkv=Hkv, D=D, V=V)
        return serve.Payload(d["q"], d["k_new"], d["v_new"], d["logits"], d["draft_tokens"], d["draft_probs"],
                             d["accept_u"], d["sample_u"])

    state = {"F": F, "batches": 0, "logged": 0}

    def check(res, payloads):
        sids = res.sids
        bt = [tables[s][:] for s in sids]
        bc = [ctx[s] for s in sids]
        bk = [len(p.draft_tokens) for p in payloads]
        F1, codes = kvm.reserve_append(bt, stack, state["F"], bc, bk, NB, np.concatenate([p.k_new for p in payloads]),
                                       np.concatenate([p.v_new for p in payloads]), kc, vc)
        assert codes == [0] * len(sids)
        assert res.block_tables.tolist() == bt and res.context_lens.tolist() == bc
        hb = wl.VerifyBatch(
            name="served", B=len(sids), Hq=Hq, Hkv=Hkv, D=D, V=V, block_size=16, dtype="bf16",
            request_ids=np.array(sids, np.int64), draft_lens=np.array(bk, np.int32),
            context_lens=np.array(bc, np.int32), block_tables=np.array(bt, np.int32), num_blocks=NB,
            q=np.concatenate([p.q for p in payloads]), k_cache=kc, v_cache=vc,
            logits=np.concatenate([p.logits for p in payloads]),
            draft_tokens=np.concatenate([p.draft_tokens for p in payloads]).astype(np.int32),
            draft_probs=np.concatenate([p.draft_probs for p in payloads]).astype(np.float32),
            accept_uniforms=np.concatenate([p.accept_u for p in payloads]).astype(np.float32),
            sample_uniforms=np.array([p.sample_u for p in payloads], np.float32),
            sigma=np.zeros(len(sids)))
        ref = oracle_mod.accept(hb)
        n, logged = compare_accept(hb, res.accepted_len, res.next_token, ref)
        state["logged"] += len(logged)
        err = attn_max_err(res.out.float().cpu().numpy(), oracle_mod.attention(hb))
        assert err <= ATTN_TOL["bf16"], f"attention max abs error {err}"
        F2, codes = kvm.commit(bt, stack, F1, bc, bk, [int(x) for x in res.accepted_len])
        assert codes == [0] * len(sids)
        for i, s in enumerate(sids):
            tables[s], ctx[s] = bt[i], bc[i]
        state["F"] = F2
        state["batches"] += 1
        assert sess.tables.cpu().numpy().tolist() == tables
        assert sess.ctx.cpu().numpy().tolist() == ctx
        assert int(sess.free_count.item()) == F2
        assert sess.free_blocks.cpu().numpy()[:F2].tolist() == stack[:F2]

    # sessions of three SLO classes, all first rounds at t = 0 (the first epoch batches them)
    trace = []
    for s in range(N_SESS):
        k = int(ks[s])
        trace.append(Request(rid=s, device=s, arrival=0.0, k=k, ctx=int(prefixes[s]),
                             alpha=0.7, speed=float([20.0, 40.0, 80.0][s % 3]), t_draft=0.002 * k, t_net=0.003))
    # the estimator, fitted beforehand on scratch sessions of the same shape (a separate pool)
    scratch = serve.PagedSessions(8, Hkv, D, "bf16", 600, MB)
    pre = [wl.make_round((8, s, 0), k=1, Hq=Hq, Hkv=Hkv, D=D, V=V, prefix=int(100 + 80 * s)) for s in range(8)]
    scratch.prefill(list(range(8)), [f["prefix_k"] for f in pre], [f["prefix_v"] for f in pre])

    def cal_payload(sid, k, i):
        d = wl.make_round((9, sid, i), k=k, Hq=Hq, Hkv=Hkv, D=D, V=V)
        return serve.Payload(d["q"], d["k_new"], d["v_new"], d["logits"], d["draft_tokens"], d["draft_probs"],
                             d["accept_u"], d["sample_u"])

    coef0, fit = serve.calibrate(serve.VerifyServer(scratch, Hq, V), list(range(8)), cal_payload,
                                 [(B, k) for B in (1, 2, 4, 8) for k in (1, 3, 6)])
    server = serve.VerifyServer(sess, Hq, V)
    records, coef = serve.serve_trace(server, trace, payload, max_rounds=ROUNDS, T0=coef0, refit=False,
                                      on_batch=check)
    summary = serve.summarise(records)
    print("calibration fit:", coef0, fit)
    print("serve trace:", summary)
    assert summary["requests"] == N_SESS * ROUNDS
    assert state["batches"] == len(records)
    assert summary["predicted_batches"] > 0 and np.isfinite(summary["mape_pct"])
    assert any(len(r.sids) > 1 for r in records)  # the scheduler batched requests together
    assert [int(x) for x in sess.ctx.cpu()] == ctx
