"""Serving loop: Algorithm 1's batches dispatched to real verification steps on the GPU.

At every dispatch epoch (Sec. 4.3) the loop asks `scheduler.schedule_epoch` for a batch of pending
requests and runs it through the library over one shared paged KV pool (Sec. 4.5):

    wisp_kv_reserve_append   pages for c + k + 1 tokens, the k + 1 new K/V rows written at c .. c + k
    wisp_verify_step         attention over the pool and the acceptance pass (Eq. 1-3)
    wisp_kv_commit           c <- c + 1 + L; the rejected drafts' pages go back to the pool

all enqueued on one stream and timed with CUDA events.  The server's clock advances by the measured
batch time; every request's completion is checked against its deadline (its SLO), and the measured
time is recorded beside the estimator's prediction T_hat(B) (Eq. batch_time, Sec. 4.4).  The
estimator is refitted on the batches measured so far (ordinary least squares), so that each
prediction used for scheduling is made before its batch is measured.

This module is host logic (argument marshalling, batching, bookkeeping) around the C ABI: every
step on the data path runs in the library's kernels.  The per-request payloads (query rows, new
K/V rows, logits, draft tokens and distributions, uniforms) come from the caller.
"""
from __future__ import annotations

import dataclasses
import heapq

import numpy as np
import torch

from . import binding as wb
from . import estimator as est
from .scheduler import BatchTime, schedule_epoch, schedule_fcfs

PAGE = 16


@dataclasses.dataclass
class Payload:
    """One verification round of one request: k drafted tokens (k + 1 query rows)."""
    q: np.ndarray             # [k + 1, Hq, D]  (bf16 as uint16 bits, or float32)
    k_new: np.ndarray         # [k + 1, Hkv, D]
    v_new: np.ndarray         # [k + 1, Hkv, D]
    logits: np.ndarray        # [k + 1, V]
    draft_tokens: np.ndarray  # [k] int32
    draft_probs: np.ndarray   # [k, V] float32
    accept_u: np.ndarray      # [k] float32
    sample_u: float


def _cat(arrays, tail_shape, dtype):
    return np.concatenate(arrays) if arrays else np.zeros((0, *tail_shape), dtype)


class PagedSessions:
    """n sessions over one shared paged KV pool, all state on the device: the pool, the free-page
    stack, per-session block-table rows and context lengths."""

    def __init__(self, n_sessions, Hkv, D, dtype, num_blocks, max_blocks, device="cuda"):
        self.dev = torch.device(device)
        self.dtype = dtype
        tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
        self.k_cache = torch.zeros((num_blocks, Hkv, PAGE, D), dtype=tdt, device=self.dev)
        self.v_cache = torch.zeros_like(self.k_cache)
        self.free_blocks = torch.arange(num_blocks, dtype=torch.int32, device=self.dev).flip(0).contiguous()
        self.free_count = torch.tensor([num_blocks], dtype=torch.int32, device=self.dev)
        self.tables = torch.full((n_sessions, max_blocks), -1, dtype=torch.int32, device=self.dev)
        self.ctx = torch.zeros(n_sessions, dtype=torch.int32, device=self.dev)
        self.num_blocks, self.max_blocks, self.Hkv, self.D = num_blocks, max_blocks, Hkv, D
        self.kv_ws = None

    def _ws(self, args):
        n = wb.wisp_kv_workspace_size(args)
        if self.kv_ws is None or self.kv_ws.numel() < n:
            self.kv_ws = wb.alloc_workspace(n, self.dev)
        return self.kv_ws

    def _dev(self, a, torch_dtype=None):
        if self.dtype == "bf16" and a.dtype == np.uint16:
            return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16).to(self.dev)
        t = torch.from_numpy(np.ascontiguousarray(a))
        return t.to(self.dev, dtype=torch_dtype) if torch_dtype else t.to(self.dev)

    def prefill(self, sids, k_rows, v_rows, stream=None):
        """Give sessions `sids` (empty so far) their prefixes: reserve pages for len(k_rows[i]) tokens,
        write the rows, and commit them all (as a round whose drafts are all accepted)."""
        idx = torch.tensor(sids, dtype=torch.long, device=self.dev)
        lens = [len(x) for x in k_rows]
        draft = torch.tensor([n - 1 for n in lens], dtype=torch.int32, device=self.dev)
        ctx = self.ctx[idx].contiguous()
        tables = self.tables[idx].contiguous()
        kn, vn = self._dev(np.concatenate(k_rows)), self._dev(np.concatenate(v_rows))
        args = wb.make_kv_args(draft_lens=draft, context_lens=ctx, block_tables=tables, free_blocks=self.free_blocks,
                               free_count=self.free_count, k_cache=self.k_cache, v_cache=self.v_cache, k_new=kn,
                               v_new=vn, total_q_rows=int(sum(lens)))
        ws = self._ws(args)
        wb.wisp_kv_reserve_append(args, ws, stream)
        acc = draft.clone()
        args = wb.make_kv_args(draft_lens=draft, context_lens=ctx, block_tables=tables, free_blocks=self.free_blocks,
                               free_count=self.free_count, k_cache=self.k_cache, v_cache=self.v_cache,
                               accepted_len=acc, total_q_rows=int(sum(lens)))
        wb.wisp_kv_commit(args, ws, stream)
        torch.cuda.synchronize(self.dev)
        code, rid = wb.wisp_verify_get_device_status(ws)
        if code != 0:
            raise RuntimeError(f"prefill: device status {code} (request {rid})")
        self.tables[idx] = tables
        self.ctx[idx] = ctx


@dataclasses.dataclass
class BatchResult:
    sids: list
    accepted_len: np.ndarray
    next_token: np.ndarray
    gpu_ms: float                 # reserve_append + step + commit, CUDA events on the stream
    out: torch.Tensor             # attention output [T_q, Hq, D] (device)
    block_tables: np.ndarray      # the batch's table rows as the step read them (after reserve)
    context_lens: np.ndarray      # c before the commit


class VerifyServer:
    """Runs verification batches of sessions through the library (reserve -> step -> commit)."""

    def __init__(self, sessions: PagedSessions, Hq: int, V: int, stream=None):
        self.s = sessions
        self.Hq, self.V = Hq, V
        self.stream = stream
        self.ws = None

    def run_batch(self, sids, payloads) -> BatchResult:
        s, dev = self.s, self.s.dev
        B = len(sids)
        k = [len(p.draft_tokens) for p in payloads]
        Tq = int(sum(k)) + B
        idx = torch.tensor(sids, dtype=torch.long, device=dev)
        draft = torch.tensor(k, dtype=torch.int32, device=dev)
        ctx = s.ctx[idx].contiguous()
        tables = s.tables[idx].contiguous()
        q = s._dev(np.concatenate([p.q for p in payloads]))
        kn = s._dev(np.concatenate([p.k_new for p in payloads]))
        vn = s._dev(np.concatenate([p.v_new for p in payloads]))
        logits = s._dev(np.concatenate([p.logits for p in payloads]))
        tokens = s._dev(_cat([p.draft_tokens for p in payloads], (), np.int32).astype(np.int32))
        probs = s._dev(_cat([p.draft_probs for p in payloads], (self.V,), np.float32).astype(np.float32))
        au = s._dev(_cat([p.accept_u for p in payloads], (), np.float32).astype(np.float32))
        su = s._dev(np.array([p.sample_u for p in payloads], np.float32))
        rid = torch.tensor(sids, dtype=torch.int64, device=dev)
        out = torch.empty_like(q)
        acc = torch.full((B,), -7, dtype=torch.int32, device=dev)
        tok = torch.full((B,), -7, dtype=torch.int32, device=dev)
        kv = wb.make_kv_args(draft_lens=draft, context_lens=ctx, block_tables=tables, free_blocks=s.free_blocks,
                             free_count=s.free_count, k_cache=s.k_cache, v_cache=s.v_cache, k_new=kn, v_new=vn,
                             accepted_len=acc, request_ids=rid, total_q_rows=Tq)
        attn = wb.make_attn_args(draft_lens=draft, context_lens=ctx, block_tables=tables, q=q, k_cache=s.k_cache,
                                 v_cache=s.v_cache, out=out, request_ids=rid, num_blocks=s.num_blocks)
        accp = wb.make_accept_args(draft_lens=draft, target_logits=logits, draft_tokens=tokens, draft_probs=probs,
                                   accept_uniforms=au, sample_uniforms=su, accepted_len=acc, next_token=tok,
                                   request_ids=rid)
        kws = s._ws(kv)
        n = wb.wisp_verify_workspace_size(attn, accp)
        if self.ws is None or self.ws.numel() < n:
            self.ws = wb.alloc_workspace(n, dev)
        stream = self.stream or torch.cuda.current_stream(dev)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(stream):
            a.record(stream)
            wb.wisp_kv_reserve_append(kv, kws, stream)
            tables_read = tables.clone()  # the rows the step reads (commit rewrites them)
            ctx_read = ctx.clone()
            wb.wisp_verify_step(attn, accp, self.ws, stream)
            wb.wisp_kv_commit(kv, kws, stream)
            b.record(stream)
        stream.synchronize()
        for ws, what in ((kws, "kv"), (self.ws, "verify")):
            code, r = wb.wisp_verify_get_device_status(ws)
            if code != 0:
                raise RuntimeError(f"{what}: device status {code} (request {r})")
        s.tables[idx] = tables
        s.ctx[idx] = ctx
        return BatchResult(list(sids), acc.cpu().numpy(), tok.cpu().numpy(), a.elapsed_time(b), out,
                           tables_read.cpu().numpy(), ctx_read.cpu().numpy())


@dataclasses.dataclass
class EpochRecord:
    t: float                  # dispatch time (s, server clock)
    sids: list
    measured_ms: float
    predicted_ms: float | None  # T_hat(batch) at dispatch (None before the first fit)
    violations: int
    verified: int             # accepted draft tokens in the batch


def calibrate(server: VerifyServer, sids, payload_fn, grid, reps=3):
    """Fit the estimator (Eq. batch_time) on this server: for every (B, k) of `grid`, batches of the
    first B sessions of `sids`, each drafting k tokens, measured `reps` times (after one warm-up
    batch).  payload_fn(sid, k, i) gives a Payload.  The sessions' contexts grow as their rounds
    commit.  Returns (coefficients, fit metrics)."""
    X, Y, i = [], [], 0
    server.run_batch(list(sids[:1]), [payload_fn(sids[0], 1, i)])
    for B, k in grid:
        for _ in range(reps):
            i += 1
            ctx = server.s.ctx[torch.tensor(sids[:B], device=server.s.dev)].cpu().numpy()
            res = server.run_batch(list(sids[:B]), [payload_fn(sid, k, i) for sid in sids[:B]])
            X.append(est.features(ctx, [k] * B))
            Y.append(res.gpu_ms * 1e-3)
    X, Y = np.array(X), np.array(Y)
    coef = est.fit_ols(X, Y)
    return coef, est.metrics(Y, est.predict(coef, X))


def serve_trace(server: VerifyServer, trace, payload_fn, *, policy="wisp", horizon=1e9, max_rounds=None,
                mem_budget=None, delta=0.002, max_batch=256, min_fit=6, T0=None, refit=True, on_batch=None):
    """Drive `trace` (a list of the first Request of each session; a session's next request arrives
    T_draft + T_network after its previous one completes, with the session's new context) through
    the server until every session has had `max_rounds` rounds or `horizon` passes.
    payload_fn(request, round_no) gives the round's Payload; its k must equal request.k.
    T0: the estimator to schedule with (coefficients, e.g. from `calibrate`); with refit it is
    refitted on the batches measured so far once there are min_fit of them.
    on_batch(result, payloads), if given, sees every batch.  Returns (records, coefficients in use
    at the end)."""
    mem_budget = mem_budget if mem_budget is not None else server.s.num_blocks
    coef = None if T0 is None else np.asarray(T0, np.float64)
    T = BatchTime(coef if coef is not None else [0.0, 0.0, 1e-9, 1e-4])
    events, seq = [], 0
    rounds = {}
    next_rid = max((r.rid for r in trace), default=0) + 1
    for r in trace:
        heapq.heappush(events, (r.arrival, seq, r))
        seq += 1
        rounds[r.device] = 0
    pending, t, busy_until = [], 0.0, 0.0
    X, Y, records = [], [], []
    while events or pending:
        if not pending or (events and events[0][0] <= busy_until):
            t, _, r = heapq.heappop(events)
            if t > horizon:
                break
            pending.append(r)
            continue
        t = max(t, busy_until)
        if t > horizon:
            break
        if policy == "wisp":
            batch = schedule_epoch(pending, t, mem_budget, delta, T)
            if not batch:  # nothing feasible: the most urgent request alone
                batch = [min(pending, key=lambda r: (r.deadline, r.rid))]
        else:
            batch = schedule_fcfs(pending, t, mem_budget, max_batch)
        pred = T(batch) * 1e3 if coef is not None else None
        payloads = [payload_fn(r, rounds[r.device]) for r in batch]
        res = server.run_batch([r.device for r in batch], payloads)
        if on_batch:
            on_batch(res, payloads)
        finish = t + res.gpu_ms * 1e-3
        ids = {r.rid for r in batch}
        pending = [r for r in pending if r.rid not in ids]
        viol = 0
        for r, L in zip(batch, res.accepted_len):
            viol += finish > r.deadline
            rounds[r.device] += 1
            if max_rounds is not None and rounds[r.device] >= max_rounds:
                continue
            nxt = dataclasses.replace(r, rid=next_rid, arrival=finish + r.t_draft + r.t_net, ctx=r.ctx + 1 + int(L))
            next_rid += 1
            heapq.heappush(events, (nxt.arrival, seq, nxt))
            seq += 1
        records.append(EpochRecord(t, [r.device for r in batch], res.gpu_ms, pred, viol, int(res.accepted_len.sum())))
        X.append(est.features([r.ctx for r in batch], [r.k for r in batch]))
        Y.append(res.gpu_ms * 1e-3)
        if refit and len(Y) >= min_fit:
            coef = est.fit_ols(np.array(X), np.array(Y))
            T = BatchTime(coef)
        busy_until = finish
    return records, coef


def summarise(records) -> dict:
    """Measured-vs-predicted error (MAPE over the batches predicted by a fit) and SLO outcomes."""
    pr = [(r.measured_ms, r.predicted_ms) for r in records if r.predicted_ms is not None]
    mape = float(100.0 * np.mean([abs(m - p) / m for m, p in pr])) if pr else None
    n = sum(len(r.sids) for r in records)
    return {"batches": len(records), "requests": n, "violations": sum(r.violations for r in records),
            "verified_tokens": sum(r.verified for r in records), "mape_pct": mape, "predicted_batches": len(pr),
            "mean_batch": n / max(1, len(records)), "gpu_ms_total": float(sum(r.measured_ms for r in records))}
