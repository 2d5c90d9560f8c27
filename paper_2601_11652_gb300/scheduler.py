"""SLO-aware verification batch scheduling (Sec. 4.3, Algorithm 1) and a trace-driven simulator.

Per request i the scheduler knows (Sec. 4.3):
  * the expected verified tokens  g_i = N^v_i = alpha_i * N_d,i                     (Eq. nv-est)
  * a deadline  d_i = a_i + tau_c(i),  tau_c = alpha N_d / s_c - T_draft - T_network (Eq. server-budget)
  * its verification cost v_i: read here as the estimator's time of verifying i alone,
    T_hat({i}) (Sec. 4.4), so that the latest start time below is conservative
  * a memory footprint m_i: the KV pages of its c + k + 1 tokens
and at each dispatch epoch t builds a batch with Algorithm 1: utility U_i = g_i / v_i, latest start
time LST_i = d_i - v_i - delta (Eq. lst); requests with t >= LST_i are critical and admitted first in
earliest-deadline order, then the rest by decreasing utility, each addition checked against the
memory budget and the deadline of every request in the batch (t + T_hat(B) <= min d_j), stopping at
the first violation.

`simulate` drives FCFS or this scheduler over synthetic edge devices (SLO classes of target token
speeds, per-device acceptance rates and draft lengths), with the batch time from the fitted
estimator of this library's verification step.  Host-side Python; no GPU.
"""
from __future__ import annotations

import dataclasses
import heapq
import math

import numpy as np

from . import estimator as est

PAGE = 16


@dataclasses.dataclass
class Request:
    rid: int
    device: int
    arrival: float        # a_i (s)
    k: int                # draft length N_d
    ctx: int              # cached prefix c (tokens)
    alpha: float          # acceptance estimate of the device
    speed: float          # target token speed s_c of the device's SLO class (tokens/s)
    t_draft: float        # T_draft of this round (s)
    t_net: float          # T_network of this round (s)

    @property
    def gain(self) -> float:           # g_i = N^v_i (Eq. nv-est)
        return self.alpha * self.k

    @property
    def deadline(self) -> float:       # d_i = a_i + tau_c (Eq. server-budget)
        return self.arrival + self.alpha * self.k / self.speed - self.t_draft - self.t_net

    @property
    def pages(self) -> int:            # m_i
        return (self.ctx + self.k + 1 + PAGE - 1) // PAGE


class BatchTime:
    """T_hat(B) = a N_linear + b_compute N_interactions + b_read N_cached + c (Eq. batch_time)."""

    def __init__(self, coef):
        self.coef = np.asarray(coef, dtype=np.float64)

    def __call__(self, batch) -> float:
        if not batch:
            return 0.0
        f = est.features([r.ctx for r in batch], [r.k for r in batch])
        return float(f @ self.coef[:3] + self.coef[3])


def schedule_epoch(pending, t: float, mem_budget: int, delta: float, T) -> list:
    """Algorithm 1 at dispatch epoch t: the batch to dispatch (possibly empty)."""
    cost = {r.rid: T([r]) for r in pending}
    crit = [r for r in pending if t >= r.deadline - cost[r.rid] - delta]
    crit_ids = {r.rid for r in crit}
    non = [r for r in pending if r.rid not in crit_ids]
    crit.sort(key=lambda r: (r.deadline, r.rid))                          # EDF
    non.sort(key=lambda r: (-r.gain / cost[r.rid], r.rid))                # decreasing utility

    batch, mem, dmin = [], 0, math.inf

    def feasible_add(r) -> bool:
        return mem + r.pages <= mem_budget and t + T(batch + [r]) <= min(dmin, r.deadline)

    stop = False
    for r in crit:
        if feasible_add(r):
            batch.append(r)
            mem += r.pages
            dmin = min(dmin, r.deadline)
        else:
            stop = True
            break
    if not stop:
        for r in non:
            if feasible_add(r):
                batch.append(r)
                mem += r.pages
                dmin = min(dmin, r.deadline)
            else:
                break
    return batch


def schedule_fcfs(pending, t: float, mem_budget: int, max_batch: int) -> list:
    """First come, first served: arrival order up to the memory budget and a batch-size cap."""
    batch, mem = [], 0
    for r in sorted(pending, key=lambda r: (r.arrival, r.rid)):
        if len(batch) >= max_batch or mem + r.pages > mem_budget:
            break
        batch.append(r)
        mem += r.pages
    return batch


@dataclasses.dataclass
class SimResult:
    requests: int
    violations: int
    verified_tokens: float
    horizon: float

    @property
    def violation_rate(self) -> float:
        return self.violations / max(1, self.requests)

    @property
    def goodput(self) -> float:       # verified (committed) tokens per second
        return self.verified_tokens / self.horizon


def simulate(policy: str, n_devices: int, T, horizon: float = 30.0, seed: int = 0, mem_budget: int = 200000,
             delta: float = 0.005, max_batch: int = 256, speeds=(2.0, 4.0, 6.0, 8.0)) -> SimResult:
    """Edge devices draft k tokens (T_draft = k * per-token time), send them (T_network), wait for the
    verification and repeat; the server dispatches a batch whenever it is idle and requests wait.
    A request's verified tokens are drawn from the device's acceptance law (geometric, truncated at
    k) plus the extra token; it violates its SLO when it completes after its deadline."""
    rng = np.random.default_rng(seed)
    dev_speed = rng.choice(speeds, size=n_devices)
    dev_alpha = rng.uniform(0.4, 0.9, size=n_devices)
    dev_tok = rng.uniform(0.01, 0.04, size=n_devices)        # edge seconds per drafted token
    dev_net = rng.uniform(0.005, 0.03, size=n_devices)       # network seconds per round
    dev_ctx = rng.integers(256, 4096, size=n_devices)
    events = []                                              # (time, seq, request)
    seq = 0
    rid = 0

    def new_round(dv, t0):
        nonlocal seq, rid
        k = int(rng.integers(2, 9))
        td = k * dev_tok[dv]
        r = Request(rid, dv, t0 + td + dev_net[dv], k, int(dev_ctx[dv]), float(dev_alpha[dv]), float(dev_speed[dv]),
                    td, float(dev_net[dv]))
        rid += 1
        heapq.heappush(events, (r.arrival, seq, r))
        seq += 1

    for dv in range(n_devices):
        new_round(dv, float(rng.uniform(0.0, 0.2)))
    pending, t, busy_until = [], 0.0, 0.0
    done = viol = 0
    verified = 0.0
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
            if not batch:   # nothing feasible: dispatch the most urgent request alone
                batch = [min(pending, key=lambda r: (r.deadline, r.rid))]
        else:
            batch = schedule_fcfs(pending, t, mem_budget, max_batch)
        finish = t + T(batch)
        ids = {r.rid for r in batch}
        pending = [r for r in pending if r.rid not in ids]
        for r in batch:
            done += 1
            viol += finish > r.deadline
            acc = 0
            while acc < r.k and rng.random() < r.alpha:
                acc += 1
            verified += acc + 1
            dev_ctx[r.device] += acc + 1
            new_round(r.device, finish + dev_net[r.device] / 2)
        busy_until = finish
    return SimResult(done, viol, verified, horizon)
