#!/usr/bin/env python
"""Benchmark of the batched speculative-verification step (WISP, Sec. 4.5).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME] [--impl ours|reference]
                    [--no-per-config]

One step = one call of wisp_verify_step on one synthetic verification batch:
paged GQA attention for every request's k+1 new tokens (Sec. 4.4-4.5) and the
in-order acceptance pass with the extra-token draw (Eq. 1-3).  The headline
workload is the largest single-GPU configuration, hetero_b512 (512 requests,
Qwen-like vocabulary, mixed contexts); the line's `per_config` object carries
the same measurements for the other workloads (llama3_8b_b32, fanin_b256,
longctx_b16).  Prints one JSON line (rank 0).  Under torchrun every rank
verifies its own batch (requests are independent: weak scaling, no collective
on the data path).

Per workload: the K timed steps (L2 flushed between steps), a sustained loop
of the same step for at least two seconds with the SM clocks sampled under
load (median and p90), the two entry points alone for two seconds each (their
HBM rooflines), the end-to-end step fed from pinned host memory through one
staging buffer, and the fp64 oracle on a bounded sample (cpu_baseline).

--impl reference times the fp64 CPU oracle (the baseline this library is
checked against) on the host cores, on bounded samples of the same workload.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "verified draft tokens/sec per verify step; achieved HBM GB/s (% of GB300 peak)"
UNIT = "verified_tokens/s"
FLUSH_BYTES = 512 << 20  # > 4x the 126 MB L2: written between timed steps


# --------------------------------------------------------------------------
# algorithmic bytes (what the method must move; per step)
# --------------------------------------------------------------------------
def attention_bytes(b) -> int:
    s = 2 if b.dtype == "bf16" else 4
    n = b.context_lens.astype(np.int64) + b.draft_lens + 1
    kv = int(n.sum()) * b.Hkv * b.D * 2 * s          # K and V of every visible token, read once
    qo = int(b.total_q_rows) * b.Hq * b.D * 2 * s     # Q read, O written
    bt = int(((n + 15) // 16).sum()) * 4              # block-table entries
    return kv + qo + bt


def accept_bytes(b, L) -> int:
    s = 2 if b.dtype == "bf16" else 4
    L = np.asarray(L, np.int64)
    k = b.draft_lens.astype(np.int64)
    rows = int((L + 1).sum()) * b.V * s               # logit rows 0..L (the walk stops at the first rejection)
    qrow = int((L < k).sum()) * b.V * 4               # the draft row at the rejection (residual draw)
    decisions = int(np.minimum(L + 1, k).sum())
    gathers = decisions * (32 + 32 + 4 + 4)           # sectors of z(y), q(y); token, uniform
    return rows + qrow + gathers + b.B * 16


def _launches_per_step(b) -> int:
    """Kernels of this library one wisp_verify_step launches: planner, attention (tensor-core
    kernel for bf16; SIMT kernel + combine for fp32), acceptance (one persistent kernel)."""
    return 3 if b.dtype == "bf16" else 4


def _peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


# the sources each profiled kernel is built from (its launch set-up in api.cu included)
KERNEL_SOURCES = {
    "attention": ("api.cu", "attn.cuh", "attn_tc.cu", "common.cuh", "plan.cu", "plan.cuh", "sm100_ptx.cuh"),
    "accept": ("accept.cu", "accept.cuh", "api.cu", "common.cuh", "plan.cu", "plan.cuh", "sm100_ptx.cuh"),
}


def _kernel_sha(kernel: str = None) -> str:
    """sha256 (16 hex digits) of the kernel's sources, or of every csrc/*.cu, *.cuh if kernel is None."""
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2601_11652_gb300", "csrc")
    want = KERNEL_SOURCES.get(kernel)
    for name in sorted(os.listdir(csrc)):
        if name.endswith((".cu", ".cuh")) and (want is None or name in want):
            with open(os.path.join(csrc, name), "rb") as f:
                h.update(name.encode() + f.read())
    return h.hexdigest()[:16]


def _profile_traffic(kernel: str, workload: str):
    """DRAM bytes per launch of `kernel` from the committed ncu summary, if it matches this source."""
    path = os.path.join(ROOT, "profiles", f"{kernel}_{workload}.md")
    try:
        text = open(path).read()
    except OSError:
        return None
    sha = re.search(r"kernel_source_sha:\s*(\w+)", text)
    tr = re.search(r"dram_bytes_per_launch:\s*([0-9.eE+]+)", text)
    if not sha or not tr or sha.group(1) != _kernel_sha(kernel):
        return None
    return float(tr.group(1))


def _profile_inst(kernel: str, workload: str):
    """Warp instructions per launch summed over the kernels of the committed ncu summary of
    `kernel`, if it matches this source (None otherwise)."""
    path = os.path.join(ROOT, "profiles", f"{kernel}_{workload}.md")
    try:
        text = open(path).read()
    except OSError:
        return None
    sha = re.search(r"kernel_source_sha:\s*(\w+)", text)
    inst = re.findall(r"\|\s*smsp__inst_executed\.sum\s*\|\s*([0-9.eE+]+)\s*inst", text)
    if not sha or not inst or sha.group(1) != _kernel_sha(kernel):
        return None
    return float(sum(float(x) for x in inst))


def issue_roofline(warp_inst: float, ms: float, sms: int, sm_mhz: float):
    """Instruction-issue view of a kernel group bound by arithmetic and barriers rather than bytes:
    warp instructions per second against the issue peak, sms x 4 schedulers x 1 warp instruction
    per clock at the given SM clock."""
    if not warp_inst or not ms or not sms or not sm_mhz:
        return None
    achieved = warp_inst / (ms * 1e-3) / 1e9
    peak = sms * 4 * sm_mhz * 1e6 / 1e9
    return {"bound": "issue", "achieved": achieved, "peak": peak, "unit": "G warp-inst/s",
            "frac": achieved / peak, "warp_inst_per_launch": warp_inst}


# --------------------------------------------------------------------------
# clocks during the timed region
# --------------------------------------------------------------------------
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.idx = gpu_index
        self.proc = None
        # raw samples: $BENCH_CLOCKS_DIR if set, else the temporary directory (the JSON line
        # carries their summary)
        out_dir = os.environ.get("BENCH_CLOCKS_DIR") or tempfile.gettempdir()
        self.path = os.path.join(out_dir, f"clocks_bench_{os.getpid()}.csv")

    def start(self):
        try:
            os.makedirs(os.path.dirname(self.path), exist_ok=True)
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.idx), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=self.f, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.f.close()
        return self.summarise(self.path)

    @staticmethod
    def summarise(path: str):
        """Median SM clock, max clock and the throttle reasons seen in a sample file."""
        rows = []
        for line in open(path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                rows.append((float(parts[1]), float(parts[2]), parts[5:9]))
            except ValueError:
                continue
        if not rows:
            return None
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for _, _, flags in rows for i, v in enumerate(flags) if v.lower() == "active"})
        return {"sm_mhz": statistics.median(r[0] for r in rows), "sm_max_mhz": max(r[1] for r in rows),
                "reasons": reasons, "samples": len(rows)}


# --------------------------------------------------------------------------
# oracle timing (cpu_baseline, and the reference arm)
# --------------------------------------------------------------------------
def time_oracle(batch, budget_s: float, start: int = 0):
    """Run the oracle (attention + acceptance) on consecutive requests until budget_s is spent."""
    import oracle
    threads = os.cpu_count() or 1
    t0 = time.perf_counter()
    done, verified = 0, 0
    r = start
    while True:
        sub = batch.subset([r % batch.B])
        oracle.attention(sub, nthreads=threads)
        res = oracle.accept(sub, nthreads=threads)
        verified += int(res["accepted_len"].sum())
        done += 1
        r += 1
        if time.perf_counter() - t0 >= budget_s:
            break
    return done, verified, time.perf_counter() - t0, threads


def cpu_baseline(batch, budget_s=10.0):
    done, verified, dt, threads = time_oracle(batch, budget_s)
    return {"value": verified / dt, "unit": UNIT, "cores": threads, "kind": "oracle",
            "sample": f"{done} requests of {batch.name} (attention + acceptance, fp64), {dt:.1f} s"}


def run_reference(args, batch):
    """The oracle as the reference arm: each step is a bounded sample of the workload, the
    requests that follow the previous step's (cycling through the batch) until about
    per_step_s of oracle work is done (at least one request), so that the whole run stays within a
    few minutes whatever the requests' sizes."""
    per_step_s = min(3.0, 240.0 / max(1, args.steps + args.warmup))
    nxt = 0
    for _ in range(args.warmup):
        d = time_oracle(batch, per_step_s, start=nxt)[0]
        nxt += d
    ms, verified, done, threads = [], 0, 0, 1
    for _ in range(args.steps):
        d, v, dt, threads = time_oracle(batch, per_step_s, start=nxt)
        nxt += d
        ms.append(dt * 1e3)
        verified += v
        done += d
    total_s = sum(ms) / 1e3
    value = verified / total_s
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": sum(ms) / len(ms),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": _config(batch, args),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": threads, "kind": "oracle",
                             "sample": f"about {per_step_s:.1f} s of requests of {batch.name} per step (at least one), "
                                       f"{done} in total"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def _config(batch, args):
    return {"workload": batch.name, "B": batch.B, "Hq": batch.Hq, "Hkv": batch.Hkv, "D": batch.D, "V": batch.V,
            "kv_tokens": batch.kv_tokens(), "draft_tokens": batch.total_draft, "block_size": 16,
            "kv_dtype": batch.dtype, "accumulate": "fp32", "parallelism": f"replicas{args.gpus}",
            "l2": "flushed between timed steps (512 MiB write)"}


# --------------------------------------------------------------------------
# our arm
# --------------------------------------------------------------------------
HEADLINE = "hetero_b512"  # the largest configuration that fits one GPU
PER_CONFIG = ("llama3_8b_b32", "fanin_b256", "longctx_b16")
SUSTAIN_S = 2.0           # seconds of device time per sustained / per-entry-point loop


def _time_loop(fn, steps, flush, torch):
    """Device time (ms) of each of `steps` calls of fn, the L2 flushed (outside the events) before each."""
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    for i in range(steps):
        flush.zero_()
        starts[i].record()
        fn()
        ends[i].record()
    torch.cuda.synchronize()
    return [s.elapsed_time(e) for s, e in zip(starts, ends)]


def _time_for(fn, seconds, flush, torch):
    """Like _time_loop, repeated until `seconds` of device time are measured (at least 20 calls)."""
    probe = _time_loop(fn, 5, flush, torch)
    n = max(20, int(seconds * 1e3 / max(1e-3, float(np.median(probe)))))
    return _time_loop(fn, n, flush, torch)


def _stats(ms):
    a = np.asarray(ms, np.float64)
    return {"ms_mean": float(a.mean()), "ms_median": float(np.median(a)), "ms_p90": float(np.percentile(a, 90)),
            "steps": int(a.size), "seconds": float(a.sum() / 1e3)}


def aggregate_ranks(total_ms: float, verified: int, world: int, device):
    """Whole-job numbers of N replicas: the slowest rank's time (max) and every rank's verified
    tokens (sum).  The replicas verify independent batches, so this is the only collective."""
    if world <= 1:
        return total_ms, verified
    import torch
    import torch.distributed as dist
    t = torch.tensor([total_ms], device=device, dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    v = torch.tensor([verified], device=device, dtype=torch.int64)
    dist.all_reduce(v, op=dist.ReduceOp.SUM)
    dist.barrier()
    return float(t.item()), int(v.item())


def _h2d_gbs(host, dst, torch):
    """Measured host-to-device bandwidth (GB/s) of one copy of the pinned tensor `host` into `dst`."""
    for _ in range(2):
        dst.copy_(host, non_blocking=True)
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for _ in range(5):
        dst.copy_(host, non_blocking=True)
    b.record()
    torch.cuda.synchronize()
    return 5 * host.numel() * host.element_size() / (a.elapsed_time(b) * 1e-3) / 1e9


def _e2e(batch, db, verified, torch, dev, seconds=None):
    """End to end through the library's public path: each step copies its inputs from one pinned
    staging buffer (one host-to-device copy, overlapped with the previous step on a copy stream),
    verifies, and reads its results back (one device-to-host copy).  Throughput over the steps."""
    from paper_2601_11652_gb300.device_batch import StagedSteps
    seconds = SUSTAIN_S if seconds is None else seconds
    st = StagedSteps(batch, device=dev, pool=(db.t["k_cache"], db.t["v_cache"]))
    for _ in range(3):
        out = st.enqueue()
    torch.cuda.synchronize()
    assert int(out[0].sum()) == verified, "end-to-end results differ from the resident batch's"
    one = float(np.median(_time_loop(st.enqueue, 3, torch.empty(16, device=dev), torch)))
    n = max(10, int(seconds * 1e3 / max(one, 1e-3)))
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    a.record()
    for _ in range(n):
        out = st.enqueue()
    b.record()
    torch.cuda.synchronize()
    ms = a.elapsed_time(b) / n
    assert int(out[0].sum()) == verified
    gbs = _h2d_gbs(st.host, st.bufs[0], torch)
    res = {"value": verified / (ms / 1e3), "unit": UNIT, "h2d_bytes_per_step": st.h2d_bytes,
           "d2h_bytes_per_step": st.d2h_bytes, "ms_per_step": ms, "steps": n,
           "h2d_gbs_measured": gbs, "copy_bound_ms": st.nbytes / (gbs * 1e9) * 1e3,
           "note": "inputs staged in one pinned buffer, one copy per step overlapped with the previous step; "
                   "the paged KV cache (prefix cache) stays resident in HBM"}
    del st
    return res


def measure(batch, db, verified, L, torch, dev, flush, sampler_cls, local_rank, cpu_s):
    """Everything but the exact-K timed region for one workload: the sustained step loop (clocks
    sampled), the entry points alone, the rooflines, end to end and the oracle sample."""
    sampler = sampler_cls(local_rank)
    sampler.start()
    time.sleep(0.3)
    sus = _time_for(db.step, SUSTAIN_S, flush, torch)
    attn_ms = _time_for(db.attention, SUSTAIN_S, flush, torch)
    acc_ms = _time_for(db.accept, SUSTAIN_S, flush, torch)
    clocks = sampler.stop()
    code, rid = db.device_status()
    if code != 0:
        raise RuntimeError(f"device status {code} at request {rid} ({batch.name})")
    ab, cb = attention_bytes(batch), accept_bytes(batch, L)
    peak, peak_kind = _peaks()
    ta, tc = float(np.median(attn_ms)), float(np.median(acc_ms))
    attn_gbs, acc_gbs = ab / (ta * 1e-3) / 1e9, cb / (tc * 1e-3) / 1e9
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    try:
        acc_issue = issue_roofline(_profile_inst("accept", batch.name), tc, sms,
                                   clocks["sm_mhz"] if clocks else None)
    except Exception:
        acc_issue = None
    sus_stats = _stats(sus)
    return {
        "sustained": sus_stats,
        "roofline": {"bound": "hbm", "kernel": "attention entry point (planner + tensor-core attention kernel)",
                     "achieved": attn_gbs, "peak": peak, "peak_kind": peak_kind, "unit": "GB/s",
                     "frac": attn_gbs / peak, "traffic": _profile_traffic("attention", batch.name),
                     "algorithmic_bytes_per_launch": ab, "ms_median": ta,
                     "ms_p90": float(np.percentile(attn_ms, 90)), "steps": len(attn_ms)},
        "accept_roofline": {"bound": "hbm", "kernel": "acceptance entry point (planner + acceptance kernel)",
                            "achieved": acc_gbs, "peak": peak, "peak_kind": peak_kind, "unit": "GB/s",
                            "frac": acc_gbs / peak, "algorithmic_bytes_per_launch": cb,
                            "traffic": _profile_traffic("accept", batch.name), "issue": acc_issue,
                            "ms_median": tc, "ms_p90": float(np.percentile(acc_ms, 90)), "steps": len(acc_ms)},
        "step_algorithmic_gbs": (ab + cb) / (sus_stats["ms_median"] * 1e-3) / 1e9,
        "mean_acceptance": _acceptance(batch, L),
        "e2e": _e2e(batch, db, verified, torch, dev),
        "cpu_baseline": cpu_baseline(batch, cpu_s),
        "clocks": clocks,
    }


def _acceptance(batch, L):
    """Measured acceptance rate (accepted / drafted tokens) and the configuration's target: the
    workload draws its draft noise so that a single-token decision accepts with the configured
    probability alpha; the per-request walk stops at the first rejection, so the fraction of all
    drafted tokens that are accepted is lower than alpha."""
    from paper_2601_11652_gb300 import workload as wl
    rule = wl.SPECS[batch.name].noise_rule if batch.name in wl.SPECS else None
    target = None
    if rule and rule[0] == "alpha":
        target = float(rule[1])
    elif rule and rule[0] == "alpha_uniform":
        target = [float(rule[1]), float(rule[2])]
    return {"accepted_over_drafted": float(np.sum(L) / max(1, batch.total_draft)),
            "config_alpha_per_decision": target}


def _prepare(name, torch, dev, warmup, flush):
    from paper_2601_11652_gb300 import workload as wl
    from paper_2601_11652_gb300.device_batch import DeviceBatch
    batch = wl.make_batch(name)
    db = DeviceBatch.from_host(batch, device=dev)
    for _ in range(max(3, warmup)):
        flush.zero_()
        db.step()
    torch.cuda.synchronize()
    code, rid = db.device_status()
    if code != 0:
        raise RuntimeError(f"device status {code} at request {rid} ({name})")
    L = db.results()["accepted_len"]
    return batch, db, L, int(L.sum())


def run_ours(args, rank, world, local_rank):
    import torch
    import torch.distributed as dist

    from paper_2601_11652_gb300 import build

    build.build()
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    if world > 1:
        dist.init_process_group("nccl", device_id=dev)
    flush = torch.empty(FLUSH_BYTES, dtype=torch.uint8, device=dev)

    batch, db, L, verified = _prepare(args.workload, torch, dev, args.warmup, flush)
    sampler = ClockSampler(local_rank) if rank == 0 else None
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    if sampler:
        sampler.start()
        time.sleep(0.3)
    ms = _time_loop(db.step, args.steps, flush, torch)   # the timed region: exactly K steps
    torch.cuda.synchronize()
    code, rid = db.device_status()
    if code != 0:
        raise RuntimeError(f"device status {code} at request {rid} after the timed steps")
    total_ms, verified_all = aggregate_ranks(sum(ms), verified, world, dev)
    ms_per_step = total_ms / args.steps
    value = verified_all / (ms_per_step / 1e3)
    # the same step for two more seconds, so that the clock record holds samples under load
    tail = _time_for(db.step, SUSTAIN_S, flush, torch)
    clocks = sampler.stop() if sampler else None
    if rank != 0:
        if world > 1:
            dist.barrier()
        return
    extra = measure(batch, db, verified, L, torch, dev, flush, ClockSampler, local_rank, 10.0)
    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_per_step, **{k: v for k, v in _stats(ms).items()
                                                                  if k in ("ms_median", "ms_p90")},
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": batch.dtype,
            "data": "synthetic", "config": _config(batch, args)}
    line.update({k: extra[k] for k in ("roofline", "accept_roofline", "step_algorithmic_gbs", "mean_acceptance",
                                        "cpu_baseline", "e2e")})
    line["sustained"] = _stats(tail)
    line["emitted_tokens_per_s"] = (verified_all + batch.B * world) / (ms_per_step / 1e3)
    line["gpu_launches"] = _launches_per_step(batch) * args.steps
    line["clocks"] = dict(clocks or {}, window="the K timed steps and 2 s more of the same step")
    line["clocks_entry_points"] = extra["clocks"]
    del db
    torch.cuda.empty_cache()
    if args.per_config:
        per = {}
        for name in PER_CONFIG:
            if name == args.workload:
                continue
            b2, db2, L2, v2 = _prepare(name, torch, dev, args.warmup, flush)
            k = _time_loop(db2.step, args.steps, flush, torch)
            ent = {"config": _config(b2, args), "value": v2 / (float(np.mean(k)) / 1e3), "unit": UNIT,
                   "ms_per_step": float(np.mean(k)), "ms_median": float(np.median(k)),
                   "ms_p90": float(np.percentile(k, 90)), "steps": len(k)}
            ent.update(measure(b2, db2, v2, L2, torch, dev, flush, ClockSampler, local_rank, 5.0))
            per[name] = ent
            del db2
            torch.cuda.empty_cache()
        line["per_config"] = per
    print(json.dumps(line), flush=True)
    if world > 1:
        dist.barrier()


# --------------------------------------------------------------------------
# latency table for the verification-time estimator (Sec. 4.4, Eq. batch_time)
# --------------------------------------------------------------------------
LT_BATCHES = (1, 2, 4, 8, 16, 32, 64, 128, 256, 512)
LT_DRAFTS = (1, 2, 4, 8, 16)   # draft tokens per request (sum k = B * this)


def latency_table(path: str, max_b: int, reps: int):
    """Step / attention / acceptance times over batch size x draft length on the Llama-3-8B-shaped
    layer (32/8/128 bf16 KV, V = 128256, contexts ~ U{512..4096}), with the estimator's features;
    writes a CSV and fits T_step = a N_linear + b_compute N_interactions + b_read N_cached + c."""
    import csv
    import torch
    from paper_2601_11652_gb300 import build, estimator as est, workload as wl
    from paper_2601_11652_gb300.device_batch import DeviceBatch
    build.build()
    flush = torch.empty(FLUSH_BYTES, dtype=torch.uint8, device="cuda")
    rng = np.random.default_rng(2601_11652)
    rows = []
    for B in LT_BATCHES:
        if B > max_b:
            continue
        for kk in LT_DRAFTS:
            k = np.full(B, kk, np.int32)
            c = rng.integers(512, 4097, size=B).astype(np.int32)
            batch = wl.make_batch_from_lengths(f"lt_b{B}_k{kk}", draft_lens=k, context_lens=c, Hq=32, Hkv=8, D=128,
                                               V=128256, dtype="bf16", sigma=float(wl.sigma_for_alpha(0.7)),
                                               key=(7000 + B, kk), shuffle_blocks=False, extra_blocks=1)
            db = DeviceBatch.from_host(batch)
            for _ in range(3):
                db.step()
            t = {}
            for fn in ("step", "attention", "accept"):
                ms = _time_loop(getattr(db, fn), reps, flush, torch)
                t[fn] = float(np.median(ms))
            code, rid = db.device_status()
            if code != 0:
                raise RuntimeError(f"device status {code} at request {rid}")
            f = est.features(c, k)
            rows.append({"B": B, "k": kk, "sum_k": int(k.sum()), "N_linear": f[0], "N_interactions": f[1],
                         "N_cached": f[2], "t_step_ms": t["step"], "t_attention_ms": t["attention"],
                         "t_accept_ms": t["accept"]})
            print(json.dumps(rows[-1]), flush=True)
            del db
            torch.cuda.empty_cache()
    with open(path, "w", newline="") as fh:
        w = csv.DictWriter(fh, fieldnames=list(rows[0]))
        w.writeheader()
        w.writerows(rows)
    X = np.array([[r[n] for n in est.FEATURES] for r in rows])
    y = np.array([r["t_step_ms"] for r in rows]) * 1e-3
    fit = est.fit_with_validation(X, y)
    print(fit.report("s"), flush=True)


# --------------------------------------------------------------------------
# verification interference (Sec. 3): solo short, solo long, co-batched
# --------------------------------------------------------------------------
def interference(reps: int):
    """Step time of a short cached request B (500-token prefix, 5 drafts) alone, of a long request A
    (8 drafts over a growing prefix) alone, and of both in one batch, on the Llama-3-8B-shaped layer:
    the co-batched step is dictated by A, so B inherits A's latency."""
    import torch
    from paper_2601_11652_gb300 import build, workload as wl
    from paper_2601_11652_gb300.device_batch import DeviceBatch
    build.build()
    flush = torch.empty(FLUSH_BYTES, dtype=torch.uint8, device="cuda")

    def t_step(k, c, key):
        b = wl.make_batch_from_lengths(f"intf{key}", draft_lens=np.array(k, np.int32), context_lens=np.array(c, np.int32),
                                       Hq=32, Hkv=8, D=128, V=128256, dtype="bf16", sigma=float(wl.sigma_for_alpha(0.7)),
                                       key=(9100, key), shuffle_blocks=False, extra_blocks=1)
        db = DeviceBatch.from_host(b)
        for _ in range(3):
            db.step()
        ms = float(np.median(_time_loop(db.step, reps, flush, torch)))
        del db
        torch.cuda.empty_cache()
        return ms

    solo_b = t_step([5], [500], 0)
    for i, ca in enumerate((1000, 4000, 16000, 64000, 128000)):
        solo_a = t_step([8], [ca], 1 + i)
        both = t_step([8, 5], [ca, 500], 10 + i)
        print(json.dumps({"long_prefix": ca, "solo_short_ms": solo_b, "solo_long_ms": solo_a, "batched_ms": both,
                          "short_slowdown": both / solo_b}), flush=True)


def entry_only(args):
    """One entry point alone on one workload: warm-up calls, then timed calls (L2 flushed before
    each), median printed.  Used for single-kernel ncu captures on a small case."""
    import torch
    from paper_2601_11652_gb300 import build, workload as wl
    from paper_2601_11652_gb300.device_batch import DeviceBatch
    build.build()
    b = wl.make_batch(args.workload)
    # the acceptance pass reads no KV: a placeholder pool keeps the device footprint to its inputs
    pool = None
    if args.entry == "accept":
        dt = torch.bfloat16 if b.dtype == "bf16" else torch.float32
        pool = tuple(torch.zeros((1, b.Hkv, 16, b.D), dtype=dt, device="cuda") for _ in range(2))
    db = DeviceBatch.from_host(b, pool=pool)
    fn = getattr(db, args.entry)
    for _ in range(args.warmup):
        fn()
    torch.cuda.synchronize()
    flush = torch.empty(FLUSH_BYTES, dtype=torch.uint8, device="cuda")
    ms = _time_loop(fn, args.steps, flush, torch)
    code, rid = db.device_status()
    print(json.dumps({"entry": args.entry, "workload": args.workload, "calls": args.steps,
                      "ms_median": float(np.median(ms)), "device_status": [code, rid]}), flush=True)
    if code != 0:
        raise SystemExit(f"device status {code} (request {rid})")


def main():
    global SUSTAIN_S
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--workload", default=HEADLINE)
    ap.add_argument("--sustain-s", type=float, default=SUSTAIN_S,
                    help="seconds of device time per sustained / per-entry-point / end-to-end loop")
    ap.add_argument("--no-per-config", dest="per_config", action="store_false",
                    help="only the headline workload (no per_config object)")
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--latency-table", metavar="CSV", help="sweep batch size x draft length for the estimator "
                    "(Sec. 4.4) instead of the benchmark line; writes CSV and prints the fit")
    ap.add_argument("--lt-max-b", type=int, default=512)
    ap.add_argument("--lt-reps", type=int, default=20)
    ap.add_argument("--interference", action="store_true", help="solo / co-batched step times of a short and a long "
                    "request (Sec. 3) instead of the benchmark line")
    ap.add_argument("--entry", choices=["attention", "accept"],
                    help="call only this entry point, --warmup + --steps times on --workload, and print its "
                    "median time (a short run for single-kernel profiles) instead of the benchmark line")
    args = ap.parse_args()
    SUSTAIN_S = args.sustain_s
    if args.entry:
        entry_only(args)
        return
    if args.interference:
        interference(20)
        return
    if args.latency_table:
        latency_table(args.latency_table, args.lt_max_b, args.lt_reps)
        return
    rank = int(os.environ.get("RANK", 0))
    world = int(os.environ.get("WORLD_SIZE", 1))
    local_rank = int(os.environ.get("LOCAL_RANK", 0))
    from paper_2601_11652_gb300 import workload as wl

    if args.impl == "reference":
        if rank != 0:
            return
        run_reference(args, wl.make_batch(args.workload))
        return
    # each rank verifies its own copy of the batch (independent requests, no collective)
    run_ours(args, rank, world, local_rank)


if __name__ == "__main__":
    main()
