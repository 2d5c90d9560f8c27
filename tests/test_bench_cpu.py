"""CPU: the host-side arithmetic of bench.py -- algorithmic bytes, the per-kernel source hashes
that decide whether a committed ncu summary still describes the sources, the clock summary -- and
the reference arm's JSON line."""
import os
import shutil

import numpy as np

import bench
from paper_2601_11652_gb300 import workload as wl


def test_attention_bytes_counts_every_visible_token_once():
    b = wl.make_small_batch(3, B=4, Hq=8, Hkv=2, D=64, V=512, dtype="bf16", k_range=(0, 5), ctx_range=(0, 90))
    kv = qo = bt = 0
    for r in range(b.B):
        n = int(b.context_lens[r]) + int(b.draft_lens[r]) + 1
        kv += n * b.Hkv * b.D * 2 * 2          # K and V, bf16
        qo += (int(b.draft_lens[r]) + 1) * b.Hq * b.D * 2 * 2
        bt += -(-n // 16) * 4
    assert bench.attention_bytes(b) == kv + qo + bt


def test_accept_bytes_rows_up_to_the_rejection_and_one_draft_row():
    b = wl.make_small_batch(4, B=3, Hq=4, Hkv=4, D=64, V=1000, dtype="f32", k_range=(3, 3), ctx_range=(0, 10))
    L = [0, 3, 1]  # rejection at 0, all accepted, rejection at 1
    rows = (1 + 4 + 2) * 1000 * 4
    qrow = 2 * 1000 * 4
    decisions = 1 + 3 + 2
    assert bench.accept_bytes(b, L) == rows + qrow + decisions * 72 + 3 * 16


def _copy_sources(tmp_path):
    root = tmp_path / "repo"
    shutil.copytree(os.path.join(bench.ROOT, "paper_2601_11652_gb300", "csrc"),
                    root / "paper_2601_11652_gb300" / "csrc")
    return root


def test_kernel_sources_exist():
    csrc = os.path.join(bench.ROOT, "paper_2601_11652_gb300", "csrc")
    for kernel, files in bench.KERNEL_SOURCES.items():
        for f in files:
            assert os.path.isfile(os.path.join(csrc, f)), (kernel, f)


def test_kernel_hash_follows_only_its_own_sources(tmp_path, monkeypatch):
    root = _copy_sources(tmp_path)
    monkeypatch.setattr(bench, "ROOT", str(root))
    before = {k: bench._kernel_sha(k) for k in (None, "attention", "accept")}
    with open(root / "paper_2601_11652_gb300" / "csrc" / "accept.cu", "a") as f:
        f.write("\n// edit\n")
    after = {k: bench._kernel_sha(k) for k in (None, "attention", "accept")}
    assert after["attention"] == before["attention"]
    assert after["accept"] != before["accept"]
    assert after[None] != before[None]
    with open(root / "paper_2601_11652_gb300" / "csrc" / "common.cuh", "a") as f:
        f.write("\n// shared header\n")
    assert bench._kernel_sha("attention") != before["attention"]


def test_profile_traffic_only_while_the_sources_match(tmp_path, monkeypatch):
    root = _copy_sources(tmp_path)
    monkeypatch.setattr(bench, "ROOT", str(root))
    (root / "profiles").mkdir()
    prof = root / "profiles" / "accept_demo.md"
    prof.write_text(f"kernel_source_sha: {bench._kernel_sha('accept')}  (note)\n\ndram_bytes_per_launch: 12345\n")
    assert bench._profile_traffic("accept", "demo") == 12345.0
    assert bench._profile_traffic("attention", "demo") is None  # no such file
    with open(root / "paper_2601_11652_gb300" / "csrc" / "accept.cuh", "a") as f:
        f.write("\n")
    assert bench._profile_traffic("accept", "demo") is None


def test_clock_summary(tmp_path):
    p = tmp_path / "clocks.csv"
    na, act = "Not Active", "Active"
    lines = [f"0, {mhz}, 2070, 900.0, 0x0, {na}, {na}, {na}, {cap}" for mhz, cap in
             [(2070, na), (1980, act), (2010, na), (1500, na), (2070, na)]]
    p.write_text("\n".join(lines + ["garbage line", "0, [N/A], 2070, 1, 0x0, a, b, c, d"]) + "\n")
    s = bench.ClockSampler.summarise(str(p))
    assert s == {"sm_mhz": 2010.0, "sm_max_mhz": 2070.0, "reasons": ["sw_power_cap"], "samples": 5}
    empty = tmp_path / "empty.csv"
    empty.write_text("")
    assert bench.ClockSampler.summarise(str(empty)) is None
    assert np.isfinite(s["sm_mhz"])


def test_issue_roofline_from_the_profile(tmp_path, monkeypatch):
    root = _copy_sources(tmp_path)
    monkeypatch.setattr(bench, "ROOT", str(root))
    (root / "profiles").mkdir()
    prof = root / "profiles" / "accept_demo.md"
    prof.write_text(f"kernel_source_sha: {bench._kernel_sha('accept')}\n\n"
                    "| smsp__inst_executed.sum | 1000000.000000 inst |\n"
                    "| smsp__inst_executed.sum | 3000000.000000 inst |\n")
    w = bench._profile_inst("accept", "demo")
    assert w == 4.0e6
    r = bench.issue_roofline(w, 0.01, 100, 2000.0)  # 4e6 warp instructions in 10 us on 100 SMs at 2 GHz
    assert abs(r["achieved"] - 400.0) < 1e-9 and abs(r["peak"] - 800.0) < 1e-9 and abs(r["frac"] - 0.5) < 1e-12
    assert bench.issue_roofline(None, 0.01, 100, 2000.0) is None
    assert bench.issue_roofline(w, 0.01, 100, None) is None
    with open(root / "paper_2601_11652_gb300" / "csrc" / "accept.cu", "a") as f:
        f.write("\n")
    assert bench._profile_inst("accept", "demo") is None


def test_reference_arm_prints_the_contract_line():
    """bench.py --impl reference: the oracle timed on the host cores on the workload's requests,
    one JSON line with the reference keys (here the small fp32 workload, one short step)."""
    import json
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    out = subprocess.run([sys.executable, os.path.join(root, "bench.py"), "--impl", "reference", "--workload",
                          "tiny_f32", "--steps", "1", "--warmup", "0"], capture_output=True, text=True, timeout=300,
                         cwd=root)
    assert out.returncode == 0, out.stderr[-2000:]
    line = json.loads(out.stdout.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["steps"] == 1 and line["value"] > 0
    assert line["unit"] == "verified_tokens/s" and line["higher_is_better"] is True
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["cores"] >= 1
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["e2e"]["d2h_bytes_per_step"] == 0
    assert line["config"]["workload"] == "tiny_f32"
