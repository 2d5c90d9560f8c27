"""The acceptance kernels' certified error bound assumes that the hardware ex2.approx.ftz.f32
has a relative error below kEx2RelErr (csrc/common.cuh) for every argument in [-126, 0].  This
test measures the largest error exhaustively on the GPU (tests/probes/ex2_error.cu) and checks
the assumption."""
import ctypes
import os
import re
import subprocess

import pytest
import torch

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _assumed_bound() -> float:
    text = open(os.path.join(ROOT, "paper_2601_11652_gb300", "csrc", "common.cuh")).read()
    m = re.search(r"constexpr float kEx2RelErr = 0x1p-(\d+)f;", text)
    assert m, "kEx2RelErr not found"
    return 2.0 ** -int(m.group(1))


def test_ex2_relative_error_below_assumed_bound(tmp_path):
    if not torch.cuda.is_available():
        pytest.fail("GPU tests need a CUDA device")
    so = tmp_path / "ex2probe.so"
    subprocess.run(["nvcc", "-gencode", "arch=compute_103a,code=sm_103a", "-O3", "-Xcompiler", "-fPIC", "-shared",
                    os.path.join(ROOT, "tests", "probes", "ex2_error.cu"), "-o", str(so)], check=True)
    lib = ctypes.CDLL(str(so))
    out = ctypes.c_float()
    assert lib.ex2_max_rel_error(ctypes.byref(out)) == 0
    assert 0.0 < out.value <= _assumed_bound(), f"measured {out.value}, assumed {_assumed_bound()}"
