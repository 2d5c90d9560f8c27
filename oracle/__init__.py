"""fp64 CPU oracle of the WISP verification step -- TEST INFRASTRUCTURE ONLY.

Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline / reference
legs may import this package.  It compiles oracle.c with the host C compiler
(no CUDA, no code shared with the GPU library) and exposes:

  attention(batch)  -> float64 [T_q, Hq, D]   (Sec. 4.4-4.5 attention over L_total keys)
  accept(batch)     -> dict of per-request arrays (Eq. 1-3 acceptance + target token)
  row_softmax(row)  -> float64 [V]

`batch` is any object with the attributes of a verification batch (B, Hq, Hkv,
D, V, block_size, dtype, draft_lens, context_lens, block_tables, num_blocks,
q, k_cache, v_cache, logits, draft_tokens, draft_probs, accept_uniforms,
sample_uniforms).  Every function is pinned by tests/test_oracle_attention.py and
tests/test_oracle_accept.py (library routines, closed forms, hand-worked
examples, invariants, exact enumeration, chi-square); none is parity-unpinned.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_OUT_DIR = os.path.join(_HERE, "_build")
_LIB = os.path.join(_OUT_DIR, "liboracle.so")
_lock = threading.Lock()
_lib = None

F32, BF16 = 0, 1
STATUS_NAMES = {0: "ok", 1: "bad_arg", 2: "bad_length", 3: "bad_block", 4: "bad_token", 5: "bad_prob"}


def build(force: bool = False) -> str:
    """Compile oracle.c into a shared library (plain gcc, OpenMP)."""
    os.makedirs(_OUT_DIR, exist_ok=True)
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        cmd = ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fopenmp", "-fPIC", "-shared",
               _SRC, "-o", tmp, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            P = ctypes.c_void_p
            I = ctypes.c_int
            lib.oracle_attention.argtypes = [I, I, I, I, I, I, I, P, P, P, I, P, P, P, P, I]
            lib.oracle_attention.restype = I
            lib.oracle_accept.argtypes = [I, I, P, I, P, P, P, P, P, P, P, P, P, P, I]
            lib.oracle_accept.restype = I
            lib.oracle_row_softmax.argtypes = [I, I, P, P]
            lib.oracle_row_softmax.restype = None
            _lib = lib
    return _lib


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def _dtype_code(dtype: str) -> int:
    return {"f32": F32, "bf16": BF16}[dtype]


def default_threads() -> int:
    return os.cpu_count() or 1


def attention(batch, nthreads: int | None = None) -> np.ndarray:
    lib = _load()
    dl = np.ascontiguousarray(batch.draft_lens, dtype=np.int32)
    cl = np.ascontiguousarray(batch.context_lens, dtype=np.int32)
    bt = np.ascontiguousarray(batch.block_tables, dtype=np.int32)
    q = np.ascontiguousarray(batch.q)
    kc = np.ascontiguousarray(batch.k_cache)
    vc = np.ascontiguousarray(batch.v_cache)
    T_q = int(dl.sum()) + len(dl)
    out = np.zeros((T_q, batch.Hq, batch.D), dtype=np.float64)
    rc = lib.oracle_attention(len(dl), batch.Hq, batch.Hkv, batch.D, batch.block_size, bt.shape[1],
                              int(batch.num_blocks), _ptr(dl), _ptr(cl), _ptr(bt),
                              _dtype_code(batch.dtype), _ptr(q), _ptr(kc), _ptr(vc), _ptr(out),
                              nthreads or default_threads())
    if rc != 0:
        raise ValueError(f"oracle_attention rejected its input: {STATUS_NAMES.get(rc, rc)}")
    return out


def accept(batch, nthreads: int | None = None, check: bool = True) -> dict:
    lib = _load()
    B = len(batch.draft_lens)
    dl = np.ascontiguousarray(batch.draft_lens, dtype=np.int32)
    logits = np.ascontiguousarray(batch.logits)
    toks = np.ascontiguousarray(batch.draft_tokens, dtype=np.int32)
    probs = np.ascontiguousarray(batch.draft_probs, dtype=np.float32)
    au = np.ascontiguousarray(batch.accept_uniforms, dtype=np.float32)
    su = np.ascontiguousarray(batch.sample_uniforms, dtype=np.float32)
    L = np.empty(B, np.int32)
    tok = np.empty(B, np.int32)
    am = np.empty(B, np.float64)
    sm = np.empty(B, np.float64)
    st = np.empty(B, np.int32)
    rc = lib.oracle_accept(B, int(batch.V), _ptr(dl), _dtype_code(batch.dtype), _ptr(logits), _ptr(toks),
                           _ptr(probs), _ptr(au), _ptr(su), _ptr(L), _ptr(tok), _ptr(am), _ptr(sm),
                           _ptr(st), nthreads or default_threads())
    if check and rc != 0:
        raise ValueError(f"oracle_accept rejected its input: {STATUS_NAMES.get(rc, rc)}")
    return {"accepted_len": L, "next_token": tok, "accept_margin": am, "sample_margin": sm, "status": st}


def row_softmax(row: np.ndarray, dtype: str = "f32") -> np.ndarray:
    lib = _load()
    row = np.ascontiguousarray(row)
    p = np.empty(row.shape[-1], dtype=np.float64)
    lib.oracle_row_softmax(row.shape[-1], _dtype_code(dtype), _ptr(row), _ptr(p))
    return p


def accept_greedy(batch) -> dict:
    """Temperature-0 variant of the acceptance rule, written out with numpy (test infrastructure).

    Sampling at temperature 0 takes the most likely token: draft token i is accepted iff it equals
    the argmax of logit row i-1 (np.argmax: the lowest index among equal maxima), the walk stops at
    the first mismatch (Eq. 2) and the extra token is the argmax of row L.  NaN logits are never
    chosen; a row without a finite logit gives status 5 (bad_prob) and L = token = -1.
    """
    B = len(batch.draft_lens)
    V = int(batch.V)
    if batch.dtype == "bf16":
        z = (np.asarray(batch.logits, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)
    else:
        z = np.asarray(batch.logits, dtype=np.float32)
    z = z.reshape(-1, V).astype(np.float64)
    z = np.where(np.isnan(z), -np.inf, z)
    L = np.empty(B, np.int32)
    tok = np.empty(B, np.int32)
    st = np.zeros(B, np.int32)
    row0 = 0
    d0 = 0
    for r in range(B):
        k = int(batch.draft_lens[r])
        L[r], tok[r] = k, -1
        for i in range(k + 1):
            row = z[row0 + i]
            if not np.isfinite(row.max()):
                st[r], L[r], tok[r] = 5, -1, -1
                break
            a = int(np.argmax(row))
            if i == k:
                tok[r] = a
                break
            if int(batch.draft_tokens[d0 + i]) != a:
                L[r], tok[r] = i, a
                break
        row0 += k + 1
        d0 += k
    return {"accepted_len": L, "next_token": tok, "status": st}
