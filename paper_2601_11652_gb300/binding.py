"""ctypes binding of libwisp_verify.so (include/wisp_verify.h): argument marshalling only.

Every entry point of the C ABI has a Python function of the same name here.
Arguments are torch CUDA tensors (their data_ptr() is passed) or plain ints;
streams default to torch's current stream.  There is no CPU path: importing
this module without the built library, or calling it without a CUDA device,
raises.
"""
from __future__ import annotations

import ctypes
import os

import torch

from . import build as _build

WISP_OK, WISP_ERR_INVALID_ARG, WISP_ERR_UNSUPPORTED, WISP_ERR_CUDA, WISP_ERR_WORKSPACE = range(5)
WISP_F32, WISP_BF16 = 0, 1
DEVICE_CODES = {0: "ok", 1: "bad_length", 2: "bad_block", 3: "bad_token", 4: "bad_prob", 5: "unsupported",
                6: "timeout"}

_P = ctypes.c_void_p
_I32 = ctypes.c_int32


class wisp_attn_args(ctypes.Structure):
    _fields_ = [("B", _I32), ("Hq", _I32), ("Hkv", _I32), ("D", _I32), ("block_size", _I32),
                ("max_blocks_per_seq", _I32), ("num_blocks", _I32), ("total_q_rows", _I32),
                ("request_ids", _P), ("draft_lens", _P), ("context_lens", _P), ("block_tables", _P),
                ("qkv_dtype", ctypes.c_int), ("q", _P), ("k_cache", _P), ("v_cache", _P), ("out", _P)]


class wisp_accept_args(ctypes.Structure):
    _fields_ = [("B", _I32), ("V", _I32), ("total_q_rows", _I32), ("total_draft", _I32),
                ("request_ids", _P), ("draft_lens", _P), ("logits_dtype", ctypes.c_int),
                ("target_logits", _P), ("draft_tokens", _P), ("draft_probs", _P), ("accept_uniforms", _P),
                ("sample_uniforms", _P), ("accepted_len", _P), ("next_token", _P)]


class wisp_kv_args(ctypes.Structure):
    _fields_ = [("B", _I32), ("Hkv", _I32), ("D", _I32), ("block_size", _I32), ("max_blocks_per_seq", _I32),
                ("num_blocks", _I32), ("total_q_rows", _I32), ("request_ids", _P), ("draft_lens", _P),
                ("context_lens", _P), ("block_tables", _P), ("free_blocks", _P), ("free_count", _P),
                ("kv_dtype", ctypes.c_int), ("k_cache", _P), ("v_cache", _P), ("k_new", _P), ("v_new", _P),
                ("accepted_len", _P)]


class WispError(RuntimeError):
    def __init__(self, fn: str, code: int, text: str):
        super().__init__(f"{fn}: {text} (status {code})")
        self.code = code


_lib = None

EXPORTED = ["wisp_verify_workspace_size", "wisp_verify_attention", "wisp_verify_accept", "wisp_verify_step",
            "wisp_verify_get_device_status", "wisp_verify_status_string", "wisp_verify_device_code_string",
            "wisp_verify_accept_noalloc", "wisp_verify_accept_greedy", "wisp_kv_workspace_size",
            "wisp_kv_reserve_append", "wisp_kv_commit"]


def lib_path() -> str:
    return _build.LIB_PATH


def load(path: str | None = None):
    """Load the shared library (built in-tree by build.py); raises if it is missing."""
    global _lib
    if _lib is not None:
        return _lib
    path = path or lib_path()
    if not os.path.exists(path):
        raise RuntimeError(f"{path} is missing: build it with `python -m paper_2601_11652_gb300.build` "
                           "(the verification step has no CPU implementation)")
    lib = ctypes.CDLL(path)
    AP, CP = ctypes.POINTER(wisp_attn_args), ctypes.POINTER(wisp_accept_args)
    lib.wisp_verify_workspace_size.argtypes = [AP, CP]
    lib.wisp_verify_workspace_size.restype = ctypes.c_size_t
    lib.wisp_verify_attention.argtypes = [AP, _P, ctypes.c_size_t, _P]
    lib.wisp_verify_attention.restype = ctypes.c_int
    lib.wisp_verify_accept.argtypes = [CP, _P, ctypes.c_size_t, _P]
    lib.wisp_verify_accept.restype = ctypes.c_int
    lib.wisp_verify_step.argtypes = [AP, CP, _P, ctypes.c_size_t, _P]
    lib.wisp_verify_step.restype = ctypes.c_int
    lib.wisp_verify_accept_greedy.argtypes = [CP, _P, ctypes.c_size_t, _P]
    lib.wisp_verify_accept_greedy.restype = ctypes.c_int
    lib.wisp_verify_accept_noalloc.argtypes = [CP, _P]
    lib.wisp_verify_accept_noalloc.restype = ctypes.c_int
    lib.wisp_verify_get_device_status.argtypes = [_P, ctypes.POINTER(_I32), ctypes.POINTER(ctypes.c_int64)]
    lib.wisp_verify_get_device_status.restype = ctypes.c_int
    lib.wisp_verify_status_string.argtypes = [ctypes.c_int]
    lib.wisp_verify_status_string.restype = ctypes.c_char_p
    lib.wisp_verify_device_code_string.argtypes = [_I32]
    lib.wisp_verify_device_code_string.restype = ctypes.c_char_p
    KP = ctypes.POINTER(wisp_kv_args)
    lib.wisp_kv_workspace_size.argtypes = [KP]
    lib.wisp_kv_workspace_size.restype = ctypes.c_size_t
    for fn in ("wisp_kv_reserve_append", "wisp_kv_commit"):
        getattr(lib, fn).argtypes = [KP, _P, ctypes.c_size_t, _P]
        getattr(lib, fn).restype = ctypes.c_int
    _lib = lib
    return lib


def _check(fn: str, code: int):
    if code != WISP_OK:
        raise WispError(fn, code, load().wisp_verify_status_string(code).decode())


def _ptr(t) -> int | None:
    if t is None:
        return None
    if isinstance(t, int):
        return t
    if not t.is_cuda:
        raise ValueError("device tensors only: the verification step runs on the GPU")
    if not t.is_contiguous():
        raise ValueError("tensors must be contiguous")
    return t.data_ptr()


def _stream(stream) -> int | None:
    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else stream


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.float32:
        return WISP_F32
    if t.dtype == torch.bfloat16:
        return WISP_BF16
    raise ValueError(f"unsupported dtype {t.dtype}")


def make_attn_args(*, draft_lens, context_lens, block_tables, q, k_cache, v_cache, out, request_ids=None,
                   num_blocks=None, total_q_rows=None) -> wisp_attn_args:
    """Fill wisp_attn_args from device tensors (shapes as in include/wisp_verify.h)."""
    B = draft_lens.shape[0]
    T_q, Hq, D = q.shape
    nb, Hkv, bs, D2 = k_cache.shape
    assert D2 == D and v_cache.shape == k_cache.shape and out.shape == q.shape and out.dtype == q.dtype
    a = wisp_attn_args()
    a.B, a.Hq, a.Hkv, a.D, a.block_size = B, Hq, Hkv, D, bs
    a.max_blocks_per_seq = block_tables.shape[1] if block_tables.dim() == 2 else 0
    a.num_blocks = nb if num_blocks is None else num_blocks
    a.total_q_rows = T_q if total_q_rows is None else total_q_rows
    a.request_ids, a.draft_lens, a.context_lens = _ptr(request_ids), _ptr(draft_lens), _ptr(context_lens)
    a.block_tables = _ptr(block_tables)
    a.qkv_dtype = _dtype_code(q)
    a.q, a.k_cache, a.v_cache, a.out = _ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(out)
    return a


def make_accept_args(*, draft_lens, target_logits, draft_tokens, draft_probs, accept_uniforms,
                     sample_uniforms, accepted_len, next_token, request_ids=None, total_q_rows=None,
                     total_draft=None) -> wisp_accept_args:
    """Fill wisp_accept_args from device tensors (shapes as in include/wisp_verify.h)."""
    c = wisp_accept_args()
    c.B = draft_lens.shape[0]
    c.V = target_logits.shape[1]
    c.total_q_rows = target_logits.shape[0] if total_q_rows is None else total_q_rows
    c.total_draft = draft_tokens.shape[0] if total_draft is None else total_draft
    c.request_ids, c.draft_lens = _ptr(request_ids), _ptr(draft_lens)
    c.logits_dtype = _dtype_code(target_logits)
    c.target_logits = _ptr(target_logits)
    c.draft_tokens = _ptr(draft_tokens) if draft_tokens.numel() else None
    c.draft_probs = _ptr(draft_probs) if draft_probs.numel() else None
    c.accept_uniforms = _ptr(accept_uniforms) if accept_uniforms.numel() else None
    c.sample_uniforms, c.accepted_len, c.next_token = _ptr(sample_uniforms), _ptr(accepted_len), _ptr(next_token)
    return c


def wisp_verify_workspace_size(attn: wisp_attn_args | None, acc: wisp_accept_args | None) -> int:
    n = load().wisp_verify_workspace_size(ctypes.byref(attn) if attn else None, ctypes.byref(acc) if acc else None)
    if n == 0:
        raise WispError("wisp_verify_workspace_size", WISP_ERR_INVALID_ARG, "invalid arguments")
    return int(n)


def alloc_workspace(nbytes: int, device=None) -> torch.Tensor:
    """Caller-owned workspace (torch allocates; the library never does). 256-byte aligned."""
    t = torch.empty(nbytes + 256, dtype=torch.uint8, device=device or "cuda")
    off = (-t.data_ptr()) % 256
    return t[off: off + nbytes]


def wisp_verify_attention(attn: wisp_attn_args, workspace: torch.Tensor, stream=None) -> None:
    _check("wisp_verify_attention", load().wisp_verify_attention(
        ctypes.byref(attn), _ptr(workspace), workspace.numel(), _stream(stream)))


def wisp_verify_accept(acc: wisp_accept_args, workspace: torch.Tensor, stream=None) -> None:
    _check("wisp_verify_accept", load().wisp_verify_accept(
        ctypes.byref(acc), _ptr(workspace), workspace.numel(), _stream(stream)))


def wisp_verify_accept_greedy(acc: wisp_accept_args, workspace: torch.Tensor, stream=None) -> None:
    _check("wisp_verify_accept_greedy", load().wisp_verify_accept_greedy(
        ctypes.byref(acc), _ptr(workspace), workspace.numel(), _stream(stream)))


def wisp_verify_accept_noalloc(acc: wisp_accept_args, stream=None) -> None:
    _check("wisp_verify_accept_noalloc", load().wisp_verify_accept_noalloc(ctypes.byref(acc), _stream(stream)))


def wisp_verify_step(attn: wisp_attn_args, acc: wisp_accept_args, workspace: torch.Tensor, stream=None) -> None:
    _check("wisp_verify_step", load().wisp_verify_step(
        ctypes.byref(attn), ctypes.byref(acc), _ptr(workspace), workspace.numel(), _stream(stream)))


def wisp_verify_get_device_status(workspace: torch.Tensor) -> tuple[int, int]:
    code, rid = _I32(0), ctypes.c_int64(0)
    _check("wisp_verify_get_device_status",
           load().wisp_verify_get_device_status(_ptr(workspace), ctypes.byref(code), ctypes.byref(rid)))
    return int(code.value), int(rid.value)


# ---- paged KV maintenance (include/wisp_kv.h) ---------------------------------------------------
def make_kv_args(*, draft_lens, context_lens, block_tables, free_blocks, free_count, k_cache=None, v_cache=None,
                 k_new=None, v_new=None, accepted_len=None, request_ids=None, total_q_rows=None) -> wisp_kv_args:
    """Fill wisp_kv_args from device tensors (k_cache / v_cache [num_blocks, Hkv, 16, D])."""
    a = wisp_kv_args()
    a.B = draft_lens.shape[0]
    a.max_blocks_per_seq = block_tables.shape[1]
    a.num_blocks = free_blocks.shape[0]
    ref = k_cache if k_cache is not None else k_new
    a.Hkv = ref.shape[1] if ref is not None else 1
    a.D = ref.shape[-1] if ref is not None else 128
    a.block_size = 16
    a.total_q_rows = int(draft_lens.sum().item()) + a.B if total_q_rows is None else total_q_rows
    a.request_ids, a.draft_lens, a.context_lens = _ptr(request_ids), _ptr(draft_lens), _ptr(context_lens)
    a.block_tables, a.free_blocks, a.free_count = _ptr(block_tables), _ptr(free_blocks), _ptr(free_count)
    a.kv_dtype = _dtype_code(ref) if ref is not None else WISP_BF16
    a.k_cache, a.v_cache, a.k_new, a.v_new = _ptr(k_cache), _ptr(v_cache), _ptr(k_new), _ptr(v_new)
    a.accepted_len = _ptr(accepted_len)
    return a


def wisp_kv_workspace_size(kv: wisp_kv_args) -> int:
    n = load().wisp_kv_workspace_size(ctypes.byref(kv))
    if n == 0:
        raise WispError("wisp_kv_workspace_size", WISP_ERR_INVALID_ARG, "invalid arguments")
    return int(n)


def wisp_kv_reserve_append(kv: wisp_kv_args, workspace: torch.Tensor, stream=None) -> None:
    _check("wisp_kv_reserve_append", load().wisp_kv_reserve_append(
        ctypes.byref(kv), _ptr(workspace), workspace.numel(), _stream(stream)))


def wisp_kv_commit(kv: wisp_kv_args, workspace: torch.Tensor, stream=None) -> None:
    _check("wisp_kv_commit", load().wisp_kv_commit(ctypes.byref(kv), _ptr(workspace), workspace.numel(), _stream(stream)))
