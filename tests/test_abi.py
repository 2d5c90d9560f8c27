"""The C ABI without a GPU: the library builds, loads, exports every declared entry
point, and rejects host-visible bad arguments before touching the device."""
import ctypes
import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "wisp_verify.h")
HEADERS = [HEADER, os.path.join(ROOT, "include", "wisp_kv.h")]


@pytest.fixture(scope="module")
def lib():
    from paper_2601_11652_gb300 import binding, build
    build.build()
    return binding.load()


def declared_functions():
    names = set()
    for h in HEADERS:
        text = re.sub(r"/\*.*?\*/", "", open(h).read(), flags=re.S)
        names |= set(re.findall(r"\b(wisp_(?:verify|kv)_\w+)\s*\(", text))
    return sorted(names)


def test_header_declares_the_abi():
    names = declared_functions()
    for n in ["wisp_verify_attention", "wisp_verify_accept", "wisp_verify_step", "wisp_verify_workspace_size",
              "wisp_verify_get_device_status"]:
        assert n in names


def test_library_exports_every_declared_symbol(lib):
    from paper_2601_11652_gb300 import binding
    out = subprocess.run(["nm", "-D", "--defined-only", binding.lib_path()], capture_output=True, text=True,
                         check=True).stdout
    exported = set(re.findall(r"\sT\s(\w+)", out))
    for n in declared_functions():
        assert n in exported, n
        assert hasattr(lib, n)


def test_header_compiles_as_c(tmp_path):
    src = tmp_path / "t.c"
    src.write_text('#include "wisp_verify.h"\n#include "wisp_kv.h"\n'
                   'int main(void){ return (int)(sizeof(wisp_attn_args) + sizeof(wisp_kv_args)) > 0 ? 0 : 1; }\n')
    subprocess.run(["gcc", "-std=c99", "-Wall", "-Werror", "-I", os.path.join(ROOT, "include"), "-c", str(src),
                    "-o", str(tmp_path / "t.o")], check=True)


def _attn(**kw):
    from paper_2601_11652_gb300 import binding as wb
    a = wb.wisp_attn_args()
    base = dict(B=2, Hq=8, Hkv=2, D=128, block_size=16, max_blocks_per_seq=4, num_blocks=8, total_q_rows=4,
                request_ids=None, draft_lens=0x1000, context_lens=0x2000, block_tables=0x3000, qkv_dtype=1,
                q=0x10000, k_cache=0x20000, v_cache=0x30000, out=0x40000)
    base.update(kw)
    for k, v in base.items():
        setattr(a, k, v)
    return a


def _acc(**kw):
    from paper_2601_11652_gb300 import binding as wb
    c = wb.wisp_accept_args()
    base = dict(B=2, V=1000, total_q_rows=4, total_draft=2, request_ids=None, draft_lens=0x1000, logits_dtype=0,
                target_logits=0x10000, draft_tokens=0x2000, draft_probs=0x20000, accept_uniforms=0x3000,
                sample_uniforms=0x4000, accepted_len=0x5000, next_token=0x6000)
    base.update(kw)
    for k, v in base.items():
        setattr(c, k, v)
    return c


BAD_ATTN = [dict(B=-1), dict(Hq=0), dict(Hq=6, Hkv=4), dict(D=96), dict(block_size=32), dict(draft_lens=None),
            dict(q=None), dict(out=0x40004), dict(qkv_dtype=7), dict(total_q_rows=1), dict(num_blocks=0),
            dict(max_blocks_per_seq=0)]
BAD_ACC = [dict(B=-2), dict(V=0), dict(total_draft=-1), dict(target_logits=None), dict(draft_probs=None),
           dict(logits_dtype=3), dict(total_q_rows=1), dict(V=(1 << 24) + 1), dict(next_token=None)]


@pytest.mark.parametrize("kw", BAD_ATTN, ids=[str(k) for k in BAD_ATTN])
def test_attention_rejects_bad_arguments(lib, kw):
    from paper_2601_11652_gb300 import binding as wb
    a = _attn(**kw)
    rc = lib.wisp_verify_attention(ctypes.byref(a), ctypes.c_void_p(0x100000), 1 << 30, None)
    assert rc in (wb.WISP_ERR_INVALID_ARG, wb.WISP_ERR_UNSUPPORTED)
    assert lib.wisp_verify_workspace_size(ctypes.byref(a), None) == 0


@pytest.mark.parametrize("kw", BAD_ACC, ids=[str(k) for k in BAD_ACC])
def test_accept_rejects_bad_arguments(lib, kw):
    from paper_2601_11652_gb300 import binding as wb
    c = _acc(**kw)
    rc = lib.wisp_verify_accept(ctypes.byref(c), ctypes.c_void_p(0x100000), 1 << 30, None)
    assert rc in (wb.WISP_ERR_INVALID_ARG, wb.WISP_ERR_UNSUPPORTED)


@pytest.mark.parametrize("kw", BAD_ACC + [dict(B=8193, total_q_rows=8193, total_draft=0),
                                           dict(B=100, total_q_rows=131073, total_draft=0)],
                         ids=[str(k) for k in BAD_ACC] + ["B=8193", "rows=131073"])
def test_accept_noalloc_rejects_bad_arguments(lib, kw):
    # checked on the host before any device call; a batch beyond the fixed scratch is unsupported
    from paper_2601_11652_gb300 import binding as wb
    c = _acc(**kw)
    rc = lib.wisp_verify_accept_noalloc(ctypes.byref(c), None)
    assert rc in (wb.WISP_ERR_INVALID_ARG, wb.WISP_ERR_UNSUPPORTED)
    if kw.get("B") == 8193 or kw.get("total_q_rows") == 131073:
        assert rc == wb.WISP_ERR_UNSUPPORTED


def test_step_rejects_mismatched_batches(lib):
    from paper_2601_11652_gb300 import binding as wb
    rc = lib.wisp_verify_step(ctypes.byref(_attn()), ctypes.byref(_acc(B=3, total_q_rows=5)),
                              ctypes.c_void_p(0x100000), 1 << 30, None)
    assert rc == wb.WISP_ERR_INVALID_ARG


def test_status_strings(lib):
    for code in range(5):
        assert lib.wisp_verify_status_string(code)
    for code in range(8):
        assert lib.wisp_verify_device_code_string(code) != b"unknown device code"
    assert lib.wisp_verify_get_device_status(None, None, None) == 1
