"""A verification batch resident on the GPU, wired to the C ABI.

`DeviceBatch.from_host(batch)` copies a host batch (numpy arrays, the layout of
include/wisp_verify.h) into torch device tensors once, allocates the outputs
and a caller-owned workspace, and fills the two argument structs.  `step()`,
`attention()` and `accept()` only enqueue the library's kernels.
"""
from __future__ import annotations

import numpy as np
import torch

from . import binding as wb


def _to_dev(a: np.ndarray, device, dtype_name: str | None = None) -> torch.Tensor:
    if dtype_name == "bf16":
        t = torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16)
    else:
        t = torch.from_numpy(np.ascontiguousarray(a))
    return t.to(device, non_blocking=False)


class DeviceBatch:
    def __init__(self):
        self.t = {}

    @classmethod
    def from_host(cls, b, device="cuda", pool=None) -> "DeviceBatch":
        """`pool` = (k_cache, v_cache) device tensors to reuse instead of copying the host pool."""
        self = cls()
        t = self.t
        self.B, self.V, self.Hq, self.D = b.B, b.V, b.Hq, b.D
        t["request_ids"] = _to_dev(b.request_ids.astype(np.int64), device)
        t["draft_lens"] = _to_dev(b.draft_lens.astype(np.int32), device)
        t["context_lens"] = _to_dev(b.context_lens.astype(np.int32), device)
        t["block_tables"] = _to_dev(b.block_tables.astype(np.int32), device)
        t["q"] = _to_dev(b.q, device, b.dtype)
        if pool is None:
            t["k_cache"] = _to_dev(b.k_cache, device, b.dtype)
            t["v_cache"] = _to_dev(b.v_cache, device, b.dtype)
        else:
            t["k_cache"], t["v_cache"] = pool
        t["logits"] = _to_dev(b.logits, device, b.dtype)
        t["draft_tokens"] = _to_dev(b.draft_tokens.astype(np.int32), device)
        t["draft_probs"] = _to_dev(b.draft_probs.astype(np.float32), device)
        t["accept_u"] = _to_dev(b.accept_uniforms.astype(np.float32), device)
        t["sample_u"] = _to_dev(b.sample_uniforms.astype(np.float32), device)
        t["out"] = torch.empty_like(t["q"])
        t["accepted_len"] = torch.full((b.B,), -7, dtype=torch.int32, device=device)
        t["next_token"] = torch.full((b.B,), -7, dtype=torch.int32, device=device)
        self.num_blocks = int(b.num_blocks)
        self._make_args()
        n = wb.wisp_verify_workspace_size(self.attn_args, self.accept_args)
        t["workspace"] = wb.alloc_workspace(n, device)
        return self

    def _make_args(self):
        t = self.t
        self.attn_args = wb.make_attn_args(
            draft_lens=t["draft_lens"], context_lens=t["context_lens"], block_tables=t["block_tables"],
            q=t["q"], k_cache=t["k_cache"], v_cache=t["v_cache"], out=t["out"], request_ids=t["request_ids"],
            num_blocks=self.num_blocks)
        self.accept_args = wb.make_accept_args(
            draft_lens=t["draft_lens"], target_logits=t["logits"], draft_tokens=t["draft_tokens"],
            draft_probs=t["draft_probs"], accept_uniforms=t["accept_u"], sample_uniforms=t["sample_u"],
            accepted_len=t["accepted_len"], next_token=t["next_token"], request_ids=t["request_ids"])

    @property
    def workspace(self) -> torch.Tensor:
        return self.t["workspace"]

    def step(self, stream=None):
        wb.wisp_verify_step(self.attn_args, self.accept_args, self.workspace, stream)

    def attention(self, stream=None):
        wb.wisp_verify_attention(self.attn_args, self.workspace, stream)

    def accept(self, stream=None):
        wb.wisp_verify_accept(self.accept_args, self.workspace, stream)

    def device_status(self):
        return wb.wisp_verify_get_device_status(self.workspace)

    def results(self) -> dict:
        t = self.t
        out = t["out"].float().cpu().numpy()
        return {"out": out, "accepted_len": t["accepted_len"].cpu().numpy(),
                "next_token": t["next_token"].cpu().numpy()}
