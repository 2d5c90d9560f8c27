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
    def from_tensors(cls, t: dict, num_blocks: int, device="cuda") -> "DeviceBatch":
        """Wire existing device tensors (the names of `from_host`; outputs included) to the C ABI
        and allocate the workspace."""
        self = cls()
        self.t = t
        self.B, self.V = int(t["draft_lens"].numel()), int(t["logits"].shape[1])
        self.Hq, self.D = int(t["q"].shape[1]), int(t["q"].shape[2])
        self.num_blocks = int(num_blocks)
        self._make_args()
        n = wb.wisp_verify_workspace_size(self.attn_args, self.accept_args)
        t["workspace"] = wb.alloc_workspace(n, device)
        return self

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


# per-step inputs of a verification step (everything but the resident paged KV cache), in the
# order they are packed into one contiguous staging buffer
STEP_INPUTS = ("request_ids", "draft_lens", "context_lens", "block_tables", "q", "logits", "draft_tokens",
               "draft_probs", "accept_u", "sample_u")


def _host_inputs(b) -> dict:
    """The per-step inputs of host batch `b` as numpy arrays in the C ABI's dtypes (bf16 as uint16)."""
    return {"request_ids": b.request_ids.astype(np.int64), "draft_lens": b.draft_lens.astype(np.int32),
            "context_lens": b.context_lens.astype(np.int32), "block_tables": b.block_tables.astype(np.int32),
            "q": b.q, "logits": b.logits, "draft_tokens": b.draft_tokens.astype(np.int32),
            "draft_probs": b.draft_probs.astype(np.float32), "accept_u": b.accept_uniforms.astype(np.float32),
            "sample_u": b.sample_uniforms.astype(np.float32)}


class StagedSteps:
    """Verification steps fed from host memory: every step's inputs are copied from ONE contiguous
    pinned staging buffer into one of `depth` device buffers of the same layout (one host-to-device
    copy per step, on a copy stream), the step runs on the compute stream, and the two results
    (accepted_len, next_token; contiguous) come back in one device-to-host copy.  The copy of step
    n + 1 overlaps step n; a device buffer is refilled only after the step that read it is done.
    The paged KV cache stays resident (it is the prefix cache, not a per-step input)."""

    def __init__(self, b, device="cuda", depth: int = 2, pool=None):
        dev = torch.device(device)
        host = _host_inputs(b)
        self.layout, off = {}, 0
        for n in STEP_INPUTS:
            a = np.ascontiguousarray(host[n])
            self.layout[n] = (off, a.nbytes, a.shape, a.dtype)
            off = (off + a.nbytes + 255) // 256 * 256
        self.nbytes = off
        self.h2d_bytes = sum(v[1] for v in self.layout.values())
        self.host = torch.empty(self.nbytes, dtype=torch.uint8, pin_memory=True)
        hv = self.host.numpy()
        for n in STEP_INPUTS:
            o, nb, _, _ = self.layout[n]
            hv[o:o + nb] = np.ascontiguousarray(host[n]).reshape(-1).view(np.uint8)
        if pool is None:
            pool = (_to_dev(b.k_cache, dev, b.dtype), _to_dev(b.v_cache, dev, b.dtype))
        self.B = b.B
        self.bufs, self.batches, self.outs = [], [], []
        for _ in range(depth):
            buf = torch.empty(self.nbytes, dtype=torch.uint8, device=dev)
            t = {}
            for n in STEP_INPUTS:
                o, nb, shape, dt = self.layout[n]
                view = buf[o:o + nb]
                if n in ("q", "logits") and b.dtype == "bf16":
                    t[n] = view.view(torch.bfloat16).view(shape)
                else:
                    t[n] = view.view(torch.from_numpy(np.empty(0, dt)).dtype).view(shape)
            t["k_cache"], t["v_cache"] = pool
            t["out"] = torch.empty_like(t["q"])
            res = torch.full((2, b.B), -7, dtype=torch.int32, device=dev)
            t["accepted_len"], t["next_token"] = res[0], res[1]
            t["results"] = res
            self.bufs.append(buf)
            self.batches.append(DeviceBatch.from_tensors(t, b.num_blocks, dev))
            self.outs.append(torch.empty((2, b.B), dtype=torch.int32, pin_memory=True))
        self.d2h_bytes = 2 * b.B * 4
        self.copy_stream = torch.cuda.Stream(device=dev)
        self.copied = [torch.cuda.Event() for _ in range(depth)]
        self.done = [torch.cuda.Event() for _ in range(depth)]
        self.n = 0

    def enqueue(self):
        """Enqueue one step (copy in, verify, copy the results out) on the current stream; returns
        the pinned host tensor its results land in once the current stream has reached this point."""
        i = self.n % len(self.bufs)
        self.n += 1
        cur = torch.cuda.current_stream()
        with torch.cuda.stream(self.copy_stream):
            self.copy_stream.wait_event(self.done[i])  # the step that last read buffer i has finished
            self.bufs[i].copy_(self.host, non_blocking=True)
            self.copied[i].record(self.copy_stream)
        cur.wait_event(self.copied[i])
        db = self.batches[i]
        db.step(cur.cuda_stream)
        self.done[i].record(cur)
        self.outs[i].copy_(db.t["results"], non_blocking=True)
        return self.outs[i]
