"""Seeded synthetic verification batches (inputs only; none of the method's arithmetic).

A verification batch is what WISP's scheduler hands the verification engine
(Sec. 4.5): for every request a draft block y_1..y_k with its draft
distribution q, the cached-prefix length (L_cached, Sec. 4.4) and a paged KV
block table (PageAttention layout, Sec. 4.5), plus the target logits of the
k+1 new positions.  This module only *draws* such batches; the oracle and the
CUDA library both consume them and share nothing else.

Layouts (row-major, all integer ids 0-based):
  q            [T_q, Hq, D]              T_q = sum_r (k_r + 1)
  k_cache      [num_blocks, Hkv, 16, D]  (v_cache likewise)
  block_tables [B, max_blocks_per_seq]   int32, -1 past a request's last block
  logits       [T_q, V]                  rows of request r are contiguous
  draft_tokens [T_d], draft_probs [T_d, V], accept_uniforms [T_d]
  sample_uniforms [B]
bf16 tensors are stored as uint16 bit patterns (round-to-nearest-even of a
float32 draw), so both sides read exactly the same values.

Draft noise.  q = softmax(z + N(0, sigma^2)) with z the target logits of the
same position.  For many vocabulary entries the expected acceptance
sum_v min(p_v, q_v) tends to erfc(sigma / (2 sqrt 2)) whatever the logit
scale, so sigma for a target acceptance alpha is 2 sqrt(2) erfcinv(alpha)
(the acceptance notion alpha of Eq. 3, N^v = alpha * N_d, read as the
per-token coupling probability of the acceptance rule, Eq. 1).
"""
from __future__ import annotations

import dataclasses
import math
import os
from concurrent.futures import ThreadPoolExecutor

import numpy as np

ROOT_SEED = 260111652
BLOCK_SIZE = 16
_CHUNK = 1 << 24  # elements per independently seeded chunk of a large tensor


# --------------------------------------------------------------------------
# configurations (the five verification workloads this library is measured on)
# --------------------------------------------------------------------------
@dataclasses.dataclass(frozen=True)
class WorkloadSpec:
    name: str
    config_id: int
    B: int
    Hq: int
    Hkv: int
    D: int
    V: int
    dtype: str                 # "f32" or "bf16" (Q/K/V and logits)
    k_rule: tuple              # ("fixed", [..]) | ("uniform", lo, hi)
    ctx_rule: tuple            # ("fixed", [..]) | ("uniform", lo, hi) | ("lognormal", median, ln_sd, lo, hi) | ("bimodal", p_short, (lo, hi), (lo, hi))
    noise_rule: tuple          # ("sigma", s) | ("alpha", a) | ("alpha_uniform", lo, hi)
    shuffle_blocks: bool = False
    logit_sd: float = 2.0


SPECS = {
    s.name: s
    for s in [
        WorkloadSpec("tiny_f32", 0, 4, 4, 4, 64, 1000, "f32",
                     ("fixed", [1, 2, 3, 4]), ("fixed", [16, 40, 77, 128]), ("sigma", 0.5)),
        WorkloadSpec("llama3_8b_b32", 1, 32, 32, 8, 128, 128256, "bf16",
                     ("uniform", 1, 8), ("uniform", 512, 4096), ("alpha", 0.7)),
        WorkloadSpec("fanin_b256", 2, 256, 32, 8, 128, 128256, "bf16",
                     ("uniform", 1, 16), ("lognormal", 2048.0, 1.0, 1, 16384), ("alpha_uniform", 0.4, 0.9)),
        WorkloadSpec("longctx_b16", 3, 16, 32, 8, 128, 128256, "bf16",
                     ("uniform", 4, 8), ("uniform", 32768, 131072), ("alpha", 0.7), shuffle_blocks=True),
        WorkloadSpec("hetero_b512", 4, 512, 28, 4, 128, 152064, "bf16",
                     ("uniform", 0, 12), ("bimodal", 0.7, (256, 1024), (8192, 32768)), ("alpha_uniform", 0.3, 0.95)),
    ]
}
CONFIG_ORDER = ["tiny_f32", "llama3_8b_b32", "fanin_b256", "longctx_b16", "hetero_b512"]


@dataclasses.dataclass
class VerifyBatch:
    name: str
    B: int
    Hq: int
    Hkv: int
    D: int
    V: int
    block_size: int
    dtype: str
    request_ids: np.ndarray
    draft_lens: np.ndarray
    context_lens: np.ndarray
    block_tables: np.ndarray
    num_blocks: int
    q: np.ndarray
    k_cache: np.ndarray
    v_cache: np.ndarray
    logits: np.ndarray
    draft_tokens: np.ndarray
    draft_probs: np.ndarray
    accept_uniforms: np.ndarray
    sample_uniforms: np.ndarray
    sigma: np.ndarray          # per-request draft noise used (for reporting only)

    @property
    def total_q_rows(self) -> int:
        return int(self.draft_lens.sum()) + self.B

    @property
    def total_draft(self) -> int:
        return int(self.draft_lens.sum())

    @property
    def max_blocks_per_seq(self) -> int:
        return int(self.block_tables.shape[1])

    def q_row_start(self) -> np.ndarray:
        return np.concatenate([[0], np.cumsum(self.draft_lens + 1)]).astype(np.int64)

    def draft_start(self) -> np.ndarray:
        return np.concatenate([[0], np.cumsum(self.draft_lens)]).astype(np.int64)

    def kv_tokens(self) -> int:
        return int((self.context_lens.astype(np.int64) + self.draft_lens + 1).sum())

    def subset(self, reqs) -> "VerifyBatch":
        """The same requests as a smaller batch (shares the KV pool)."""
        reqs = np.asarray(reqs, dtype=np.int64)
        qs, ds = self.q_row_start(), self.draft_start()
        qrows = np.concatenate([np.arange(qs[r], qs[r + 1]) for r in reqs]).astype(np.int64)
        drows = np.concatenate([np.arange(ds[r], ds[r + 1]) for r in reqs] + [np.zeros(0, np.int64)]).astype(np.int64)
        return dataclasses.replace(
            self, B=len(reqs), request_ids=self.request_ids[reqs].copy(),
            draft_lens=self.draft_lens[reqs].copy(), context_lens=self.context_lens[reqs].copy(),
            block_tables=self.block_tables[reqs].copy(), q=self.q[qrows], logits=self.logits[qrows],
            draft_tokens=self.draft_tokens[drows], draft_probs=self.draft_probs[drows],
            accept_uniforms=self.accept_uniforms[drows], sample_uniforms=self.sample_uniforms[reqs].copy(),
            sigma=self.sigma[reqs].copy())


# --------------------------------------------------------------------------
# primitive draws
# --------------------------------------------------------------------------
def _ss(*key) -> np.random.SeedSequence:
    return np.random.SeedSequence([ROOT_SEED, *[int(k) for k in key]])


def _rng(*key) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(_ss(*key)))


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 to bfloat16 (nearest, ties to even); returns uint16 bits."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    r = (u + np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))) >> np.uint32(16)
    return r.astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def _normal_fill(out_flat: np.ndarray, key: tuple, scale: float, as_bf16: bool, threads: int = 8) -> None:
    """Fill out_flat with scale*N(0,1) draws; each 2^24-element chunk has its own seed."""
    n = out_flat.size
    nchunks = (n + _CHUNK - 1) // _CHUNK

    def work(c):
        lo, hi = c * _CHUNK, min(n, (c + 1) * _CHUNK)
        x = _rng(*key, c).standard_normal(hi - lo, dtype=np.float32)
        if scale != 1.0:
            x *= np.float32(scale)
        out_flat[lo:hi] = f32_to_bf16_bits(x) if as_bf16 else x

    if nchunks == 1:
        work(0)
    else:
        with ThreadPoolExecutor(max_workers=threads) as ex:
            list(ex.map(work, range(nchunks)))


def _normal_tensor(shape, key, scale, dtype):
    as_bf16 = dtype == "bf16"
    out = np.empty(int(np.prod(shape)), dtype=np.uint16 if as_bf16 else np.float32)
    _normal_fill(out, key, scale, as_bf16)
    return out.reshape(shape)


def sigma_for_alpha(alpha):
    """Draft-noise sigma giving expected acceptance alpha (large-vocabulary limit)."""
    from scipy.special import erfcinv
    return 2.0 * math.sqrt(2.0) * erfcinv(np.asarray(alpha, dtype=np.float64))


def alpha_for_sigma(sigma):
    from scipy.special import erfc
    return erfc(np.asarray(sigma, dtype=np.float64) / (2.0 * math.sqrt(2.0)))


def _draw_lengths(spec: WorkloadSpec, rng: np.random.Generator, rule, B):
    kind = rule[0]
    if kind == "fixed":
        v = np.asarray(rule[1], dtype=np.int64)
        assert len(v) == B
        return v
    if kind == "uniform":
        return rng.integers(rule[1], rule[2] + 1, size=B)
    if kind == "lognormal":
        _, median, ln_sd, lo, hi = rule
        x = np.round(rng.lognormal(math.log(median), ln_sd, size=B))
        return np.clip(x, lo, hi).astype(np.int64)
    if kind == "bimodal":
        _, p_short, (a0, a1), (b0, b1) = rule
        short = rng.random(B) < p_short
        return np.where(short, rng.integers(a0, a1 + 1, size=B), rng.integers(b0, b1 + 1, size=B))
    raise ValueError(rule)


# --------------------------------------------------------------------------
# batch assembly
# --------------------------------------------------------------------------
def make_batch_from_lengths(name, *, draft_lens, context_lens, Hq, Hkv, D, V, dtype,
                            sigma, key, shuffle_blocks=False, logit_sd=2.0,
                            extra_blocks=0) -> VerifyBatch:
    """Assemble a batch for given per-request lengths; every tensor drawn from `key`."""
    draft_lens = np.asarray(draft_lens, dtype=np.int32)
    context_lens = np.asarray(context_lens, dtype=np.int32)
    B = len(draft_lens)
    sigma = np.broadcast_to(np.asarray(sigma, dtype=np.float64), (B,)).copy()
    kv_len = context_lens.astype(np.int64) + draft_lens + 1
    nblk = (kv_len + BLOCK_SIZE - 1) // BLOCK_SIZE
    num_blocks = int(nblk.sum()) + int(extra_blocks)
    max_blocks = int(max(1, nblk.max() if B else 1))
    phys = np.arange(num_blocks, dtype=np.int64)
    if shuffle_blocks:
        phys = _rng(*key, 1).permutation(num_blocks)
    bt = np.full((B, max_blocks), -1, dtype=np.int32)
    off = 0
    for r in range(B):
        bt[r, : nblk[r]] = phys[off: off + nblk[r]]
        off += int(nblk[r])

    T_q = int(draft_lens.sum()) + B
    T_d = int(draft_lens.sum())
    q = _normal_tensor((T_q, Hq, D), (*key, 2), 1.0, dtype)
    k_cache = _normal_tensor((num_blocks, Hkv, BLOCK_SIZE, D), (*key, 3), 1.0, dtype)
    v_cache = _normal_tensor((num_blocks, Hkv, BLOCK_SIZE, D), (*key, 4), 1.0, dtype)
    logits = _normal_tensor((T_q, V), (*key, 5), logit_sd, dtype)

    # draft distributions q_j = softmax(z_{j-1} + sigma * N(0,1)), stored fp32, and y_j ~ q_j
    draft_probs = np.empty((T_d, V), dtype=np.float32)
    draft_tokens = np.empty(T_d, dtype=np.int32)
    qs = np.concatenate([[0], np.cumsum(draft_lens + 1)])
    ds = np.concatenate([[0], np.cumsum(draft_lens)])
    z_f32 = (lambda rows: bf16_bits_to_f32(logits[rows])) if dtype == "bf16" else (lambda rows: logits[rows])
    def one_request(r):
        # request r's noise and token draws come from its own stream, so requests run in parallel
        k = int(draft_lens[r])
        if k == 0:
            return
        rng = _rng(*key, 6, r)
        base = z_f32(np.arange(qs[r], qs[r] + k)).astype(np.float64)
        x = base + sigma[r] * rng.standard_normal((k, V))
        x -= x.max(axis=1, keepdims=True)
        np.exp(x, out=x)
        x /= x.sum(axis=1, keepdims=True)
        qf = x.astype(np.float32)
        draft_probs[ds[r]: ds[r] + k] = qf
        cdf = np.cumsum(qf.astype(np.float64), axis=1)
        u = rng.random(k)
        for j in range(k):
            t = int(np.searchsorted(cdf[j], u[j] * cdf[j, -1], side="right"))
            t = min(t, V - 1)
            while qf[j, t] == 0.0 and t > 0:  # never hand out a token the draft gave zero mass
                t -= 1
            draft_tokens[ds[r] + j] = t

    with ThreadPoolExecutor(max_workers=min(32, os.cpu_count() or 1)) as ex:
        list(ex.map(one_request, range(B)))
    accept_u = _rng(*key, 8).random(T_d, dtype=np.float32)
    sample_u = _rng(*key, 9).random(B, dtype=np.float32)
    return VerifyBatch(
        name=name, B=B, Hq=Hq, Hkv=Hkv, D=D, V=V, block_size=BLOCK_SIZE, dtype=dtype,
        request_ids=(np.arange(B, dtype=np.int64) + 1000 * (key[0] + 1)),
        draft_lens=draft_lens, context_lens=context_lens, block_tables=bt, num_blocks=num_blocks,
        q=q, k_cache=k_cache, v_cache=v_cache, logits=logits, draft_tokens=draft_tokens,
        draft_probs=draft_probs, accept_uniforms=accept_u, sample_uniforms=sample_u, sigma=sigma)


def make_batch(name: str, variant: int = 0) -> VerifyBatch:
    """One of the named workloads; `variant` selects an independent seed."""
    spec = SPECS[name]
    key = (spec.config_id, variant)
    lrng = _rng(*key, 0)
    k = _draw_lengths(spec, lrng, spec.k_rule, spec.B)
    c = _draw_lengths(spec, lrng, spec.ctx_rule, spec.B)
    nr = spec.noise_rule
    if nr[0] == "sigma":
        sigma = np.full(spec.B, nr[1])
    elif nr[0] == "alpha":
        sigma = np.full(spec.B, float(sigma_for_alpha(nr[1])))
    else:
        sigma = sigma_for_alpha(lrng.uniform(nr[1], nr[2], size=spec.B))
    return make_batch_from_lengths(
        name, draft_lens=k, context_lens=c, Hq=spec.Hq, Hkv=spec.Hkv, D=spec.D, V=spec.V,
        dtype=spec.dtype, sigma=sigma, key=key, shuffle_blocks=spec.shuffle_blocks,
        logit_sd=spec.logit_sd)


def make_small_batch(seed: int, *, B=5, Hq=8, Hkv=2, D=128, V=4096, dtype="bf16",
                     k_range=(0, 9), ctx_range=(0, 700), alpha=0.7, shuffle_blocks=True) -> VerifyBatch:
    """A small random batch (oracle finishes in seconds) spanning several KV tiles and ragged tails."""
    key = (100 + seed, 0)
    lrng = _rng(*key, 0)
    k = lrng.integers(k_range[0], k_range[1] + 1, size=B)
    c = lrng.integers(ctx_range[0], ctx_range[1] + 1, size=B)
    return make_batch_from_lengths(
        f"small{seed}", draft_lens=k, context_lens=c, Hq=Hq, Hkv=Hkv, D=D, V=V, dtype=dtype,
        sigma=float(sigma_for_alpha(alpha)), key=key, shuffle_blocks=shuffle_blocks, extra_blocks=3)


def make_round(key, *, k, Hq, Hkv, D, V, dtype="bf16", alpha=0.7, prefix=0) -> dict:
    """One verification round of one session, drawn from `key`: the k + 1 query rows, the k + 1 new
    K/V rows, k + 1 logit rows, k draft tokens with their distributions and uniforms, one sample
    uniform; with prefix > 0 also `prefix` K/V rows for the session's first context."""
    b = make_batch_from_lengths(f"round{key}", draft_lens=[k], context_lens=[prefix], Hq=Hq, Hkv=Hkv, D=D, V=V,
                                dtype=dtype, sigma=float(sigma_for_alpha(alpha)), key=tuple(key))
    pos = np.arange(prefix + k + 1)
    pages = b.block_tables[0, pos // BLOCK_SIZE]
    kr = b.k_cache[pages, :, pos % BLOCK_SIZE, :]   # [prefix + k + 1, Hkv, D] in token order
    vr = b.v_cache[pages, :, pos % BLOCK_SIZE, :]
    return {"prefix_k": kr[:prefix], "prefix_v": vr[:prefix], "q": b.q, "k_new": kr[prefix:], "v_new": vr[prefix:],
            "logits": b.logits, "draft_tokens": b.draft_tokens, "draft_probs": b.draft_probs,
            "accept_u": b.accept_uniforms, "sample_u": float(b.sample_uniforms[0])}
