"""Seeded synthetic gradient generators and workload shapes.

This module is shared by the CUDA path's tests/benchmark and by the oracle's
tests.  It holds none of the method's arithmetic: bucket offsets are passed
in (from either side's plan), and it only draws and scales random numbers.

The paper's gradients come from fine-tuning 1B-8B LLMs on eight languages
(Figure 1, Appendix E); none of that data or those weights are available, so
every workload is synthetic with the tensor shapes of the named architecture.
Each language's gradient over a tensor is a shared direction plus a
language-specific one:

    g_k = sigma_t * (eps_k * rho_t * s + sqrt(1 - rho_t^2) * u_k)

with s, u_k i.i.d. N(0, 1) per element, sigma_t a per-tensor scale and rho_t
the per-bucket shared fraction.  Taken literally with eps_k = 1 the expected
pairwise cosine is rho^2 >= 0, so a negative rho could not produce the
conflicts the workloads ask for; a negative rho therefore flips the shared
part on odd languages (eps_k = (-1)^k), giving cosine -rho^2 between the two
groups and +rho^2 within them.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Sequence

import numpy as np

MiB = 1 << 20


# --------------------------------------------------------------------------
# Architecture tensor lists (registration order, element counts)
# --------------------------------------------------------------------------

def gpt2_small_sizes() -> list[int]:
    """GPT-2 small: 12 layers, d=768, FFN 3072, vocab 50257, 1024 positions,
    tied LM head (so no separate head tensor).  148 tensors, 124,439,808
    parameters."""
    d, f, v, p = 768, 3072, 50257, 1024
    sizes = [v * d, p * d]
    for _ in range(12):
        sizes += [d, d,                 # ln_1 weight, bias
                  d * 3 * d, 3 * d,     # attn.c_attn weight, bias
                  d * d, d,             # attn.c_proj weight, bias
                  d, d,                 # ln_2 weight, bias
                  d * f, f,             # mlp.c_fc weight, bias
                  f * d, d]             # mlp.c_proj weight, bias
    sizes += [d, d]                     # ln_f weight, bias
    return sizes


def llama32_1b_sizes() -> list[int]:
    """Llama-3.2-1B: 16 layers, hidden 2048, 32 q / 8 kv heads of 64, SwiGLU
    8192, vocab 128256, tied embedding.  146 tensors, 1,235,814,400
    parameters."""
    h, kv, f, v = 2048, 8 * 64, 8192, 128256
    sizes = [v * h]
    for _ in range(16):
        sizes += [h * h, kv * h, kv * h, h * h,   # q, k, v, o projections
                  f * h, f * h, h * f,            # gate, up, down
                  h, h]                           # input / post-attention RMSNorm
    sizes += [h]                                  # final norm
    return sizes


def qwen3_8b_sizes() -> list[int]:
    """Qwen3-8B: 36 layers, hidden 4096, 32 q / 8 kv heads of 128, q/k RMSNorm
    of 128, SwiGLU 12288, vocab 151936, untied LM head.  399 tensors,
    8,190,735,360 parameters."""
    h, kv, hd, f, v = 4096, 8 * 128, 128, 12288, 151936
    sizes = [v * h]
    for _ in range(36):
        sizes += [h * h, kv * h, kv * h, h * h,   # q, k, v, o projections
                  hd, hd,                         # q_norm, k_norm
                  f * h, f * h, h * f,            # gate, up, down
                  h, h]                           # input / post-attention RMSNorm
    sizes += [h, v * h]                           # final norm, lm_head
    return sizes


# --------------------------------------------------------------------------
# Workloads
# --------------------------------------------------------------------------

@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    K: int
    dtype: str                      # "f32" or "bf16"
    param_sizes: tuple[int, ...]    # registration order
    bucket_bytes: int
    rules: tuple[str, ...]
    kind: str                       # "tiny" | "shared"
    rho_lo: float = 0.0
    rho_hi: float = 0.0
    conflict_frac: float = 0.0      # fraction of buckets forced to rho_conflict
    rho_conflict: float = 0.0
    flip_frac: float = 0.0          # fraction of buckets with one language negated
    sigma_lognormal: bool = False   # per-tensor scale ~ LogNormal(0, 1)
    max_iter: int = 256
    seed: int = 0

    @property
    def elem_bytes(self) -> int:
        return 4 if self.dtype == "f32" else 2

    @property
    def n_elems(self) -> int:
        return int(sum(self.param_sizes))


TINY_COSINES = (-0.8, -0.2, 0.3, 0.9)


def tiny() -> Workload:
    """K=2, one fp32 vector of 1,048,576 elements in 4 buckets of 262,144 with
    pairwise cosines -0.8, -0.2, 0.3, 0.9 (one per bucket)."""
    return Workload("tiny-k2-f32", 2, "f32", (1 << 20,), MiB, ("mgda",), "tiny")


def gpt2_small() -> Workload:
    return Workload("gpt2-small-k4-f32", 4, "f32", tuple(gpt2_small_sizes()), 25 * MiB,
                    ("mgda", "pcgrad"), "shared", rho_lo=-0.3, rho_hi=0.95,
                    sigma_lognormal=True)


def llama32_1b() -> Workload:
    return Workload("llama3.2-1b-k8-bf16", 8, "bf16", tuple(llama32_1b_sizes()), 25 * MiB,
                    ("mgda",), "shared", rho_lo=-0.3, rho_hi=0.95, flip_frac=0.10,
                    sigma_lognormal=True, max_iter=20)


def qwen3_8b() -> Workload:
    return Workload("qwen3-8b-k4-bf16", 4, "bf16", tuple(qwen3_8b_sizes()), 25 * MiB,
                    ("mgda", "cagrad"), "shared", rho_lo=0.2, rho_hi=0.95,
                    conflict_frac=0.02, rho_conflict=-0.7, sigma_lognormal=True)


def qwen3_8b_layers(n_layers: int) -> Workload:
    """Qwen3-8B decoder-layer shapes only (no embedding / LM head), n_layers
    layers: the same kernels as the full model on a few GB (profiling)."""
    sizes = qwen3_8b_sizes()[1:1 + 11 * n_layers]
    return dataclasses.replace(qwen3_8b(), name="qwen3-8b-%dlayers-k4-bf16" % n_layers,
                               param_sizes=tuple(sizes))


def sweep(K: int, bucket_mib: int, n: int = 1_000_000_000) -> Workload:
    """1e9-element fp32 vector, N(0,1) gradients with a shared part at rho=0.3."""
    return Workload(f"sweep-k{K}-{bucket_mib}mib-f32", K, "f32", (n,), bucket_mib * MiB,
                    ("mgda", "pcgrad", "cagrad"), "shared", rho_lo=0.3, rho_hi=0.3)


SWEEP_K = (2, 4, 8, 16)
SWEEP_BUCKET_MIB = (1, 4, 25, 100)


def scaled(w: Workload, name: str, param_sizes: Sequence[int], bucket_bytes: int) -> Workload:
    """Same generator and rules on other shapes (small parity cases)."""
    return dataclasses.replace(w, name=name, param_sizes=tuple(int(s) for s in param_sizes),
                               bucket_bytes=int(bucket_bytes))


# --------------------------------------------------------------------------
# Per-bucket draws (host, numpy; tiny) and element generation (torch)
# --------------------------------------------------------------------------

@dataclasses.dataclass
class BucketDraws:
    rho: np.ndarray        # [B] shared fraction (signed)
    flip: np.ndarray       # [B] language index negated, or -1
    sigma: np.ndarray      # [n_tensors] per-tensor scale (registration order)


def bucket_draws(w: Workload, offsets: np.ndarray) -> BucketDraws:
    B = len(offsets) - 1
    rng = np.random.default_rng([w.seed, 0x5EED])
    if w.kind == "tiny":
        rho = np.array([TINY_COSINES[b % len(TINY_COSINES)] for b in range(B)])
    else:
        rho = rng.uniform(w.rho_lo, w.rho_hi, size=B)
        if w.conflict_frac > 0:
            n_c = max(1, int(round(w.conflict_frac * B)))
            idx = rng.choice(B, size=n_c, replace=False)
            rho[idx] = w.rho_conflict
    flip = np.full(B, -1, dtype=np.int64)
    if w.flip_frac > 0:
        n_f = max(1, int(round(w.flip_frac * B)))
        idx = rng.choice(B, size=n_f, replace=False)
        flip[idx] = rng.integers(0, w.K, size=n_f)
    if w.sigma_lognormal:
        sigma = np.exp(rng.standard_normal(len(w.param_sizes)))
    else:
        sigma = np.ones(len(w.param_sizes))
    return BucketDraws(rho=rho, flip=flip, sigma=sigma)


def _shared_coefs(w: Workload, rho: float, K: int):
    """(shared coefficient per language, specific coefficient)."""
    if w.kind == "tiny":
        # cos(g_1, g_2) = r exactly in expectation: a = sqrt|r|, c = sqrt(1-|r|),
        # shared part negated on the second language when r < 0.
        a, c = math.sqrt(abs(rho)), math.sqrt(1.0 - abs(rho))
        eps = [1.0] + [(-1.0 if rho < 0 else 1.0)] * (K - 1)
        return [a * e for e in eps], c
    r = abs(rho)
    eps = [((-1.0) ** k if rho < 0 else 1.0) for k in range(K)]
    return [r * e for e in eps], math.sqrt(max(0.0, 1.0 - r * r))


def tensor_offsets_flat(param_sizes: Sequence[int]) -> np.ndarray:
    """Start of each tensor (registration index) in the flat gradient, which
    lists tensors in reverse registration order.  Returns [n_tensors + 1]
    boundaries in flat order and the registration index of each flat slot."""
    rev = list(reversed(range(len(param_sizes))))
    bounds = np.zeros(len(param_sizes) + 1, dtype=np.int64)
    for i, t in enumerate(rev):
        bounds[i + 1] = bounds[i] + int(param_sizes[t])
    return bounds, np.array(rev, dtype=np.int64)


def generate(w: Workload, offsets: np.ndarray, device, buckets=None, out=None):
    """K flat gradients (torch tensors of w.dtype on `device`).

    offsets: the bucket boundaries (either side's plan).  buckets: optional
    iterable of bucket indices to fill (default all); out: optional list of K
    preallocated tensors.  Each bucket draws from its own torch.Generator
    seeded by (w.seed, bucket), so any subset is reproducible on its own.
    """
    import torch

    K = w.K
    tdt = torch.float32 if w.dtype == "f32" else torch.bfloat16
    N = int(offsets[-1])
    if out is None:
        out = [torch.empty(N, dtype=tdt, device=device) for _ in range(K)]
    draws = bucket_draws(w, offsets)
    bounds, reg_of_slot = tensor_offsets_flat(w.param_sizes)
    sig_flat = draws.sigma[reg_of_slot]             # per flat tensor slot
    B = len(offsets) - 1
    gen = torch.Generator(device=device)
    for b in (range(B) if buckets is None else buckets):
        lo, hi = int(offsets[b]), int(offsets[b + 1])
        n = hi - lo
        gen.manual_seed(int(w.seed) * 1_000_003 + 7919 * b + 1)
        s = torch.randn(n, generator=gen, device=device, dtype=torch.float32)
        # per-element sigma over the tensor pieces that overlap the bucket
        t0 = int(np.searchsorted(bounds, lo, side="right") - 1)
        t1 = int(np.searchsorted(bounds, hi, side="left"))
        pieces = []
        for t in range(t0, t1):
            a, z = max(lo, int(bounds[t])), min(hi, int(bounds[t + 1]))
            if z > a:
                pieces.append((z - a, float(sig_flat[t])))
        sig = torch.cat([torch.full((m,), v, dtype=torch.float32, device=device)
                         for m, v in pieces]) if len(pieces) > 1 else None
        sig0 = pieces[0][1] if len(pieces) == 1 else None
        shared, spec = _shared_coefs(w, float(draws.rho[b]), K)
        for k in range(K):
            u = torch.randn(n, generator=gen, device=device, dtype=torch.float32)
            g = u.mul_(spec).add_(s, alpha=shared[k])
            if sig is not None:
                g.mul_(sig)
            else:
                g.mul_(sig0)
            if draws.flip[b] == k:
                g.neg_()
            out[k][lo:hi].copy_(g)
    return out


def host_view(t) -> np.ndarray:
    """numpy view of a CPU torch tensor as the oracle reads it (float32, or
    uint16 bf16 bit patterns)."""
    import torch

    t = t.detach().cpu().contiguous()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy().view(np.uint16)
    if t.dtype == torch.float32:
        return t.numpy()
    raise TypeError(t.dtype)
