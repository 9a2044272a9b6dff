"""Shared comparison helpers of the GPU parity tests.

Tolerances (per bucket):
  offsets: bit-exact.
  beta: within 1e-4 absolute of the oracle.
  d: ||d_gpu - d_oracle|| <= rtol ||d_oracle|| + (K + 2) 2^-24 sum_k |beta_k| ||g_k||
     with rtol = 1e-5 for fp32 output and 2e-3 for bf16 output.  The second
     term is the rounding floor of forming sum_k beta_k x_k in fp32 (K fused
     multiply-adds, each within 2^-24 of the running sum's magnitude, plus
     the fp32 rounding of beta); it only matters where d_oracle is near 0
     (opposed or linearly dependent gradients, Theorem 3.1 (a)), where a
     pure relative error is undefined.  bf16 output: round-to-nearest-even
     has a relative error of at most 2^-8 per element, so
     ||bf16(d) - d|| <= 2^-8 ||d|| always; 2e-3 is the rms that a long
     bucket reaches (about 1.6e-3), so buckets under 4096 elements are held
     to the hard bound 2^-8 instead.
  Gram: |G_gpu - G_oracle| <= 1e-5 sqrt(G_ii G_jj).  Each entry is summed in
     fp32 over at most 128 products per thread, then through a 5-level fp32
     shuffle tree, then in fp64; the fp32 stages contribute at most
     (128 + 5) u ~ 7.9e-6 (u = 2^-24) of sum |x_i x_j| <= sqrt(G_ii G_jj).
"""
import numpy as np

BETA_ATOL = 1e-4
D_RTOL = {"f32": 1e-5, "bf16": 2e-3}
GRAM_RTOL = 1e-5


def gram_close(Gg, Go):
    scale = np.sqrt(np.outer(np.diag(Go), np.diag(Go)))
    err = np.abs(Gg - Go)
    ok = err <= GRAM_RTOL * scale + 1e-30
    return bool(ok.all()), float((err / np.maximum(scale, 1e-300)).max())


def d_check(d_gpu, d_or, beta_or, g_norms, out_dt):
    """(ok, relative error) of one bucket's direction."""
    nd = float(np.linalg.norm(d_or))
    err = float(np.linalg.norm(d_gpu - d_or))
    floor = (len(g_norms) + 2) * 2.0 ** -24 * float(np.dot(np.abs(beta_or), g_norms))
    rtol = D_RTOL[out_dt]
    if out_dt == "bf16" and len(d_or) < 4096:
        rtol = 2.0 ** -8
    ok = err <= rtol * nd + floor
    return ok, (err / nd if nd > 0 else err)


def beta_unique(G):
    """beta is unique when G is positive definite (MGDA, CAGrad)."""
    ev = np.linalg.eigvalsh(G)
    return ev.min() > 1e-10 * max(np.trace(G), 1e-300)


def widen(h):
    if h.dtype == np.uint16:
        return (h.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    return h.astype(np.float64)
