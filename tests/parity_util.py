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

PCGrad near ties: the conflict test <d_t, g_j> < 0 (Eq. 5) is
discontinuous, so where the oracle saw |<d_t, g_j>| within 1e-6 of
||d_t|| ||g_j|| either outcome is correct.  A bucket that fails against the
oracle's own branch is compared with every alternative result
(oracle.pcgrad_alternatives) and passes if one of them matches.
"""
import dataclasses

import numpy as np

from oracle import oracle as orc

BETA_ATOL = 1e-4
D_RTOL = {"f32": 1e-5, "bf16": 2e-3}
GRAM_RTOL = 1e-5
NOT_CONVERGED = 7           # BKMOO_ERR_NOT_CONVERGED (an accepted bucket status)
ORC_RULE = {"mgda": orc.MGDA, "pcgrad": orc.PCGRAD, "cagrad": orc.CAGRAD, "mean": orc.MEAN}


def gram_close(Gg, Go):
    scale = np.sqrt(np.outer(np.diag(Go), np.diag(Go)))
    err = np.abs(Gg - Go)
    ok = err <= GRAM_RTOL * scale + 1e-30
    return bool(ok.all()), float((err / np.maximum(scale, 1e-300)).max())


def d_rtol(out_dt, n):
    if out_dt == "bf16" and n < 4096:
        return 2.0 ** -8
    return D_RTOL[out_dt]


def d_check(d_gpu, d_or, beta_or, g_norms, out_dt):
    """(ok, relative error) of one bucket's direction."""
    nd = float(np.linalg.norm(d_or))
    err = float(np.linalg.norm(d_gpu - d_or))
    floor = (len(g_norms) + 2) * 2.0 ** -24 * float(np.dot(np.abs(beta_or), g_norms))
    ok = err <= d_rtol(out_dt, len(d_or)) * nd + floor
    return ok, (err / nd if nd > 0 else err)


def beta_unique(G):
    """beta is unique when G is positive definite (MGDA, CAGrad)."""
    ev = np.linalg.eigvalsh(G)
    return ev.min() > 1e-10 * max(np.trace(G), 1e-300)


def widen(h):
    if h.dtype == np.uint16:
        return (h.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    return h.astype(np.float64)


@dataclasses.dataclass
class Run:
    """One GPU resolve to compare: its plan, rule and results (beta and
    status as numpy arrays over the whole plan, out the device direction)."""
    name: str
    off: np.ndarray
    rule: str
    out: object
    beta: np.ndarray
    status: np.ndarray
    out_dt: str
    seed: int = 0
    step: int = 0
    mgda_mode: int = orc.MGDA_EXACT
    max_iter: int = 256
    cagrad_c: float = 0.5
    checked: int = 0

    def oracle_key(self):
        return (id(self.off), self.rule, self.seed, self.step, self.mgda_mode, self.max_iter,
                self.cagrad_c)


def oracle_window(hv, off, b0, b1, run, n_threads=0):
    """The oracle over buckets [b0, b1) of `off`, where hv holds elements
    [off[b0], off[b1]) of each gradient (the bucket indices stay those of the
    whole plan, so PCGrad's order is the plan's)."""
    shifted = np.ascontiguousarray(off - off[b0], dtype=np.int64)
    return orc.resolve(hv, shifted, ORC_RULE[run.rule], b0=b0, b1=b1, mgda_mode=run.mgda_mode,
                       max_iter=run.max_iter, cagrad_c=run.cagrad_c, seed=run.seed,
                       step=run.step, want_gram=True,
                       n_threads=n_threads or orc.max_threads())


def check_window(hv, b0, b1, ref, run):
    """Every bucket of [b0, b1) of `run` against the oracle result `ref`
    (oracle_window over the same buckets).  Returns the worst relative error
    of d.  The direction is compared on the device (fp64)."""
    import torch

    off = run.off
    K = len(hv)
    lo0, hi0 = int(off[b0]), int(off[b1])
    nb = b1 - b0
    G = ref["gram"]
    st = run.status[b0:b1]
    bad = np.nonzero(~np.isin(st, (0, NOT_CONVERGED)))[0]
    assert len(bad) == 0, (run.name, "status", b0 + bad[:5], st[bad[:5]])
    dev = run.out.device
    d_or = torch.from_numpy(ref["d"]).to(dev)
    d_gp = run.out[lo0:hi0].to(torch.float64)
    diff = d_gp - d_or
    rel = off[b0:b1 + 1] - lo0
    errs, nds = [], []
    for i in range(nb):
        s, e = int(rel[i]), int(rel[i + 1])
        errs.append(torch.linalg.vector_norm(diff[s:e]))
        nds.append(torch.linalg.vector_norm(d_or[s:e]))
    err = torch.stack(errs).cpu().numpy()
    nd = torch.stack(nds).cpu().numpy()
    lens = np.diff(rel)
    gn = np.sqrt(np.clip(np.einsum("bkk->bk", G), 0, None))
    bo = ref["beta"]
    floor = (K + 2) * 2.0 ** -24 * np.einsum("bk,bk->b", np.abs(bo), gn)
    rtol = np.array([d_rtol(run.out_dt, int(n)) for n in lens])
    d_ok = err <= rtol * nd + floor
    beta_err = np.abs(run.beta[b0:b1].astype(np.float64) - bo).max(axis=1)
    beta_ok = beta_err <= BETA_ATOL
    if run.rule in ("mgda", "cagrad"):
        for i in np.nonzero(~beta_ok)[0]:
            beta_ok[i] = not beta_unique(G[i])
    for i in np.nonzero(~(d_ok & beta_ok))[0]:
        b = b0 + int(i)
        if run.rule == "pcgrad" and _pcgrad_tie_ok(hv, run, b, G[i], int(rel[i]), int(lens[i]),
                                                   d_gp[int(rel[i]):int(rel[i + 1])], gn[i]):
            continue
        raise AssertionError((run.name, run.rule, "bucket", b, "beta err", float(beta_err[i]),
                              "d err", float(err[i]), "|d|", float(nd[i]),
                              "allowed", float(rtol[i] * nd[i] + floor[i])))
    run.checked += nb
    with np.errstate(divide="ignore", invalid="ignore"):
        r = np.where(nd > 0, err / nd, err)
    return float(r.max()) if nb else 0.0


def _pcgrad_tie_ok(hv, run, b, G, start, n, d_gpu, gn):
    alts = orc.pcgrad_alternatives(G, run.seed, run.step, b)
    if len(alts) < 2:
        return False
    dg = d_gpu.cpu().numpy()
    bg = run.beta[b].astype(np.float64)
    K = len(hv)
    for a in alts:
        if np.abs(bg - a).max() > BETA_ATOL:
            continue
        da = orc.combine(hv, a, start, n)
        floor = (K + 2) * 2.0 ** -24 * float(np.dot(np.abs(a), gn))
        if np.linalg.norm(dg - da) <= d_rtol(run.out_dt, n) * np.linalg.norm(da) + floor:
            return True
    return False


def window_bounds(off, max_elems, min_buckets=1):
    """Element boundaries of consecutive windows of whole buckets of `off`:
    each window holds at least min_buckets buckets (the last may hold fewer)
    and otherwise at most max_elems elements."""
    bounds = [0]
    B = len(off) - 1
    b = 0
    while b < B:
        e = b + 1
        while e < B and (e - b < min_buckets or off[e + 1] - off[b] <= max_elems):
            e += 1
        bounds.append(int(off[e]))
        b = e
    return bounds


def compare_all(grads, runs, bounds):
    """Stream the gradients to the host window by window (bounds: element
    boundaries that are bucket boundaries of every run's plan) and compare
    every bucket of every run with the oracle; each distinct oracle
    configuration runs once per window.  Asserts that every bucket of every
    run was compared; returns {run name: worst relative d error}."""
    import torch

    from paper_2606_05613_gb300 import inputs

    widest = max(b - a for a, b in zip(bounds[:-1], bounds[1:]))
    stage = [torch.empty(widest, dtype=g.dtype, pin_memory=True) for g in grads]
    worst = {r.name: 0.0 for r in runs}
    for lo, hi in zip(bounds[:-1], bounds[1:]):
        n = hi - lo
        for s, g in zip(stage, grads):
            s[:n].copy_(g[lo:hi])
        hv = [inputs.host_view(s[:n]) for s in stage]
        groups = {}
        for r in runs:
            groups.setdefault(r.oracle_key(), []).append(r)
        for same in groups.values():
            r0 = same[0]
            b0 = int(np.searchsorted(r0.off, lo))
            b1 = int(np.searchsorted(r0.off, hi))
            assert r0.off[b0] == lo and r0.off[b1] == hi, (r0.name, lo, hi)
            ref = oracle_window(hv, r0.off, b0, b1, r0)
            for r in same:
                worst[r.name] = max(worst[r.name], check_window(hv, b0, b1, ref, r))
            del ref
    for r in runs:
        assert r.checked == len(r.off) - 1, (r.name, r.checked, len(r.off) - 1)
    return worst
