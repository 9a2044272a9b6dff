"""Full-size workloads on the GPU, in the launch configuration the benchmark
times: every bucket is resolved on the device; a sample of buckets is
recomputed one by one by the oracle (bucket data copied to the host) and
compared element by element; properties that hold at any size are checked on
every bucket."""
import dataclasses

import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2606_05613_gb300 import build as nb
from paper_2606_05613_gb300 import inputs
from paper_2606_05613_gb300 import native as bk
from tests.parity_util import BETA_ATOL, beta_unique, d_check, gram_close, widen

pytestmark = pytest.mark.gpu

DEV = torch.device("cuda:0")
ORC_RULE = {"mgda": orc.MGDA, "pcgrad": orc.PCGRAD, "cagrad": orc.CAGRAD, "mean": orc.MEAN}


@pytest.fixture(scope="module", autouse=True)
def _built():
    nb.build()
    bk.load()
    orc.build()


def _tdt(dt):
    return torch.float32 if dt == "f32" else torch.bfloat16


def _bucket_host(grads, lo, hi):
    return [inputs.host_view(g[lo:hi]) for g in grads]


def _check_sampled(w, off, grads, out, beta, status, rule, buckets, *, seed=0, step=0,
                   mgda_mode=orc.MGDA_EXACT, max_iter=256, out_dt=None):
    out_dt = out_dt or w.dtype
    for b in buckets:
        lo, hi = int(off[b]), int(off[b + 1])
        hv = _bucket_host(grads, lo, hi)
        sub = np.array([0, hi - lo], dtype=np.int64)
        # PCGrad's order depends on the bucket index: resolve the single
        # bucket as bucket b by shifting the oracle's bucket range
        if rule == "pcgrad":
            G = orc.gram(hv)
            bt, ties = orc.pcgrad(G, seed, step, b)
            if ties:
                continue
            ref = {"beta": bt[None, :], "d": orc.combine(hv, bt), "gram": G[None]}
        else:
            ref = orc.resolve(hv, sub, ORC_RULE[rule], cagrad_c=0.5, mgda_mode=mgda_mode,
                              max_iter=max_iter, want_gram=True)
        G = ref["gram"][0]
        assert status[b] in (0, bk.BKMOO_ERR_NOT_CONVERGED), (b, status[b])
        if rule == "pcgrad" or beta_unique(G):
            assert np.abs(beta[b] - ref["beta"][0]).max() <= BETA_ATOL, (b, beta[b], ref["beta"][0])
        d = out[lo:hi].float().cpu().numpy().astype(np.float64)
        gn = np.array([np.linalg.norm(widen(h)) for h in hv])
        ok, e = d_check(d, ref["d"], ref["beta"][0], gn, out_dt)
        assert ok, (w.name, rule, b, e)


def _mgda_properties(G_all, beta):
    """On every bucket: beta on the simplex and the min-norm optimality
    inequality <g_k, d> >= ||d||^2 (proof of Theorem 3.1) up to the fp32
    rounding of beta."""
    for b in range(len(G_all)):
        G, a = G_all[b], beta[b].astype(np.float64)
        assert abs(a.sum() - 1) <= 1e-5 and (a >= 0).all(), (b, a)
        v = G @ a
        assert (v >= a @ v - 1e-5 * np.diag(G).max()).all(), b


def _setup(w, gen_offsets=None):
    off = bk.bkmoo_plan(w.param_sizes, w.elem_bytes, w.bucket_bytes)
    np.testing.assert_array_equal(off, orc.plan(w.param_sizes, w.elem_bytes, w.bucket_bytes))
    grads = inputs.generate(w, off if gen_offsets is None else gen_offsets, DEV)
    return off, grads


def _resolve(w, off, grads, rule, params=None, res=None, out=None):
    B = len(off) - 1
    if res is None:
        res = bk.Resolver(w.K, _tdt(w.dtype), off, DEV)
    if out is None:
        out = torch.empty(int(off[-1]), dtype=_tdt(w.dtype), device=DEV)
    beta = torch.empty(B, w.K, dtype=torch.float32, device=DEV)
    status = torch.empty(B, dtype=torch.int32, device=DEV)
    res.resolve(grads, rule, out, params=params, out_weights=beta, out_status=status)
    torch.cuda.synchronize()
    assert res.status() == 0
    return res, out, beta.cpu().numpy(), status.cpu().numpy()


def _gram_all(res, grads, w, off):
    B = len(off) - 1
    G = torch.empty(B, w.K, w.K, dtype=torch.float64, device=DEV)
    res.gram(grads, G)
    return G.cpu().numpy()


def _spread(B, n):
    return sorted(set([0, B - 1] + [int(x) for x in np.linspace(0, B - 1, n)]))


def test_gpt2_small_k4_f32_mgda_pcgrad():
    w = inputs.gpt2_small()
    off, grads = _setup(w)
    assert len(off) - 1 == 22
    G = None
    for rule in ("mgda", "pcgrad"):
        p = bk.bkmoo_default_params()
        p.seed, p.step = 123, 7
        res, out, beta, st = _resolve(w, off, grads, rule, p)
        if G is None:
            G = _gram_all(res, grads, w, off)
            for b in (0, 10, 21):
                lo, hi = int(off[b]), int(off[b + 1])
                ok, err = gram_close(G[b], orc.gram(_bucket_host(grads, lo, hi)))
                assert ok, (b, err)
        if rule == "mgda":
            _mgda_properties(G, beta)
        _check_sampled(w, off, grads, out, beta, st, rule, _spread(22, 5), seed=123, step=7)


def test_llama32_1b_k8_bf16_mgda_fw20():
    w = inputs.llama32_1b()
    off, grads = _setup(w)
    B = len(off) - 1
    assert B == 134
    draws = inputs.bucket_draws(w, off)
    flipped = [int(b) for b in np.nonzero(draws.flip >= 0)[0]]
    assert len(flipped) == round(0.1 * B)
    samples = _spread(B, 4) + flipped[:3]
    # <= 20 Frank-Wolfe steps, then the exact completion: the exact minimiser
    p = bk.bkmoo_default_params()
    p.max_iter = 20
    res, out, beta, st = _resolve(w, off, grads, "mgda", p)
    assert (st == 0).all()
    _mgda_properties(_gram_all(res, grads, w, off), beta)
    _check_sampled(w, off, grads, out, beta, st, "mgda", samples)
    # <= 20 Frank-Wolfe steps alone: the oracle's Frank-Wolfe replay
    p.flags = 0
    _, out, beta, st = _resolve(w, off, grads, "mgda", p, res=res, out=out)
    _check_sampled(w, off, grads, out, beta, st, "mgda", samples, mgda_mode=orc.MGDA_FW,
                   max_iter=20)


def test_qwen3_8b_k4_bf16_mgda_cagrad():
    w = inputs.qwen3_8b()
    off, grads = _setup(w)
    B = len(off) - 1
    assert B == 672
    draws = inputs.bucket_draws(w, off)
    conflicted = [int(b) for b in np.nonzero(draws.rho < 0)[0]]
    assert len(conflicted) == round(0.02 * B)
    samples = _spread(B, 3) + conflicted[:3]
    res = None
    out = None
    for fused in (False, True):
        for rule in ("mgda", "cagrad"):
            p = bk.bkmoo_default_params()
            if fused:
                p.flags |= bk.BKMOO_FLAG_FUSED
            res, out, beta, st = _resolve(w, off, grads, rule, p, res=res, out=out)
            assert (st == 0).all(), np.unique(st, return_counts=True)
            _check_sampled(w, off, grads, out, beta, st, rule, samples)
            if rule == "mgda":
                _mgda_properties(_gram_all(res, grads, w, off), beta)


@pytest.mark.parametrize("K", inputs.SWEEP_K)
def test_sweep_1e9_f32(K):
    """1e9-element fp32 vector, every bucket size and rule; the data is drawn
    once (on the 100 MiB partition) and resolved under each partition."""
    w100 = inputs.sweep(K, 100)
    gen_off = orc.plan(w100.param_sizes, 4, w100.bucket_bytes)
    grads = inputs.generate(w100, gen_off, DEV)
    out = torch.empty(10**9, dtype=torch.float32, device=DEV)
    for mib in inputs.SWEEP_BUCKET_MIB:
        w = inputs.sweep(K, mib)
        off = bk.bkmoo_plan(w.param_sizes, 4, w.bucket_bytes)
        B = len(off) - 1
        res = bk.Resolver(K, torch.float32, off, DEV)
        # one full-size bucket and the ragged last bucket
        samples = [B // 2, B - 1]
        for rule in ("mgda", "pcgrad", "cagrad"):
            p = bk.bkmoo_default_params()
            p.seed, p.step = 9, mib
            _, out, beta, st = _resolve(w, off, grads, rule, p, res=res, out=out)
            _check_sampled(w, off, grads, out, beta, st, rule, samples if mib <= 25 else [B - 1],
                           seed=9, step=mib)
    del grads


def test_deterministic_full_size_step():
    """Two resolves of the same full-size input give bit-identical outputs."""
    w = inputs.gpt2_small()
    off, grads = _setup(w)
    res, out1, b1, _ = _resolve(w, off, grads, "mgda")
    o1 = out1.clone()
    _, out2, b2, _ = _resolve(w, off, grads, "mgda", res=res, out=out1)
    np.testing.assert_array_equal(b1, b2)
    assert torch.equal(o1, out2)
