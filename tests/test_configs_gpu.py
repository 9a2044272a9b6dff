"""Full-size workloads on the GPU, in the launch configuration the benchmark
times: every bucket is resolved on the device, and EVERY bucket of every
rule (and path) is compared with the oracle: the gradients are streamed to
the host in windows of whole buckets, the oracle resolves each window on all
host cores, and each bucket's beta and direction are checked against it
(tests/parity_util.py holds the tolerances).  MGDA's simplex and optimality
inequality are also checked on every bucket's GPU Gram."""
import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2606_05613_gb300 import build as nb
from paper_2606_05613_gb300 import inputs
from paper_2606_05613_gb300 import native as bk
from tests.parity_util import Run, compare_all, gram_close, window_bounds

pytestmark = pytest.mark.gpu

DEV = torch.device("cuda:0")
HOST_WINDOW_BYTES = 4 << 30        # gradient bytes streamed to the host per window


@pytest.fixture(scope="module", autouse=True)
def _built():
    nb.build()
    bk.load()
    orc.build()


def _tdt(dt):
    return torch.float32 if dt == "f32" else torch.bfloat16


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


def _resolve(w, off, grads, rule, params=None, res=None, out_dt=None):
    B = len(off) - 1
    if res is None:
        res = bk.Resolver(w.K, _tdt(w.dtype), off, DEV)
    out = torch.empty(int(off[-1]), dtype=_tdt(out_dt or w.dtype), device=DEV)
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


def _bounds(w, off, min_buckets=16):
    """Windows of at least 16 buckets (the oracle runs buckets in parallel
    over the host cores), otherwise of at most HOST_WINDOW_BYTES."""
    return window_bounds(off, HOST_WINDOW_BYTES // (w.K * w.elem_bytes), min_buckets)


def test_gpt2_small_k4_f32_mgda_pcgrad():
    w = inputs.gpt2_small()
    off, grads = _setup(w)
    assert len(off) - 1 == 22
    runs = []
    res = None
    for rule in ("mgda", "pcgrad"):
        p = bk.bkmoo_default_params()
        p.seed, p.step = 123, 7
        res, out, beta, st = _resolve(w, off, grads, rule, p, res=res)
        runs.append(Run("gpt2-" + rule, off, rule, out, beta, st, "f32", seed=123, step=7))
    G = _gram_all(res, grads, w, off)
    _mgda_properties(G, runs[0].beta)
    for b in range(len(off) - 1):
        lo, hi = int(off[b]), int(off[b + 1])
        hv = [inputs.host_view(g[lo:hi]) for g in grads]
        ok, err = gram_close(G[b], orc.gram(hv))
        assert ok, (b, err)
    compare_all(grads, runs, _bounds(w, off))


def test_llama32_1b_k8_bf16_mgda_fw20():
    w = inputs.llama32_1b()
    off, grads = _setup(w)
    B = len(off) - 1
    assert B == 134
    draws = inputs.bucket_draws(w, off)
    assert int((draws.flip >= 0).sum()) == round(0.1 * B)
    # <= 20 Frank-Wolfe steps, then the exact completion: the exact minimiser
    p = bk.bkmoo_default_params()
    p.max_iter = 20
    res, out, beta, st = _resolve(w, off, grads, "mgda", p)
    assert (st == 0).all()
    _mgda_properties(_gram_all(res, grads, w, off), beta)
    runs = [Run("llama-fw20+completion", off, "mgda", out, beta, st, "bf16")]
    # <= 20 Frank-Wolfe steps alone: the oracle's Frank-Wolfe replay
    p.flags = 0
    _, out2, beta2, st2 = _resolve(w, off, grads, "mgda", p, res=res)
    runs.append(Run("llama-fw20", off, "mgda", out2, beta2, st2, "bf16",
                    mgda_mode=orc.MGDA_FW, max_iter=20))
    compare_all(grads, runs, _bounds(w, off))


def test_qwen3_8b_k4_bf16_mgda_cagrad():
    w = inputs.qwen3_8b()
    off, grads = _setup(w)
    B = len(off) - 1
    assert B == 672
    draws = inputs.bucket_draws(w, off)
    assert int((draws.rho < 0).sum()) == round(0.02 * B)
    res = None
    runs = []
    for fused in (False, True):
        for rule in ("mgda", "cagrad"):
            p = bk.bkmoo_default_params()
            if fused:
                p.flags |= bk.BKMOO_FLAG_FUSED
            res, out, beta, st = _resolve(w, off, grads, rule, p, res=res)
            assert (st == 0).all(), np.unique(st, return_counts=True)
            runs.append(Run("qwen-%s-%s" % (rule, "fused" if fused else "3pass"), off, rule, out,
                            beta, st, "bf16"))
            if rule == "mgda" and not fused:
                _mgda_properties(_gram_all(res, grads, w, off), beta)
    compare_all(grads, runs, _bounds(w, off))


@pytest.mark.parametrize("K", inputs.SWEEP_K)
def test_sweep_1e9_f32(K):
    """1e9-element fp32 vector, every bucket size and rule; the data is drawn
    once (on the 100 MiB partition) and resolved under each partition; the
    windows follow the 100 MiB partition, whose boundaries are boundaries of
    every finer one."""
    w100 = inputs.sweep(K, 100)
    gen_off = orc.plan(w100.param_sizes, 4, w100.bucket_bytes)
    grads = inputs.generate(w100, gen_off, DEV)
    runs = []
    for mib in inputs.SWEEP_BUCKET_MIB:
        w = inputs.sweep(K, mib)
        off = bk.bkmoo_plan(w.param_sizes, 4, w.bucket_bytes)
        np.testing.assert_array_equal(off, orc.plan(w.param_sizes, 4, w.bucket_bytes))
        res = bk.Resolver(K, torch.float32, off, DEV)
        for rule in ("mgda", "pcgrad", "cagrad"):
            p = bk.bkmoo_default_params()
            p.seed, p.step = 9, mib
            _, out, beta, st = _resolve(w, off, grads, rule, p, res=res)
            runs.append(Run("sweep-k%d-%dmib-%s" % (K, mib, rule), off, rule, out, beta, st,
                            "f32", seed=9, step=mib))
        del res
    compare_all(grads, runs, _bounds(w100, gen_off))
    del grads, runs


def test_deterministic_full_size_step():
    """Two resolves of the same full-size input give bit-identical outputs."""
    w = inputs.gpt2_small()
    off, grads = _setup(w)
    res, out1, b1, _ = _resolve(w, off, grads, "mgda")
    _, out2, b2, _ = _resolve(w, off, grads, "mgda", res=res)
    np.testing.assert_array_equal(b1, b2)
    assert torch.equal(out1, out2)
