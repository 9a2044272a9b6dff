"""GPU parity: the CUDA path (through the C ABI) against the fp64 oracle,
element by element, on seeded inputs that span several chunks per bucket,
ragged tails and unaligned bucket starts."""
import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2606_05613_gb300 import build as nb
from paper_2606_05613_gb300 import inputs
from paper_2606_05613_gb300 import native as bk
from tests.parity_util import Run, check_window, gram_close, oracle_window

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


def _workload(K, dt, sizes, bucket_elems, rho=(-0.3, 0.95), seed=0, flip=0.0):
    eb = 4 if dt == "f32" else 2
    base = inputs.gpt2_small()
    w = inputs.scaled(base, "parity-k%d-%s" % (K, dt), sizes, bucket_elems * eb)
    import dataclasses
    return dataclasses.replace(w, K=K, dtype=dt, rho_lo=rho[0], rho_hi=rho[1], seed=seed,
                               flip_frac=flip)


# ragged tensor list: several 32768-element chunks per bucket, odd sizes,
# bucket starts that are not multiples of 8 elements
RAGGED = [70001, 3, 131071, 5, 65536, 99999, 17, 40000, 1, 77777]


def _run(w, rule, out_dt, params=None, inplace=False):
    off = bk.bkmoo_plan(w.param_sizes, w.elem_bytes, w.bucket_bytes)
    np.testing.assert_array_equal(off, orc.plan(w.param_sizes, w.elem_bytes, w.bucket_bytes))
    grads = inputs.generate(w, off, DEV)
    hv = [inputs.host_view(g) for g in grads]
    B = len(off) - 1
    res = bk.Resolver(w.K, _tdt(w.dtype), off, DEV)
    out = grads[0] if inplace else torch.empty(int(off[-1]), dtype=_tdt(out_dt), device=DEV)
    beta = torch.full((B, w.K), float("nan"), dtype=torch.float32, device=DEV)
    status = torch.full((B,), -1, dtype=torch.int32, device=DEV)
    res.resolve(grads, rule, out, params=params, out_weights=beta, out_status=status)
    torch.cuda.synchronize()
    assert res.status() == 0
    return off, hv, out, beta.cpu().numpy(), status.cpu().numpy(), res


def _check_against_oracle(w, rule, off, hv, out, beta, status, out_dt, seed=0, step=0,
                          mgda_mode=orc.MGDA_EXACT, max_iter=256):
    """Every bucket against the oracle (PCGrad near ties: either branch)."""
    B = len(off) - 1
    run = Run(w.name, np.asarray(off, dtype=np.int64), rule, out, beta, status, out_dt,
              seed=seed, step=step, mgda_mode=mgda_mode, max_iter=max_iter)
    if B == 0:
        return 0.0
    ref = oracle_window(hv, run.off, 0, B, run)
    worst = check_window(hv, 0, B, ref, run)
    assert run.checked == B
    return worst


@pytest.mark.parametrize("dt", ["f32", "bf16"])
@pytest.mark.parametrize("K", [1, 2, 3, 4, 8, 16])
def test_gram_parity(K, dt):
    w = _workload(K, dt, RAGGED, 200000, seed=K)
    off = bk.bkmoo_plan(w.param_sizes, w.elem_bytes, w.bucket_bytes)
    grads = inputs.generate(w, off, DEV)
    hv = [inputs.host_view(g) for g in grads]
    B = len(off) - 1
    res = bk.Resolver(K, _tdt(dt), off, DEV)
    G = torch.empty(B, K, K, dtype=torch.float64, device=DEV)
    res.gram(grads, G)
    G1 = G.cpu().numpy()
    res.gram(grads, G)
    G2 = G.cpu().numpy()
    np.testing.assert_array_equal(G1, G2)            # run-to-run deterministic
    for b in range(B):
        lo, n = int(off[b]), int(off[b + 1] - off[b])
        ok, err = gram_close(G1[b], orc.gram(hv, lo, n))
        assert ok, (b, err)
        np.testing.assert_array_equal(G1[b], G1[b].T)


@pytest.mark.parametrize("rule", ["mgda", "pcgrad", "cagrad", "mean"])
@pytest.mark.parametrize("dt,out_dt", [("f32", "f32"), ("bf16", "bf16"), ("bf16", "f32"),
                                       ("f32", "bf16")])
@pytest.mark.parametrize("K", [2, 4, 8])
def test_resolve_parity(rule, dt, out_dt, K):
    w = _workload(K, dt, RAGGED, 150000, seed=10 + K, flip=0.2)
    p = bk.bkmoo_default_params()
    p.seed, p.step = 5, 9
    off, hv, out, beta, status, _ = _run(w, rule, out_dt, params=p)
    _check_against_oracle(w, rule, off, hv, out, beta, status, out_dt, seed=5, step=9)


@pytest.mark.parametrize("K", list(range(1, 17)))
def test_every_k_mgda_and_cagrad_f32(K):
    w = _workload(K, "f32", [300000, 7, 123457], 100000, seed=40 + K, rho=(-0.5, 0.9))
    for rule in ("mgda", "cagrad", "pcgrad"):
        off, hv, out, beta, status, _ = _run(w, rule, "f32")
        _check_against_oracle(w, rule, off, hv, out, beta, status, "f32")


@pytest.mark.parametrize("K", [2, 3, 5, 6, 8, 12, 16])
def test_opposed_language_cagrad_and_mgda(K):
    """One language sign-flipped in every bucket over a strong shared part:
    <g_k, g0> < 0 for that language, the case where 0 may lie in the hull
    (Eq. 4's dual is then minimised away from its kink in general)."""
    w = _workload(K, "f32", [200000, 9, 77777], 90000, seed=70 + K, rho=(0.6, 0.95), flip=1.0)
    for rule in ("cagrad", "mgda"):
        off, hv, out, beta, status, _ = _run(w, rule, "f32")
        _check_against_oracle(w, rule, off, hv, out, beta, status, "f32")


@pytest.mark.parametrize("rule", ["mgda", "pcgrad", "cagrad"])
def test_in_place_equals_out_of_place(rule):
    w = _workload(4, "bf16", RAGGED, 180000, seed=3)
    off, hv, out1, beta1, _, _ = _run(w, rule, "bf16")
    _, _, out2, beta2, _, _ = _run(w, rule, "bf16", inplace=True)
    np.testing.assert_array_equal(beta1, beta2)
    assert torch.equal(out1, out2)


def test_frank_wolfe_replay_without_polish():
    """Capped Frank-Wolfe (20 steps, no completion, no K=2 closed form) is the
    oracle's Frank-Wolfe replay."""
    w = _workload(8, "bf16", RAGGED, 120000, seed=77, flip=0.2)
    p = bk.bkmoo_default_params()
    p.max_iter, p.flags = 20, 0
    off, hv, out, beta, status, _ = _run(w, "mgda", "bf16", params=p)
    _check_against_oracle(w, "mgda", off, hv, out, beta, status, "bf16",
                          mgda_mode=orc.MGDA_FW, max_iter=20)


def test_tiny_k2_closed_form_vs_frank_wolfe():
    """K=2 closed form and Frank-Wolfe (+ completion) give the same weights on
    the four cosines -0.8, -0.2, 0.3, 0.9."""
    w = inputs.tiny()
    off, hv, out_cf, beta_cf, st, _ = _run(w, "mgda", "f32")
    assert len(off) == 5
    _check_against_oracle(w, "mgda", off, hv, out_cf, beta_cf, st, "f32")
    p = bk.bkmoo_default_params()
    p.flags = bk.BKMOO_FLAG_POLISH
    _, _, out_fw, beta_fw, st2, _ = _run(w, "mgda", "f32", params=p)
    np.testing.assert_allclose(beta_fw, beta_cf, atol=1e-6)
    ref = orc.resolve(hv, off, orc.MGDA, want_gram=True)
    for b in range(4):
        np.testing.assert_allclose(orc.mgda_k2(ref["gram"][b]), beta_cf[b], atol=1e-6)


def test_opposed_gradients_give_exact_zero():
    K, n = 2, 300001
    g = torch.randn(n, device=DEV)
    grads = [g.clone(), (-g).clone()]
    off = np.array([0, 100000, n], dtype=np.int64)
    res = bk.Resolver(K, torch.float32, off, DEV)
    out = torch.empty(n, device=DEV)
    beta = torch.empty(2, K, device=DEV)
    for rule in ("mgda", "cagrad"):
        res.resolve(grads, rule, out, out_weights=beta)
        torch.cuda.synchronize()
        assert torch.count_nonzero(out).item() == 0
        np.testing.assert_array_equal(beta.cpu().numpy(), np.full((2, 2), 0.5, dtype=np.float32))


def test_tiny_buckets_and_vector_edges():
    """Buckets shorter than one 16-byte vector and every head/tail length."""
    sizes = [1, 2, 3, 4, 5, 6, 7, 8, 9, 15, 16, 17, 31, 33, 1000, 8191, 8193]
    for dt in ("f32", "bf16"):
        w = _workload(3, dt, sizes, 1)      # one bucket per tensor (cap 1 element? no: see below)
        import dataclasses
        w = dataclasses.replace(w, bucket_bytes=w.elem_bytes * 9000)
        off = bk.bkmoo_plan(w.param_sizes, w.elem_bytes, w.bucket_bytes)
        # force one bucket per tensor
        off = np.concatenate([[0], np.cumsum(list(reversed(sizes)))]).astype(np.int64)
        grads = inputs.generate(w, off, DEV)
        hv = [inputs.host_view(g) for g in grads]
        B = len(off) - 1
        res = bk.Resolver(3, _tdt(dt), off, DEV)
        for rule in ("mgda", "pcgrad", "cagrad"):
            out = torch.empty(int(off[-1]), dtype=_tdt(dt), device=DEV)
            beta = torch.empty(B, 3, device=DEV)
            status = torch.empty(B, dtype=torch.int32, device=DEV)
            res.resolve(grads, rule, out, out_weights=beta, out_status=status)
            torch.cuda.synchronize()
            _check_against_oracle(w, rule, off, hv, out, beta.cpu().numpy(),
                                  status.cpu().numpy(), dt)
        G = torch.empty(B, 3, 3, dtype=torch.float64, device=DEV)
        res.gram(grads, G)
        Gc = G.cpu().numpy()
        for b in range(B):
            ok, err = gram_close(Gc[b], orc.gram(hv, int(off[b]), int(off[b + 1] - off[b])))
            assert ok, (dt, b, err)


def test_nonfinite_bucket_is_flagged():
    w = _workload(4, "f32", [50000, 60000, 70000], 60000, seed=5)
    off = bk.bkmoo_plan(w.param_sizes, w.elem_bytes, w.bucket_bytes)
    grads = inputs.generate(w, off, DEV)
    grads[2][int(off[1]) + 17] = float("nan")
    B = len(off) - 1
    res = bk.Resolver(4, torch.float32, off, DEV)
    out = torch.empty_like(grads[0])
    beta = torch.empty(B, 4, device=DEV)
    status = torch.empty(B, dtype=torch.int32, device=DEV)
    res.resolve(grads, "mgda", out, out_weights=beta, out_status=status)
    st = status.cpu().numpy()
    assert st[1] == bk.BKMOO_ERR_NONFINITE
    assert (np.delete(st, 1) == 0).all()
    np.testing.assert_array_equal(beta.cpu().numpy()[1], np.full(4, 0.25, dtype=np.float32))


def test_workspace_plan_mismatch_is_detected():
    w = _workload(2, "f32", [40000, 40000], 40000, seed=6)
    off = bk.bkmoo_plan(w.param_sizes, w.elem_bytes, w.bucket_bytes)
    grads = inputs.generate(w, off, DEV)
    res = bk.Resolver(2, torch.float32, off, DEV)
    other = np.array([0, 30000, 80000], dtype=np.int64)
    out = torch.full_like(grads[0], 7.0)
    status = torch.empty(2, dtype=torch.int32, device=DEV)
    bk.bkmoo_resolve(grads, other, "mgda", out, res.ws, out_status=status)
    assert bk.bkmoo_workspace_status(res.ws) == bk.BKMOO_ERR_WORKSPACE
    assert (status.cpu().numpy() == bk.BKMOO_ERR_WORKSPACE).all()
    assert bool((out == 7.0).all())
    # the right plan still works afterwards
    res.resolve(grads, "mgda", out)
    assert res.status() == 0


def test_zero_buckets_is_a_no_op():
    off = np.array([0], dtype=np.int64)
    res = bk.Resolver(3, torch.float32, off, DEV)
    g = [torch.empty(0, device=DEV) for _ in range(3)]
    out = torch.empty(16, device=DEV)
    bk.bkmoo_resolve([torch.empty(4, device=DEV) for _ in range(3)], off, "mgda", out, res.ws)
    assert res.status() == 0
    del g


def test_all_zero_bucket_gives_zero_direction():
    K, n = 4, 70000
    grads = [torch.zeros(n, device=DEV) for _ in range(K)]
    off = np.array([0, n], dtype=np.int64)
    res = bk.Resolver(K, torch.float32, off, DEV)
    out = torch.full((n,), 3.0, device=DEV)
    for rule in ("mgda", "pcgrad", "cagrad", "mean"):
        res.resolve(grads, rule, out)
        torch.cuda.synchronize()
        assert torch.count_nonzero(out).item() == 0


@pytest.mark.parametrize("dt", ["f32", "bf16"])
def test_global_variant_is_one_bucket(dt):
    """The conventional (global) MOO is the trivial partition into one bucket
    (Section 3.1; Table 2 compares the two): its Gram is the sum of the
    bucket Grams of any finer partition (inner products decompose over
    disjoint blocks), and its resolve matches the oracle's one-bucket
    resolve."""
    K = 4
    w = _workload(K, dt, RAGGED, 150000, seed=77, flip=0.3)
    off = bk.bkmoo_plan(w.param_sizes, w.elem_bytes, w.bucket_bytes)
    assert len(off) > 3
    grads = inputs.generate(w, off, DEV)
    hv = [inputs.host_view(g) for g in grads]
    N = int(off[-1])
    one = np.array([0, N], dtype=np.int64)
    Gb = torch.empty(len(off) - 1, K, K, dtype=torch.float64, device=DEV)
    bk.Resolver(K, _tdt(dt), off, DEV).gram(grads, Gb)
    res1 = bk.Resolver(K, _tdt(dt), one, DEV)
    G1 = torch.empty(1, K, K, dtype=torch.float64, device=DEV)
    res1.gram(grads, G1)
    ok, err = gram_close(G1.cpu().numpy()[0], Gb.cpu().numpy().sum(axis=0))
    assert ok, err
    for rule in ("mgda", "pcgrad", "cagrad"):
        out = torch.empty(N, dtype=_tdt(dt), device=DEV)
        beta = torch.empty(1, K, device=DEV)
        status = torch.empty(1, dtype=torch.int32, device=DEV)
        res1.resolve(grads, rule, out, out_weights=beta, out_status=status)
        torch.cuda.synchronize()
        _check_against_oracle(w, rule, one, hv, out, beta.cpu().numpy(), status.cpu().numpy(), dt)


@pytest.mark.parametrize("dt", ["f32", "bf16"])
def test_huge_buckets_group_reduction(dt):
    """Buckets of more than 1024 chunks (their chunk partials are pre-reduced
    in groups of 512 before the per-bucket sum): Gram and every rule against
    the oracle, with ragged last groups, a small bucket between two large
    ones, and bit-identical results run to run."""
    K = 3
    ch = 16384 if dt == "f32" else 32768
    sizes = [1025 * ch + 7, 5000, 2048 * ch + 3]          # 1026, 1 and 2049 chunks
    w = _workload(K, dt, sizes, 1)
    off = np.concatenate([[0], np.cumsum(list(reversed(sizes)))]).astype(np.int64)
    grads = inputs.generate(w, off, DEV)
    hv = [inputs.host_view(g) for g in grads]
    B = len(off) - 1
    res = bk.Resolver(K, _tdt(dt), off, DEV)
    G = torch.empty(B, K, K, dtype=torch.float64, device=DEV)
    res.gram(grads, G)
    G1 = G.cpu().numpy()
    res.gram(grads, G)
    np.testing.assert_array_equal(G1, G.cpu().numpy())
    for b in range(B):
        ok, err = gram_close(G1[b], orc.gram(hv, int(off[b]), int(off[b + 1] - off[b])))
        assert ok, (b, err)
    for rule in ("mgda", "pcgrad", "cagrad"):
        out = torch.empty(int(off[-1]), dtype=_tdt(dt), device=DEV)
        beta = torch.empty(B, K, device=DEV)
        status = torch.empty(B, dtype=torch.int32, device=DEV)
        res.resolve(grads, rule, out, out_weights=beta, out_status=status)
        torch.cuda.synchronize()
        assert res.status() == 0
        _check_against_oracle(w, rule, off, hv, out, beta.cpu().numpy(), status.cpu().numpy(), dt)


# ---------------------------------------------------------------------------
# fused path (BKMOO_FLAG_FUSED): one persistent launch per resolve
# ---------------------------------------------------------------------------

def _fused_params(seed=0, step=0, flags=None):
    p = bk.bkmoo_default_params()
    p.seed, p.step = seed, step
    p.flags = (p.flags if flags is None else flags) | bk.BKMOO_FLAG_FUSED
    return p


@pytest.mark.parametrize("rule", ["mgda", "pcgrad", "cagrad", "mean"])
@pytest.mark.parametrize("dt,out_dt", [("f32", "f32"), ("bf16", "bf16"), ("bf16", "f32")])
@pytest.mark.parametrize("K", [1, 2, 3, 4, 5, 8, 16])
def test_fused_resolve_parity(rule, dt, out_dt, K):
    w = _workload(K, dt, RAGGED, 150000, seed=60 + K, flip=0.2)
    off, hv, out, beta, status, _ = _run(w, rule, out_dt, params=_fused_params(5, 9))
    _check_against_oracle(w, rule, off, hv, out, beta, status, out_dt, seed=5, step=9)


def test_fused_tiny_buckets_and_empty_slices():
    """Buckets far smaller than the grid (most slices empty) and every
    head / tail length."""
    sizes = [1, 2, 3, 4, 5, 6, 7, 8, 9, 15, 16, 17, 31, 33, 1000, 8191, 8193, 300001]
    for dt in ("f32", "bf16"):
        w = _workload(3, dt, sizes, 400000)
        off = np.concatenate([[0], np.cumsum(list(reversed(sizes)))]).astype(np.int64)
        grads = inputs.generate(w, off, DEV)
        hv = [inputs.host_view(g) for g in grads]
        B = len(off) - 1
        res = bk.Resolver(3, _tdt(dt), off, DEV)
        for rule in ("mgda", "pcgrad", "cagrad"):
            out = torch.empty(int(off[-1]), dtype=_tdt(dt), device=DEV)
            beta = torch.empty(B, 3, device=DEV)
            status = torch.empty(B, dtype=torch.int32, device=DEV)
            res.resolve(grads, rule, out, params=_fused_params(), out_weights=beta,
                        out_status=status)
            torch.cuda.synchronize()
            assert res.status() == 0
            _check_against_oracle(w, rule, off, hv, out, beta.cpu().numpy(),
                                  status.cpu().numpy(), dt)


def test_fused_deterministic_and_matches_three_pass():
    w = _workload(4, "bf16", RAGGED * 3, 250000, seed=8)
    off, hv, out_f, beta_f, _, res = _run(w, "mgda", "f32", params=_fused_params())
    o1 = out_f.clone()
    grads = inputs.generate(w, off, DEV)
    res.resolve(grads, "mgda", out_f, params=_fused_params())
    torch.cuda.synchronize()
    assert torch.equal(o1, out_f)                     # run to run
    _, _, out_3, beta_3, _, _ = _run(w, "mgda", "f32")
    np.testing.assert_allclose(beta_f, beta_3, atol=1e-5)
    d3 = out_3.cpu().numpy().astype(np.float64)
    df = o1.cpu().numpy().astype(np.float64)
    assert np.linalg.norm(df - d3) <= 1e-5 * np.linalg.norm(d3)


@pytest.mark.parametrize("rule", ["mgda", "pcgrad", "cagrad", "mean"])
@pytest.mark.parametrize("dt", ["f32", "bf16"])
@pytest.mark.parametrize("K", [1, 2, 3, 4])
def test_fused_many_buckets_per_cluster(K, dt, rule):
    """Enough buckets that every cluster of the cluster kernel resolves a
    dozen or more in turn (its pipelined hand-offs: the next bucket's Gram
    streamed while the one before is solved), with ragged bucket sizes;
    every bucket against the oracle."""
    sizes = [7001 + 37 * i for i in range(260)]
    w = _workload(K, dt, sizes, 6000, seed=70 + K, flip=0.2)
    off, hv, out, beta, status, _ = _run(w, rule, dt, params=_fused_params(3, 4))
    assert len(off) - 1 >= 12 * 15
    _check_against_oracle(w, rule, off, hv, out, beta, status, dt, seed=3, step=4)


@pytest.mark.parametrize("K", [2, 4, 8])
def test_fused_in_place_equals_out_of_place(K):
    """In place (the direction written over the first gradient) the fused
    kernels give the bit-identical result: every output position is read,
    through its thread's own prefetch, by the thread that writes it, after
    every Gram read of the bucket."""
    w = _workload(K, "bf16", RAGGED * 2, 180000, seed=30 + K)
    off, hv, out1, beta1, _, _ = _run(w, "mgda", "bf16", params=_fused_params())
    _, _, out2, beta2, _, _ = _run(w, "mgda", "bf16", params=_fused_params(), inplace=True)
    np.testing.assert_array_equal(beta1, beta2)
    assert torch.equal(out1, out2)


def test_per_plan_path_runs_the_fused_kernel_where_chosen():
    """A plan for which bkmoo_resolve_path picks the cluster kernel (K = 4,
    2 MiB fp32 buckets) resolves by it by default: the result is the one of
    the forced fused path, bit for bit, and matches the oracle."""
    K = 4
    w = _workload(K, "f32", [3 * (1 << 19) + 12345], 1 << 19, seed=91)
    off = bk.bkmoo_plan(w.param_sizes, 4, w.bucket_bytes)
    assert bk.bkmoo_resolve_path(K, bk.BKMOO_F32, "mgda", off, 0) == 1
    _, hv, out_auto, beta_auto, st, _ = _run(w, "mgda", "f32")
    _, _, out_f, beta_f, _, _ = _run(w, "mgda", "f32", params=_fused_params())
    np.testing.assert_array_equal(beta_auto, beta_f)
    assert torch.equal(out_auto, out_f)
    _check_against_oracle(w, "mgda", off, hv, out_auto, beta_auto, st, "f32")


def test_fused_workspace_mismatch_is_detected():
    w = _workload(2, "f32", [40000, 40000], 40000, seed=6)
    off = bk.bkmoo_plan(w.param_sizes, w.elem_bytes, w.bucket_bytes)
    grads = inputs.generate(w, off, DEV)
    res = bk.Resolver(2, torch.float32, off, DEV)
    other = np.array([0, 30000, 80000], dtype=np.int64)
    out = torch.full_like(grads[0], 7.0)
    status = torch.empty(2, dtype=torch.int32, device=DEV)
    bk.bkmoo_resolve(grads, other, "mgda", out, res.ws, params=_fused_params(), out_status=status)
    assert bk.bkmoo_workspace_status(res.ws) == bk.BKMOO_ERR_WORKSPACE
    assert (status.cpu().numpy() == bk.BKMOO_ERR_WORKSPACE).all()
    assert bool((out == 7.0).all())
    res.resolve(grads, "mgda", out, params=_fused_params())
    assert res.status() == 0


def test_fused_bounded_wait_reports_timeout():
    """Failure detection without a fault: with bucket 0's coefficients never
    published (a flag that nothing sets), every wait of the persistent kernel
    ends after its bound, the call reports BKMOO_ERR_TIMEOUT through the
    workspace status word, and the context stays usable: the next resolve
    succeeds and matches the oracle."""
    import time
    w = _workload(4, "bf16", RAGGED, 150000, seed=23)
    off = bk.bkmoo_plan(w.param_sizes, w.elem_bytes, w.bucket_bytes)
    grads = inputs.generate(w, off, DEV)
    res = bk.Resolver(4, torch.bfloat16, off, DEV)
    out = torch.empty(int(off[-1]), dtype=torch.bfloat16, device=DEV)
    p = _fused_params(flags=bk.bkmoo_default_params().flags | bk.BKMOO_FLAG_TEST_WITHHOLD)
    t0 = time.time()
    res.resolve(grads, "mgda", out, params=p)
    assert res.status() == bk.BKMOO_ERR_TIMEOUT
    assert time.time() - t0 < 30.0
    B = len(off) - 1
    beta = torch.empty(B, 4, device=DEV)
    status = torch.empty(B, dtype=torch.int32, device=DEV)
    res.resolve(grads, "mgda", out, params=_fused_params(), out_weights=beta, out_status=status)
    torch.cuda.synchronize()
    assert res.status() == 0
    hv = [inputs.host_view(g) for g in grads]
    _check_against_oracle(w, "mgda", off, hv, out, beta.cpu().numpy(), status.cpu().numpy(), "bf16")


def test_cluster_bounded_exchange_wait_reports_timeout():
    """Failure detection in the cluster kernel without a fault: CTA 0 of
    every cluster withholds its first bucket's partial (a hand-off that
    never comes), each peer's exchange wait ends after its bound and every
    later wait at once, the call reports BKMOO_ERR_TIMEOUT, and the context
    stays usable: the next resolve succeeds and matches the oracle."""
    import time
    K = 4
    sizes = [7001 + 37 * i for i in range(260)]
    w = _workload(K, "f32", sizes, 6000, seed=29)
    off = bk.bkmoo_plan(w.param_sizes, w.elem_bytes, w.bucket_bytes)
    grads = inputs.generate(w, off, DEV)
    res = bk.Resolver(K, torch.float32, off, DEV)
    out = torch.empty(int(off[-1]), dtype=torch.float32, device=DEV)
    p = _fused_params(flags=bk.bkmoo_default_params().flags
                      | bk.BKMOO_FLAG_TEST_WITHHOLD_EXCHANGE)
    assert bk.bkmoo_resolve_path(K, bk.BKMOO_F32, "mgda", off, p.flags) == 1
    t0 = time.time()
    res.resolve(grads, "mgda", out, params=p)
    assert res.status() == bk.BKMOO_ERR_TIMEOUT
    assert time.time() - t0 < 30.0
    B = len(off) - 1
    beta = torch.empty(B, K, device=DEV)
    status = torch.empty(B, dtype=torch.int32, device=DEV)
    res.resolve(grads, "mgda", out, params=_fused_params(), out_weights=beta, out_status=status)
    torch.cuda.synchronize()
    assert res.status() == 0
    hv = [inputs.host_view(g) for g in grads]
    _check_against_oracle(w, "mgda", off, hv, out, beta.cpu().numpy(), status.cpu().numpy(), "f32")


@pytest.mark.parametrize("K", [2, 4, 8, 16])
def test_conflict_statistics(K):
    """Figure 1 statistics from the GPU Gram against the oracle's (cosines to
    the Gram tolerance; the conflict flag exactly, except where the most
    negative cosine is within that tolerance of 0)."""
    w = _workload(K, "bf16", RAGGED, 120000, seed=90 + K, rho=(-0.6, 0.9), flip=0.3)
    off = bk.bkmoo_plan(w.param_sizes, w.elem_bytes, w.bucket_bytes)
    grads = inputs.generate(w, off, DEV)
    hv = [inputs.host_view(g) for g in grads]
    B = len(off) - 1
    res = bk.Resolver(K, torch.bfloat16, off, DEV)
    G = torch.empty(B, K, K, dtype=torch.float64, device=DEV)
    res.gram(grads, G)
    cos = torch.empty(B, K, K, dtype=torch.float32, device=DEV)
    stats = torch.empty(B, 3, dtype=torch.float32, device=DEV)
    flag = torch.empty(B, dtype=torch.int32, device=DEV)
    bk.bkmoo_conflicts(G, cos, stats, flag)
    torch.cuda.synchronize()
    cos, stats, flag = cos.cpu().numpy(), stats.cpu().numpy(), flag.cpu().numpy()
    seen = 0
    for b in range(B):
        c_or, s_or, f_or = orc.conflicts(orc.gram(hv, int(off[b]), int(off[b + 1] - off[b])))
        np.testing.assert_allclose(cos[b], c_or, atol=2e-5)
        np.testing.assert_allclose(stats[b], s_or, atol=2e-5)
        if abs(s_or[2]) > 2e-5:
            assert flag[b] == f_or, b
        seen += f_or
    assert seen > 0          # the workload has conflicting buckets
