"""Pins of the fp64 oracle against what the paper and the mathematics fix.

None of these tests compare the oracle with itself: each checks it against a
hand-derived closed form (tests/golden), an invariant stated in the paper
(Theorem 3.1, Theorem 3.2, Eq. 5), a brute-force search on tiny inputs, a
literal materialised restatement of Algorithm 1, or an independent library
routine (numpy dot products).  CPU only.
"""
import itertools
import json
import math
import os

import numpy as np
import pytest

from oracle import oracle as orc
from paper_2606_05613_gb300 import inputs

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _golden(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


def _rand_vectors(rng, K, n, corr=0.0, flip_odd=False):
    s = rng.standard_normal(n)
    out = []
    for k in range(K):
        sign = (-1.0) ** k if flip_odd else 1.0
        out.append((sign * corr * s + math.sqrt(1 - corr * corr) * rng.standard_normal(n))
                   * math.exp(rng.standard_normal()))
    return out


def _gram_np(vs):
    X = np.stack(vs)
    return X @ X.T


def _f32(vs):
    return [np.ascontiguousarray(v, dtype=np.float32) for v in vs]


# ----------------------------------------------------------------------------
# Plan (Section 3.2, Figure 4 caption; rule R1)
# ----------------------------------------------------------------------------

def test_plan_hand_cases():
    for c in _golden("plan_cases.json")["cases"]:
        got = orc.plan(c["sizes"], c["elem_bytes"], c["bucket_bytes"])
        assert got.tolist() == c["offsets"], c


def test_plan_single_tensor_is_fixed_size_chunking():
    for n, cap in [(1, 1), (10, 3), (1 << 20, 1 << 18), (1_000_003, 4096)]:
        got = orc.plan([n], 1, cap)
        want = list(range(0, n, cap)) + [n]
        assert got.tolist() == want


def test_plan_model_bucket_counts():
    g = _golden("plan_cases.json")["model_bucket_counts"]
    assert len(orc.plan(inputs.gpt2_small_sizes(), 4, 25 * inputs.MiB)) - 1 == g["gpt2_small_f32_25mib"]
    assert len(orc.plan(inputs.llama32_1b_sizes(), 2, 25 * inputs.MiB)) - 1 == g["llama32_1b_bf16_25mib"]
    assert len(orc.plan(inputs.qwen3_8b_sizes(), 2, 25 * inputs.MiB)) - 1 == g["qwen3_8b_bf16_25mib"]
    for mib, nb in g["flat_1e9_f32"].items():
        assert len(orc.plan([1_000_000_000], 4, int(mib) * inputs.MiB)) - 1 == nb
    assert sum(inputs.gpt2_small_sizes()) == 124_439_808
    assert sum(inputs.llama32_1b_sizes()) == 1_235_814_400
    assert sum(inputs.qwen3_8b_sizes()) == 8_190_735_360


def test_plan_properties_random():
    """Partition of [0, N]; no bucket above cap; a boundary inside a tensor
    sits at a multiple of cap from the tensor's start; a bucket is closed only
    when the next piece would not fit."""
    rng = np.random.default_rng(1)
    for _ in range(300):
        n_t = int(rng.integers(1, 12))
        sizes = [int(x) for x in rng.integers(0, 40, size=n_t)]
        cap = int(rng.integers(1, 30))
        off = orc.plan(sizes, 1, cap)
        N = sum(sizes)
        if N == 0:
            assert off.tolist() == [0]
            continue
        assert off[0] == 0 and off[-1] == N
        lens = np.diff(off)
        assert (lens > 0).all() and (lens <= cap).all()
        bounds, _ = inputs.tensor_offsets_flat(sizes)
        starts = set(int(b) for b in bounds)
        for o in off[1:-1]:
            if o in starts:
                continue
            t = int(np.searchsorted(bounds, o, side="right") - 1)
            assert (o - bounds[t]) % cap == 0, (sizes, cap, off)
        # greedy: bucket b closed at a tensor start means that tensor's first
        # piece (min(size, cap)) would not fit in bucket b
        for b in range(len(off) - 2):
            o = int(off[b + 1])
            if o in starts:
                t = int(np.searchsorted(bounds, o, side="right") - 1)
                while bounds[t + 1] == bounds[t]:
                    t += 1
                first = min(int(bounds[t + 1] - bounds[t]), cap)
                assert lens[b] + first > cap, (sizes, cap, off)


def test_plan_invalid():
    with pytest.raises(ValueError):
        orc.plan([4], 0, 16)
    with pytest.raises(ValueError):
        orc.plan([4], 4, 3)
    with pytest.raises(ValueError):
        orc.plan([-1], 1, 3)


# ----------------------------------------------------------------------------
# Gram (inner products of Eq. 2 / Eq. 6 / Eq. 8; decomposition in the proofs)
# ----------------------------------------------------------------------------

def test_gram_matches_numpy_dot_f32():
    rng = np.random.default_rng(2)
    vs = _f32(_rand_vectors(rng, 5, 1001, corr=0.4))
    G = orc.gram(vs)
    Gn = _gram_np([v.astype(np.float64) for v in vs])
    np.testing.assert_allclose(G, Gn, rtol=1e-12, atol=1e-12 * np.abs(Gn).max())


def test_gram_bf16_widening_exact():
    import torch
    rng = np.random.default_rng(3)
    vs = _rand_vectors(rng, 3, 777)
    ts = [torch.tensor(v, dtype=torch.float32).to(torch.bfloat16) for v in vs]
    bits = [inputs.host_view(t) for t in ts]
    G = orc.gram(bits)
    Gn = _gram_np([t.to(torch.float64).numpy() for t in ts])
    np.testing.assert_allclose(G, Gn, rtol=1e-12, atol=1e-12 * np.abs(Gn).max())
    np.testing.assert_array_equal(orc.bf16_to_f64(bits[0]), ts[0].to(torch.float64).numpy())


def test_gram_additive_over_buckets_symmetric_psd():
    rng = np.random.default_rng(4)
    vs = _f32(_rand_vectors(rng, 6, 5000, corr=-0.3, flip_odd=True))
    off = orc.plan([1234, 2000, 1766], 4, 4 * 900)
    Gs = [orc.gram(vs, int(off[b]), int(off[b + 1] - off[b])) for b in range(len(off) - 1)]
    G = orc.gram(vs)
    np.testing.assert_allclose(sum(Gs), G, rtol=1e-12, atol=1e-10)
    for Gb in Gs + [G]:
        np.testing.assert_array_equal(Gb, Gb.T)
        ev = np.linalg.eigvalsh(Gb)
        assert ev.min() >= -1e-12 * np.trace(Gb)


# ----------------------------------------------------------------------------
# MGDA (Eq. 3, Eq. 6, Theorem 3.1)
# ----------------------------------------------------------------------------

def _obj(G, a):
    return float(a @ G @ a)


def test_mgda_golden_closed_forms():
    for c in _golden("mgda_closed_form.json")["cases"]:
        G = np.array(c["G"], dtype=np.float64)
        for solver in (orc.mgda_wolfe, orc.mgda_enum):
            a = solver(G)
            np.testing.assert_allclose(a, c["alpha"], atol=1e-12)
            assert abs(_obj(G, a) - c["min_sq_norm"]) <= 1e-12
        if G.shape[0] == 2:
            np.testing.assert_allclose(orc.mgda_k2(G), c["alpha"], atol=1e-15)
            a, _ = orc.mgda_fw(G, 0, 0.0)   # FW's pair init is the closed form
            np.testing.assert_allclose(a, c["alpha"], atol=1e-15)


def test_mgda_k2_closed_form_vs_brute_force_segment():
    rng = np.random.default_rng(5)
    gam = np.linspace(0.0, 1.0, 200001)
    for _ in range(40):
        g1, g2 = _rand_vectors(rng, 2, 7, corr=rng.uniform(-0.95, 0.95))
        G = _gram_np([g1, g2])
        a = orc.mgda_k2(G)
        vals = gam ** 2 * G[0, 0] + 2 * gam * (1 - gam) * G[0, 1] + (1 - gam) ** 2 * G[1, 1]
        i = int(np.argmin(vals))
        assert _obj(G, a) <= vals[i] + 1e-12 * G.max()
        assert abs(a[0] - gam[i]) <= 2e-5


def test_mgda_brute_force_grid_k3():
    """Simplex grid of step 1e-3 (about half a million points) on K = 3."""
    rng = np.random.default_rng(6)
    h = 1e-3
    t = np.arange(0, 1 + h / 2, h)
    A1, A2 = np.meshgrid(t, t, indexing="ij")
    m = A1 + A2 <= 1 + 1e-12
    a1, a2 = A1[m], A2[m]
    a3 = np.clip(1 - a1 - a2, 0, None)
    W = np.stack([a1, a2, a3], axis=1)
    for trial in range(12):
        vs = _rand_vectors(rng, 3, 5, corr=rng.uniform(-0.9, 0.9), flip_odd=bool(trial % 2))
        G = _gram_np(vs)
        a = orc.mgda_wolfe(G)
        vals = np.einsum("ni,ij,nj->n", W, G, W)
        j = int(np.argmin(vals))
        assert _obj(G, a) <= vals[j] + 1e-12 * np.trace(G)
        assert np.abs(W[j] - a).max() <= 0.02      # unique minimiser (G PD)
        assert abs(a.sum() - 1) < 1e-12 and (a >= 0).all()


@pytest.mark.parametrize("K", [3, 4, 5, 8, 12, 16])
def test_mgda_wolfe_vs_enumeration(K):
    rng = np.random.default_rng(100 + K)
    for trial in range(20):
        vs = _rand_vectors(rng, K, 3 * K, corr=rng.uniform(-0.9, 0.95), flip_odd=bool(trial % 3 == 0))
        G = _gram_np(vs)
        aw, ae = orc.mgda_wolfe(G), orc.mgda_enum(G)
        assert abs(_obj(G, aw) - _obj(G, ae)) <= 1e-12 * np.diag(G).max()
        np.testing.assert_allclose(aw, ae, atol=1e-7)


def _kkt_ok(G, a, eps):
    v = G @ a
    xx = float(a @ v)
    lo = (v >= xx - eps).all()
    on = all(abs(v[k] - xx) <= eps for k in range(len(a)) if a[k] > 1e-6)
    return lo and on


def test_mgda_kkt_invariant_theorem_3_1():
    """<g_k, d> >= ||d||^2 for every k, equality on the support (the
    inequality in the proof of Theorem 3.1), on materialised vectors."""
    rng = np.random.default_rng(7)
    for K in (2, 3, 4, 6, 8, 16):
        for trial in range(10):
            vs = _f32(_rand_vectors(rng, K, 400, corr=rng.uniform(-0.9, 0.95), flip_odd=bool(trial % 2)))
            G = orc.gram(vs)
            a = orc.mgda_k2(G) if K == 2 else orc.mgda_wolfe(G)
            d = orc.combine(vs, a)
            dots = np.array([np.dot(v.astype(np.float64), d) for v in vs])
            dd = float(d @ d)
            eps = 1e-9 * np.diag(G).max()
            assert (dots >= dd - eps).all()
            for k in range(K):
                if a[k] > 1e-6:
                    assert abs(dots[k] - dd) <= eps


def test_mgda_opposed_gives_zero_direction():
    """g2 = -g1: 0 is in the hull, alpha = (1/2, 1/2) and d = 0 exactly (the
    refined-Pareto-stationarity signal of Theorem 3.1 (a))."""
    rng = np.random.default_rng(8)
    g = rng.standard_normal(333).astype(np.float32)
    vs = [g, (-g).astype(np.float32)]
    G = orc.gram(vs)
    for a in (orc.mgda_k2(G), orc.mgda_wolfe(G), orc.mgda_enum(G), orc.mgda_fw(G, 10, 1e-12)[0]):
        np.testing.assert_array_equal(a, [0.5, 0.5])
        assert (orc.combine(vs, a) == 0).all()
    # K=4 with two opposed pairs: min norm 0
    h = rng.standard_normal(333).astype(np.float32)
    vs4 = [g, -g, h, -h]
    a = orc.mgda_wolfe(orc.gram(vs4))
    assert np.abs(orc.combine(vs4, a)).max() <= 1e-12


def test_mgda_degenerate_k1_zero_and_duplicates():
    np.testing.assert_array_equal(orc.mgda_wolfe(np.array([[3.0]])), [1.0])
    np.testing.assert_array_equal(orc.mgda_fw(np.array([[3.0]]), 5, 0.0)[0], [1.0])
    # all-zero bucket: any alpha gives d = 0; the weights stay on the simplex
    a = orc.mgda_wolfe(np.zeros((3, 3)))
    assert abs(a.sum() - 1) < 1e-15 and (a >= 0).all()
    # duplicated language: d equals the K=2 result of the distinct pair
    rng = np.random.default_rng(9)
    g1, g2 = _rand_vectors(rng, 2, 50, corr=-0.4, flip_odd=True)
    d2 = orc.mgda_k2(_gram_np([g1, g2]))
    d2v = d2[0] * g1 + d2[1] * g2
    vs = [g1, g2, g1]
    a = orc.mgda_wolfe(_gram_np(vs))
    np.testing.assert_allclose(a[0] * g1 + a[1] * g2 + a[2] * g1, d2v, atol=1e-10)


def test_mgda_frank_wolfe_monotone_and_converges():
    rng = np.random.default_rng(10)
    for K in (3, 4, 8):
        vs = _rand_vectors(rng, K, 40, corr=0.5)
        G = _gram_np(vs)
        prev = np.inf
        for it in (0, 1, 2, 4, 8, 16, 64, 256, 4096):
            a, done = orc.mgda_fw(G, it, 0.0)
            assert done <= it
            assert abs(a.sum() - 1) < 1e-12 and (a >= -1e-15).all()
            o = _obj(G, a)
            assert o <= prev + 1e-12 * G.max()
            prev = o
        ex = _obj(G, orc.mgda_wolfe(G))
        assert prev - ex <= 1e-4 * np.diag(G).max()


def test_theorem_3_1_bucket_level_global_descent():
    """Bucket-level MGDA: for every language, <g_t, d> >= ||d||^2 over the
    whole concatenated vector (Theorem 3.1 (b))."""
    rng = np.random.default_rng(11)
    K, sizes = 4, [300, 517, 120, 999, 64]
    N = sum(sizes)
    vs = _f32(_rand_vectors(rng, K, N, corr=0.2))
    # make one bucket strongly conflicting
    vs[1][:300] *= -1
    off = orc.plan(sizes, 4, 4 * 600)
    r = orc.resolve(vs, off, orc.MGDA)
    d = r["d"]
    for v in vs:
        assert float(np.dot(v.astype(np.float64), d)) >= float(d @ d) - 1e-9 * float(d @ d)


# ----------------------------------------------------------------------------
# PCGrad (Eq. 5, Eq. 8, the PCGrad branch of Algorithm 1)
# ----------------------------------------------------------------------------

_GOLD = 0x9E3779B97F4A7C15
_M64 = (1 << 64) - 1


def _mix64_py(z):
    z &= _M64
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & _M64
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & _M64
    return z ^ (z >> 31)


def test_splitmix64_published_sequence():
    """SplitMix64 seeded with 0 (state advanced by the golden gamma before
    each output) starts 0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4."""
    assert _mix64_py(1 * _GOLD) == 0xE220A8397B1DCDAF
    assert _mix64_py(2 * _GOLD) == 0x6E789E6AA1B965F4


def test_pcgrad_order_matches_definition_and_is_permutation():
    for K in (2, 3, 4, 8, 16):
        for t in range(K):
            for seed, step, b in [(0, 0, 0), (7, 3, 11), (2**63 + 5, 12345, 671)]:
                o = orc.pcgrad_order(seed, step, b, K, t)
                assert sorted(o) == [k for k in range(K) if k != t]
                k1 = _mix64_py(seed + (step + 1) * _GOLD)
                k2 = _mix64_py(k1 + (b + 1) * _GOLD)
                k3 = _mix64_py(k2 + (t + 1) * _GOLD)
                ref = [k for k in range(K) if k != t]
                for draw, i in enumerate(range(K - 2, 0, -1)):
                    r = _mix64_py(k3 + (draw + 1) * _GOLD)
                    j = r % (i + 1)
                    ref[i], ref[j] = ref[j], ref[i]
                assert o == ref


def test_pcgrad_order_roughly_uniform():
    K, t = 4, 0
    counts = {}
    n = 6000
    for b in range(n):
        o = tuple(orc.pcgrad_order(1, 2, b, K, t))
        counts[o] = counts.get(o, 0) + 1
    assert len(counts) == 6
    for c in counts.values():
        assert abs(c - n / 6) < 5 * math.sqrt(n / 6)


def _pcgrad_literal(vs, seed, step, bucket):
    """Algorithm 1's PCGrad branch on materialised vectors, in fp64."""
    K = len(vs)
    g = [v.astype(np.float64) for v in vs]
    out = np.zeros_like(g[0])
    for t in range(K):
        d = g[t].copy()
        for j in orc.pcgrad_order(seed, step, bucket, K, t):
            p = float(np.dot(d, g[j]))
            nn = float(np.dot(g[j], g[j]))
            if p < 0 and nn > 0:
                d = d - p / nn * g[j]
        out += d
    return out


def test_pcgrad_matches_literal_algorithm():
    rng = np.random.default_rng(12)
    for K in (2, 3, 4, 5, 8):
        for trial in range(8):
            vs = _f32(_rand_vectors(rng, K, 64, corr=rng.uniform(-0.8, 0.8), flip_odd=bool(trial % 2)))
            G = orc.gram(vs)
            beta, ties = orc.pcgrad(G, 5, trial, 3)
            assert ties == 0
            d = orc.combine(vs, beta)
            ref = _pcgrad_literal(vs, 5, trial, 3)
            np.testing.assert_allclose(d, ref, rtol=1e-9, atol=1e-9 * np.abs(ref).max())


def test_pcgrad_golden_and_k2_properties():
    for c in _golden("pcgrad_cagrad_closed_form.json")["pcgrad"]["cases"]:
        beta, _ = orc.pcgrad(np.array(c["G"], dtype=np.float64), 0, 0, 0)
        np.testing.assert_allclose(beta, c["beta"], atol=1e-15)
    rng = np.random.default_rng(13)
    for _ in range(20):
        g1, g2 = _rand_vectors(rng, 2, 30, corr=0.8, flip_odd=True)
        G = _gram_np([g1, g2])
        assert G[0, 1] < 0
        beta, _ = orc.pcgrad(G, 0, 0, 0)
        d1 = g1 - G[0, 1] / G[1, 1] * g2
        d2 = g2 - G[0, 1] / G[0, 0] * g1
        assert abs(np.dot(d1, g2)) < 1e-9 * G.max() and abs(np.dot(d2, g1)) < 1e-9 * G.max()
        assert np.dot(d1, d2) >= -1e-9 * G.max()      # post-PCGrad dots non-negative
        np.testing.assert_allclose(beta[0] * g1 + beta[1] * g2, d1 + d2, atol=1e-9)


def test_pcgrad_no_conflict_is_plain_sum():
    rng = np.random.default_rng(14)
    for K in (3, 6):
        vs = [np.abs(v) for v in _rand_vectors(rng, K, 50)]
        beta, _ = orc.pcgrad(_gram_np(vs), 1, 1, 1)
        np.testing.assert_array_equal(beta, np.ones(K))


def _pcgrad_literal_all(vs, seed, step, bucket):
    """Algorithm 1's PCGrad branch on materialised fp64 vectors, taking both
    outcomes of every conflict test that lies within the near-tie bound
    |<d_t, g_j>| <= 1e-6 ||d_t|| ||g_j||: every direction d it can return."""
    K = len(vs)
    g = [v.astype(np.float64) for v in vs]

    def walk(d, order, q):
        if q == len(order):
            return [d]
        j = order[q]
        p = float(np.dot(d, g[j]))
        nn = float(np.dot(g[j], g[j]))
        tie = abs(p) <= 1e-6 * math.sqrt(float(np.dot(d, d)) * nn)
        if tie and nn > 0:
            return walk(d - p / nn * g[j], order, q + 1) + walk(d, order, q + 1)
        if p < 0 and nn > 0:
            d = d - p / nn * g[j]
        return walk(d, order, q + 1)

    per_task = [walk(g[t].copy(), orc.pcgrad_order(seed, step, bucket, K, t), 0)
                for t in range(K)]
    return [sum(ds) for ds in itertools.product(*per_task)]


def test_pcgrad_alternatives_without_ties_is_pcgrad():
    rng = np.random.default_rng(16)
    for K in (2, 3, 5, 8, 16):
        for trial in range(6):
            G = _gram_np(_rand_vectors(rng, K, 3 * K, corr=rng.uniform(-0.8, 0.8),
                                       flip_odd=bool(trial % 2)))
            beta, ties = orc.pcgrad(G, 2, trial, 11)
            alts = orc.pcgrad_alternatives(G, 2, trial, 11)
            if ties == 0:
                assert alts.shape == (1, K)
                np.testing.assert_array_equal(alts[0], beta)


def test_pcgrad_alternatives_match_literal_at_near_ties():
    """Knife-edge conflicts (a pair whose inner product is a tiny multiple of
    the norms, of either sign): the set of PCGrad results over both branches
    of each near tie equals the set of directions that Algorithm 1 on the
    materialised vectors gives with the tied tests taken either way."""
    rng = np.random.default_rng(17)
    seen_multi = 0
    for K in (2, 3, 4, 6):
        for trial in range(8):
            n = 4 * K
            vs = _rand_vectors(rng, K, n, corr=rng.uniform(-0.6, 0.6), flip_odd=bool(trial % 2))
            # make (0, 1) a near-orthogonal pair: remove the component of g1
            # along g0, then add back a tiny multiple (sign by trial)
            g0, g1 = vs[0], vs[1]
            g1 = g1 - np.dot(g1, g0) / np.dot(g0, g0) * g0
            eps = (1e-9 if trial % 4 < 2 else -1e-9) * np.linalg.norm(g1) / np.linalg.norm(g0)
            vs[1] = g1 + eps * g0
            G = _gram_np(vs)
            beta, ties = orc.pcgrad(G, 3, trial, 5)
            alts = orc.pcgrad_alternatives(G, 3, trial, 5)
            X = np.stack(vs)
            got = [a @ X for a in alts]
            ref = _pcgrad_literal_all(vs, 3, trial, 5)
            scale = np.abs(X).max() * K
            for d in ref:                       # every literal outcome is an alternative
                assert min(np.abs(d - e).max() for e in got) <= 1e-9 * scale
            for e in got:                       # and every alternative is a literal outcome
                assert min(np.abs(d - e).max() for d in ref) <= 1e-9 * scale
            assert any(np.abs(beta - a).max() <= 1e-12 for a in alts)
            assert (len(alts) > 1) <= (ties > 0)
            seen_multi += len(alts) > 1
    assert seen_multi >= 8


# ----------------------------------------------------------------------------
# CAGrad (Eq. 4, Eq. 7, Theorem 3.2)
# ----------------------------------------------------------------------------

def _F(G, w, c):
    K = len(w)
    b = G.sum(axis=1) / K
    g0 = math.sqrt(max(G.sum() / K / K, 0.0))
    return float(b @ w) + c * g0 * math.sqrt(max(float(w @ G @ w), 0.0))


def test_cagrad_golden_closed_forms():
    for c in _golden("pcgrad_cagrad_closed_form.json")["cagrad"]["cases"]:
        beta, _ = orc.cagrad(np.array(c["G"], dtype=np.float64), c["c"])
        np.testing.assert_allclose(beta, c["beta"], atol=1e-12)


def test_cagrad_c0_is_mean_and_k1():
    rng = np.random.default_rng(15)
    for K in (2, 4, 7):
        G = _gram_np(_rand_vectors(rng, K, 30, corr=0.1))
        beta, _ = orc.cagrad(G, 0.0)
        np.testing.assert_array_equal(beta, np.full(K, 1.0 / K))
    beta, _ = orc.cagrad(np.array([[2.5]]), 0.3)
    np.testing.assert_allclose(beta, [1.3], atol=1e-15)


def _cagrad_certificate(vs, c):
    """Optimality certificate of the oracle's CAGrad answer on materialised
    vectors (Eq. 4 / Eq. 7): d = beta X is feasible with the constraint
    active, w lies on the simplex, and the primal value min_k <g_k, d> equals
    the dual value F(w) (by weak duality min_k <g_k, d> <= F(w') for every
    feasible d and every w' on the simplex, so equality proves both optimal);
    plus the bound of Theorem 3.2 (a)."""
    G = _gram_np(vs)
    beta, w = orc.cagrad(G, c)
    X = np.stack(vs)
    d = beta @ X
    g0 = X.mean(axis=0)
    n0 = float(np.linalg.norm(g0))
    assert (w >= 0).all() and abs(w.sum() - 1) <= 1e-12
    assert abs(np.linalg.norm(d - g0) - c * n0) <= 1e-9 * n0
    prim = min(float(np.dot(v, d)) for v in vs)
    dual = _F(G, w, c)
    assert abs(prim - dual) <= 1e-9 * np.diag(G).max()
    assert float(np.dot(g0, d)) >= (1 - c * c) / 2 * n0 * n0 - 1e-9 * n0 * n0
    return G, w


@pytest.mark.parametrize("K", [2, 3, 4, 6, 8, 12, 16])
def test_cagrad_primal_properties(K):
    """Constraint active, zero duality gap and Theorem 3.2 (a) on random
    materialised vectors, aligned or with the shared part flipped on odd
    languages."""
    rng = np.random.default_rng(20 + K)
    for trial in range(15):
        c = [0.5, 0.2, 0.9][trial % 3]
        vs = _rand_vectors(rng, K, 5 * K, corr=rng.uniform(-0.9, 0.9), flip_odd=bool(trial % 2))
        _cagrad_certificate(vs, c)


@pytest.mark.parametrize("K", [3, 5, 8, 12, 16])
def test_cagrad_opposed_language_certificate(K):
    """One language sign-flipped over a strong shared part (<g_k, g0> < 0 for
    it, the GPU parity workload's conflict case): the same certificate, and
    the dual minimiser beats random points of the simplex (Dirichlet draws,
    dense and sparse)."""
    rng = np.random.default_rng(60 + K)
    done = 0
    for trial in range(12):
        vs = _rand_vectors(rng, K, 6 * K, corr=rng.uniform(0.6, 0.95))
        k = int(rng.integers(K))
        vs[k] = -vs[k]
        g0 = np.stack(vs).mean(axis=0)
        if np.dot(vs[k], g0) >= 0:      # the flipped language dominates the mean
            continue
        done += 1
        G, w = _cagrad_certificate(vs, 0.5)
        Fw = _F(G, w, 0.5)
        for alpha in (1.0, 0.1):
            W = rng.dirichlet(np.full(K, alpha), size=20000)
            b = G.sum(axis=1) / K
            g0n = math.sqrt(G.sum() / K / K)
            vals = W @ b + 0.5 * g0n * np.sqrt(np.clip(np.einsum("ni,ij,nj->n", W, G, W), 0, None))
            assert Fw <= vals.min() + 1e-12 * np.diag(G).max()
    assert done >= 4


def test_cagrad_primal_brute_force_low_dimension():
    """In R^3 the feasible set is a ball: no point of a dense sphere of radius
    c||g0|| around g0 beats the oracle's direction on min_k <g_k, d>."""
    rng = np.random.default_rng(30)
    n_s = 400000
    u = rng.standard_normal((n_s, 3))
    u /= np.linalg.norm(u, axis=1, keepdims=True)
    for trial in range(10):
        K = 2 + trial % 2
        vs = [rng.standard_normal(3) for _ in range(K)]
        if trial % 3 == 0:
            vs[1] = -0.7 * vs[0] + 0.3 * rng.standard_normal(3)
        c = 0.5
        G = _gram_np(vs)
        beta, _ = orc.cagrad(G, c)
        X = np.stack(vs)
        d = beta @ X
        g0 = X.mean(axis=0)
        r = c * np.linalg.norm(g0)
        cand = g0 + r * u
        best = (cand @ X.T).min(axis=1).max()
        mine = (X @ d).min()
        assert mine >= best - 1e-9
        assert mine - best <= 5e-3 * r * np.abs(X).max() * 3      # grid is dense


def test_cagrad_dual_brute_force_grid_k3():
    rng = np.random.default_rng(31)
    h = 2e-3
    t = np.arange(0, 1 + h / 2, h)
    A1, A2 = np.meshgrid(t, t, indexing="ij")
    m = A1 + A2 <= 1 + 1e-12
    W = np.stack([A1[m], A2[m], np.clip(1 - A1[m] - A2[m], 0, None)], axis=1)
    for trial in range(8):
        vs = _rand_vectors(rng, 3, 6, corr=rng.uniform(-0.9, 0.9), flip_odd=bool(trial % 2))
        G = _gram_np(vs)
        _, w = orc.cagrad(G, 0.5)
        Fw = _F(G, w, 0.5)
        b = G.sum(axis=1) / 3
        g0 = math.sqrt(G.sum() / 9)
        vals = W @ b + 0.5 * g0 * np.sqrt(np.clip(np.einsum("ni,ij,nj->n", W, G, W), 0, None))
        assert Fw <= vals.min() + 1e-12 * np.diag(G).max()


def test_cagrad_zero_mean_gives_zero_direction():
    """g0 = 0 (Theorem 3.2 (b)): d = 0."""
    rng = np.random.default_rng(32)
    g = rng.standard_normal(100).astype(np.float32)
    vs = [g, (-g).astype(np.float32)]
    beta, _ = orc.cagrad(orc.gram(vs), 0.5)
    np.testing.assert_array_equal(beta, [0.5, 0.5])
    assert (orc.combine(vs, beta) == 0).all()


def test_theorem_3_2_bucket_level_average_descent():
    rng = np.random.default_rng(33)
    K, sizes, c = 3, [200, 333, 150, 90], 0.5
    vs = _f32(_rand_vectors(rng, K, sum(sizes), corr=0.3))
    vs[2][200:533] *= -1
    off = orc.plan(sizes, 4, 4 * 350)
    r = orc.resolve(vs, off, orc.CAGRAD, cagrad_c=c)
    g0 = np.mean([v.astype(np.float64) for v in vs], axis=0)
    assert float(g0 @ r["d"]) >= (1 - c * c) / 2 * float(g0 @ g0) - 1e-9 * float(g0 @ g0)


# ----------------------------------------------------------------------------
# Combination and the whole path
# ----------------------------------------------------------------------------

def test_combine_matches_numpy_and_bf16():
    import torch
    rng = np.random.default_rng(34)
    vs = _f32(_rand_vectors(rng, 4, 999))
    beta = rng.standard_normal(4)
    np.testing.assert_allclose(orc.combine(vs, beta),
                               beta @ np.stack([v.astype(np.float64) for v in vs]), rtol=1e-13, atol=1e-13)
    ts = [torch.tensor(v).to(torch.bfloat16) for v in vs]
    bits = [inputs.host_view(t) for t in ts]
    ref = beta @ np.stack([t.to(torch.float64).numpy() for t in ts])
    np.testing.assert_allclose(orc.combine(bits, beta, 10, 500), ref[10:510], rtol=1e-13, atol=1e-13)


def test_resolve_consistent_with_steps_and_nonfinite_policy():
    rng = np.random.default_rng(35)
    K, sizes = 3, [100, 250, 61]
    vs = _f32(_rand_vectors(rng, K, sum(sizes), corr=-0.5, flip_odd=True))
    vs[1][5] = np.nan
    off = orc.plan(sizes, 4, 4 * 200)
    for rule in (orc.MGDA, orc.PCGRAD, orc.CAGRAD, orc.MEAN):
        r = orc.resolve(vs, off, rule, want_gram=True, seed=3, step=4)
        for b in range(len(off) - 1):
            lo, n = int(off[b]), int(off[b + 1] - off[b])
            G = r["gram"][b]
            if r["status"][b] == 3:
                assert not np.isfinite(G).all()
                np.testing.assert_array_equal(r["beta"][b], np.full(K, 1 / K))
                continue
            np.testing.assert_array_equal(G, orc.gram(vs, lo, n))
            if rule == orc.MGDA:
                want = orc.mgda_wolfe(G)
            elif rule == orc.PCGRAD:
                want, _ = orc.pcgrad(G, 3, 4, b)
            elif rule == orc.CAGRAD:
                want, _ = orc.cagrad(G, 0.5)
            else:
                want = np.full(K, 1 / K)
            np.testing.assert_allclose(r["beta"][b], want, rtol=0, atol=1e-15)
            np.testing.assert_allclose(r["d"][lo:lo + n], orc.combine(vs, want, lo, n), rtol=0, atol=0)
        assert r["status"][0] == 3 and (r["status"][1:] == 0).all()


def test_resolve_threads_do_not_change_results():
    rng = np.random.default_rng(36)
    vs = _f32(_rand_vectors(rng, 4, 20000, corr=0.3))
    off = orc.plan([20000], 4, 4 * 1500)
    r1 = orc.resolve(vs, off, orc.MGDA, n_threads=1)
    r4 = orc.resolve(vs, off, orc.MGDA, n_threads=4)
    np.testing.assert_array_equal(r1["beta"], r4["beta"])
    np.testing.assert_array_equal(r1["d"], r4["d"])


def test_synthetic_cosines_of_tiny_workload():
    """The tiny workload's generator hits the pairwise cosines it names."""
    import torch
    w = inputs.tiny()
    off = orc.plan(w.param_sizes, w.elem_bytes, w.bucket_bytes)
    assert off.tolist() == [0, 262144, 524288, 786432, 1048576]
    gs = inputs.generate(w, off, "cpu")
    vs = [inputs.host_view(g) for g in gs]
    for b, cos in enumerate(inputs.TINY_COSINES):
        G = orc.gram(vs, int(off[b]), int(off[b + 1] - off[b]))
        assert abs(G[0, 1] / math.sqrt(G[0, 0] * G[1, 1]) - cos) < 0.01


def test_mgda_frank_wolfe_step_is_exact_line_search():
    """One Frank-Wolfe step moves from the pair start towards the vertex of
    least gradient to the minimiser along that segment (brute-force search)."""
    rng = np.random.default_rng(37)
    gam = np.linspace(0.0, 1.0, 100001)
    for trial in range(30):
        K = 3 + trial % 4
        G = _gram_np(_rand_vectors(rng, K, 2 * K, corr=rng.uniform(-0.5, 0.9)))
        a0, _ = orc.mgda_fw(G, 0, 0.0)
        a1, done = orc.mgda_fw(G, 1, -1.0)
        if done == 0:
            continue
        t = int(np.argmin(G @ a0))
        e = np.zeros(K)
        e[t] = 1.0
        path = (1 - gam)[:, None] * a0[None, :] + gam[:, None] * e[None, :]
        vals = np.einsum("ni,ij,nj->n", path, G, path)
        j = int(np.argmin(vals))
        assert _obj(G, a1) <= vals[j] + 1e-12 * G.max()
        assert np.abs(a1 - path[j]).max() <= 2e-5


# ----------------------------------------------------------------------------
# Conflict statistics (Figure 1; Eq. 2, Definition A.4)
# ----------------------------------------------------------------------------

def test_conflicts_closed_forms():
    e1, e2 = np.array([1.0, 0, 0]), np.array([0, 1.0, 0])
    cos, st, flag = orc.conflicts(_gram_np([e1, e2]))          # orthogonal
    np.testing.assert_allclose(cos, np.eye(2), atol=1e-15)
    assert flag == 0 and st[0] == 0 and st[1] == 0 and st[2] == 0
    cos, st, flag = orc.conflicts(_gram_np([e1, -2 * e1]))     # opposed
    assert abs(cos[0, 1] + 1) < 1e-15 and flag == 1 and abs(st[2] + 1) < 1e-15
    cos, st, flag = orc.conflicts(_gram_np([e1, 3 * e1, e2]))  # 1, 0, 0
    np.testing.assert_allclose(st, [1 / 3, np.sqrt(2) / 3, 0.0], atol=1e-15)
    assert flag == 0
    cos, st, flag = orc.conflicts(_gram_np([e1, np.zeros(3), -e1]))   # zero gradient
    assert cos[1, 1] == 0 and cos[0, 1] == 0 and flag == 1


def test_conflicts_match_materialised_cosines():
    rng = np.random.default_rng(40)
    for K in (2, 3, 4, 8, 16):
        vs = _rand_vectors(rng, K, 50, corr=rng.uniform(-0.9, 0.9), flip_odd=True)
        cos, st, flag = orc.conflicts(_gram_np(vs))
        X = np.stack(vs)
        C = (X @ X.T) / np.outer(np.linalg.norm(X, axis=1), np.linalg.norm(X, axis=1))
        np.testing.assert_allclose(cos, C, atol=1e-12)
        pairs = C[np.triu_indices(K, 1)]
        np.testing.assert_allclose(st, [pairs.mean(), pairs.std(), pairs.min()], atol=1e-12)
        assert flag == int((pairs < 0).any())
