"""Per-bucket resolve during the backward pass (Algorithm 1, Figure 4):
the bucket layout on the CPU, and on the GPU the K per-language gradients
written by autograd straight into the flat buffers, each bucket resolved by
bkmoo_resolve_buckets as it completes, bit-identical to one bkmoo_resolve
over the whole plan and within tolerance of the oracle."""
import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2606_05613_gb300 import build as nb
from paper_2606_05613_gb300 import native as bk
from paper_2606_05613_gb300.hook import BucketMOO, bucket_layout


@pytest.fixture(scope="module", autouse=True)
def _built():
    nb.build()
    bk.load()
    orc.build()


def test_bucket_layout_reverse_order_and_spans():
    sizes = [10, 0, 25, 7, 3]             # registration order
    L = bucket_layout(sizes, 4, 4 * 12)   # 12-element buckets
    # flat order: 3 (idx 4), 7 (idx 3), 25 (idx 2), 10 (idx 0)
    assert L.starts == [35, 35, 10, 3, 0]
    np.testing.assert_array_equal(L.offsets, orc.plan(sizes, 4, 48))
    # the 25-element tensor fills two whole buckets; its last element opens
    # the bucket that the 10-element tensor then joins
    np.testing.assert_array_equal(L.offsets, [0, 10, 22, 34, 45])
    assert L.first[4] == 0 and L.last[4] == 0
    assert L.first[3] == 0 and L.last[3] == 0
    assert (L.first[2], L.last[2]) == (1, 3)
    assert (L.first[0], L.last[0]) == (3, 3)
    assert L.first[1] == -1
    assert L.need == [2, 1, 1, 2]


def test_bucket_layout_random_lists_cover_each_bucket():
    rng = np.random.default_rng(5)
    for _ in range(200):
        sizes = [int(x) for x in rng.integers(0, 50, size=rng.integers(1, 12))]
        if sum(sizes) == 0:
            continue
        cap = int(rng.integers(1, 60))
        L = bucket_layout(sizes, 2, 2 * cap)
        covered = np.zeros(L.n_elems, dtype=int)
        for i, n in enumerate(sizes):
            covered[L.starts[i]:L.starts[i] + n] += 1
            if n:
                assert L.offsets[L.first[i]] <= L.starts[i] < L.offsets[L.first[i] + 1]
                assert L.offsets[L.last[i]] < L.starts[i] + n <= L.offsets[L.last[i] + 1]
        assert (covered == 1).all()
        assert all(x >= 1 for x in L.need)


def _model(dt):
    torch.manual_seed(0)
    m = torch.nn.Sequential(torch.nn.Linear(64, 256), torch.nn.GELU(),
                            torch.nn.Linear(256, 256), torch.nn.GELU(),
                            torch.nn.Linear(256, 10))
    return m.to(device="cuda", dtype=dt)


@pytest.mark.gpu
@pytest.mark.parametrize("rule", ["mgda", "pcgrad", "cagrad"])
@pytest.mark.parametrize("dt", [torch.float32, torch.bfloat16])
def test_bucket_moo_in_backward_matches_resolve(rule, dt):
    K = 3
    m = _model(dt)
    params = list(m.parameters())
    eb = 4 if dt == torch.float32 else 2
    moo = BucketMOO(params, K, bucket_bytes=12000 * eb, rule=rule)
    assert moo.layout.n_buckets > 4
    gen = torch.Generator(device="cuda").manual_seed(1)
    xs = [torch.randn(32, 64, device="cuda", generator=gen).to(dt) * (1 + k) for k in range(K)]
    ys = [torch.randn(32, 10, device="cuda", generator=gen).to(dt) * (-1) ** k for k in range(K)]
    for step in range(2):                       # the second step reuses every buffer
        for k in range(K):
            moo.begin(k)
            loss = ((m(xs[k]) - ys[k]) ** 2).mean()
            loss.backward()
        d = moo.finish()
        torch.cuda.synchronize()
        # per-language gradients, flattened last-registered first
        ref = []
        for k in range(K):
            gs = torch.autograd.grad(((m(xs[k]) - ys[k]) ** 2).mean(), params)
            ref.append(torch.cat([g.reshape(-1) for g in reversed(gs)]))
            assert torch.equal(moo.grads[k], ref[k]), k
        # one resolve over the whole plan, same buffers (the three-launch
        # path, whose kernels the per-bucket resolve runs)
        out = torch.empty_like(d)
        beta = torch.empty(moo.layout.n_buckets, K, device="cuda")
        p3 = bk.bkmoo_default_params()
        p3.flags |= bk.BKMOO_FLAG_THREE_PASS
        moo.resolver.resolve(moo.grads, rule, out, params=p3, out_weights=beta)
        torch.cuda.synchronize()
        assert moo.resolver.status() == 0
        assert torch.equal(d, out)
        assert torch.equal(moo.weights, beta)
        assert (moo.status.cpu().numpy() == 0).all()
        for i, p in enumerate(params):
            s = moo.layout.starts[i]
            assert p.grad.data_ptr() == d[s:s + p.numel()].data_ptr()
    # oracle on the final buffers
    hv = [g.cpu().view(torch.int16).numpy().view(np.uint16) if dt == torch.bfloat16
          else g.cpu().numpy() for g in moo.grads]
    R = {"mgda": orc.MGDA, "pcgrad": orc.PCGRAD, "cagrad": orc.CAGRAD}[rule]
    ref = orc.resolve(hv, moo.layout.offsets, R, cagrad_c=0.5)
    np.testing.assert_allclose(beta.cpu().numpy(), ref["beta"], atol=1e-4)
    dd = d.float().cpu().numpy().astype(np.float64)
    rt = 1e-5 if dt == torch.float32 else 2 ** -8
    for b in range(moo.layout.n_buckets):
        lo, hi = int(moo.layout.offsets[b]), int(moo.layout.offsets[b + 1])
        gn = sum(abs(ref["beta"][b][k]) * np.linalg.norm(hv_k[lo:hi].astype(np.float64)
                 if dt == torch.float32 else
                 (hv_k[lo:hi].astype(np.uint32) << 16).view(np.float32).astype(np.float64))
                 for k, hv_k in enumerate(hv))
        err = np.linalg.norm(dd[lo:hi] - ref["d"][lo:hi])
        assert err <= rt * np.linalg.norm(ref["d"][lo:hi]) + (K + 2) * 2.0 ** -24 * gn, (b, err)
    moo.remove()


@pytest.mark.gpu
def test_bucket_moo_unused_parameter_resolved_in_finish():
    """A parameter that receives no gradient never completes its bucket
    during backward; finish() resolves it (its gradient is zero)."""
    m = _model(torch.float32)
    extra = torch.nn.Parameter(torch.ones(5000, device="cuda"))
    params = list(m.parameters()) + [extra]
    moo = BucketMOO(params, 2, bucket_bytes=4 * 10000, rule="mgda")
    for k in range(2):
        moo.begin(k)
        m(torch.randn(8, 64, device="cuda")).sum().backward()
    d = moo.finish()
    torch.cuda.synchronize()
    out = torch.empty_like(d)
    p3 = bk.bkmoo_default_params()
    p3.flags |= bk.BKMOO_FLAG_THREE_PASS
    moo.resolver.resolve(moo.grads, "mgda", out, params=p3)
    torch.cuda.synchronize()
    assert torch.equal(d, out)
    assert torch.count_nonzero(extra.grad).item() == 0
    moo.remove()
