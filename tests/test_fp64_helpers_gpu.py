"""The fp64 division and square root of the fast per-bucket solvers
(an fp32 seed plus one Newton-Raphson step with a residual correction)
against CUDA's correctly rounded fp64 division and square root, on 10^6
random operands spanning 1e-30 .. 1e30 of both signs and on the boundaries
of the range where the seed is used.  Bound: relative error <= 2^-46
(the seed's two fp32 roundings, about 2^-23 together, squared by the Newton
step) plus the reference's own rounding, 2^-53."""
import numpy as np
import pytest
import torch

from paper_2606_05613_gb300 import build as nb
from paper_2606_05613_gb300 import native as bk

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")
BOUND = 2.0 ** -46 + 2.0 ** -53


@pytest.fixture(scope="module", autouse=True)
def _built():
    nb.build()
    bk.load()


def _log_uniform(rng, n, lo=-30.0, hi=30.0):
    return 10.0 ** rng.uniform(lo, hi, size=n) * rng.choice([-1.0, 1.0], size=n)


def _edges():
    e = []
    for v in (1e-30, 1e30):
        e += [v, np.nextafter(v, 0), np.nextafter(v, np.inf), v * (1 + 1e-9), v * (1 - 1e-9)]
    e += [1.0, 2.0, 0.5, 3.0, 1.5, np.nextafter(1.0, 2.0), np.nextafter(1.0, 0.0),
          float(np.float32(1.0 / 3.0)), 2.0 ** -99, 2.0 ** 99]
    e = np.array(e)
    return np.concatenate([e, -e])


def _run(op, a, b=None):
    ta = torch.from_numpy(np.ascontiguousarray(a)).to(DEV)
    tb = torch.from_numpy(np.ascontiguousarray(b)).to(DEV) if b is not None else None
    out = torch.empty_like(ta)
    bk.bkmoo_selftest_fp64(op, ta, tb, out)
    ref = ta / tb if op == 0 else torch.sqrt(ta)
    torch.cuda.synchronize()
    return out.cpu().numpy(), ref.cpu().numpy()


def test_div_nr_within_bound():
    rng = np.random.default_rng(0)
    n = 1_000_000
    a = _log_uniform(rng, n)
    b = _log_uniform(rng, n)
    ed = _edges()
    a = np.concatenate([a, np.repeat(ed, len(ed)), rng.standard_normal(len(ed) ** 2)])
    b = np.concatenate([b, np.tile(ed, len(ed)), np.tile(ed, len(ed))])
    got, ref = _run(0, a, b)
    inside = (np.abs(b) > 1e-30) & (np.abs(b) < 1e30)
    rel = np.abs(got[inside] - ref[inside]) / np.abs(ref[inside])
    assert rel.max() <= BOUND, rel.max()
    # outside the seed's range: the correctly rounded quotient itself
    np.testing.assert_array_equal(got[~inside], ref[~inside])
    assert inside.sum() > n * 0.99 and (~inside).sum() > 0


def test_div_nr_special_operands():
    a = np.array([0.0, -0.0, 1.0, -1.0, 5.0, 1e300, 1e-300, 7.0])
    b = np.array([3.0, 3.0, 0.0, 0.0, np.inf, 1e-10, 1e10, 1e31])
    got, ref = _run(0, a, b)
    np.testing.assert_array_equal(got, ref)


def test_sqrt_nr_within_bound():
    rng = np.random.default_rng(1)
    n = 1_000_000
    x = np.abs(_log_uniform(rng, n))
    ed = np.abs(_edges())
    x = np.concatenate([x, ed, rng.uniform(0.0, 4.0, size=10000)])
    got, ref = _run(1, x)
    inside = (x > 1e-30) & (x < 1e30)
    rel = np.abs(got[inside] - ref[inside]) / ref[inside]
    assert rel.max() <= BOUND, rel.max()
    np.testing.assert_array_equal(got[~inside], ref[~inside])


def test_sqrt_nr_zero_and_negative_give_zero():
    x = np.array([0.0, -0.0, -1.0, -1e-40, 1e-320, 1e300])
    got, ref = _run(1, x)
    np.testing.assert_array_equal(got[:4], np.zeros(4))
    np.testing.assert_array_equal(got[4:], ref[4:])
