"""GPU: bkmoo_resolve_host (gradients and direction in host memory, buckets
streamed through three device staging slots) against the device-resident
bkmoo_resolve -- bit-identical beta, status and direction -- and against the
fp64 oracle, with windows of one and of several buckets, ragged and unaligned
bucket starts, in-place use and page-locked and pageable host buffers."""
import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2606_05613_gb300 import build as nb
from paper_2606_05613_gb300 import inputs
from paper_2606_05613_gb300 import native as bk
from tests.test_parity_gpu import RAGGED, _check_against_oracle, _tdt, _workload

pytestmark = pytest.mark.gpu

DEV = torch.device("cuda:0")


@pytest.fixture(scope="module", autouse=True)
def _built():
    nb.build()
    bk.load()
    orc.build()


def _host_run(w, rule, out_dt, window_elems, pinned=True, inplace=False, params=None):
    off = bk.bkmoo_plan(w.param_sizes, w.elem_bytes, w.bucket_bytes)
    grads = inputs.generate(w, off, DEV)
    B, N = len(off) - 1, int(off[-1])
    res = bk.Resolver(w.K, _tdt(w.dtype), off, DEV)
    # device-resident reference run on the three-launch path (the host path
    # runs the same kernels window by window)
    out_d = torch.empty(N, dtype=_tdt(out_dt), device=DEV)
    beta_d = torch.empty(B, w.K, device=DEV)
    st_d = torch.empty(B, dtype=torch.int32, device=DEV)
    p3 = params if params is not None else bk.bkmoo_default_params()
    p3.flags |= bk.BKMOO_FLAG_THREE_PASS
    res.resolve(grads, rule, out_d, params=p3, out_weights=beta_d, out_status=st_d)
    # host run
    host = [torch.empty(N, dtype=_tdt(w.dtype), pin_memory=pinned) for _ in range(w.K)]
    for h, g in zip(host, grads):
        h.copy_(g)
    hv = [inputs.host_view(h).copy() for h in host]
    out_h = host[0] if inplace else torch.full((N,), 7.0, dtype=_tdt(out_dt), pin_memory=pinned)
    staging = torch.empty(res.staging_size(_dtype(out_dt), window_elems), dtype=torch.uint8,
                          device=DEV)
    beta_h = torch.full((B, w.K), float("nan"), device=DEV)
    st_h = torch.full((B,), -1, dtype=torch.int32, device=DEV)
    res.resolve_host(host, rule, out_h, staging, params=params, out_weights=beta_h,
                     out_status=st_h)
    torch.cuda.synchronize()
    assert res.status() == 0
    return off, hv, out_d.cpu(), beta_d.cpu(), st_d.cpu(), out_h, beta_h.cpu(), st_h.cpu()


def _dtype(dt):
    return bk.BKMOO_F32 if dt == "f32" else bk.BKMOO_BF16


@pytest.mark.parametrize("rule", ["mgda", "pcgrad", "cagrad", "mean"])
@pytest.mark.parametrize("dt,out_dt", [("f32", "f32"), ("bf16", "bf16"), ("bf16", "f32"),
                                       ("f32", "bf16")])
@pytest.mark.parametrize("window", [0, 300000])
def test_host_path_bit_identical_to_device_path(rule, dt, out_dt, window):
    w = _workload(4, dt, RAGGED, 150000, seed=31, flip=0.2)
    off, hv, out_d, beta_d, st_d, out_h, beta_h, st_h = _host_run(w, rule, out_dt, window)
    assert torch.equal(st_h, st_d)
    assert torch.equal(beta_h, beta_d)
    assert torch.equal(out_h, out_d)
    _check_against_oracle(w, rule, off, hv, out_h, beta_h.numpy(), st_h.numpy(), out_dt)


@pytest.mark.parametrize("K", [1, 2, 8, 16])
def test_host_path_every_k(K):
    w = _workload(K, "bf16", RAGGED, 120000, seed=40 + K, flip=0.2)
    off, hv, out_d, beta_d, st_d, out_h, beta_h, st_h = _host_run(w, "mgda", "bf16", 0)
    assert torch.equal(beta_h, beta_d) and torch.equal(out_h, out_d)


def test_host_path_in_place_and_pageable():
    w = _workload(3, "f32", RAGGED, 100000, seed=12)
    for pinned in (True, False):
        off, hv, out_d, beta_d, _, out_h, beta_h, _ = _host_run(w, "cagrad", "f32", 0,
                                                               pinned=pinned, inplace=True)
        assert torch.equal(beta_h, beta_d)
        assert torch.equal(out_h, out_d)


def test_host_path_staging_too_small():
    w = _workload(2, "f32", [50000, 50000], 50000, seed=3)
    off = bk.bkmoo_plan(w.param_sizes, w.elem_bytes, w.bucket_bytes)
    res = bk.Resolver(2, torch.float32, off, DEV)
    need = res.staging_size(bk.BKMOO_F32)
    host = [torch.zeros(int(off[-1]), pin_memory=True) for _ in range(2)]
    out = torch.empty(int(off[-1]), pin_memory=True)
    small = torch.empty(need - 2048, dtype=torch.uint8, device=DEV)
    with pytest.raises(bk.BkmooError) as e:
        res.resolve_host(host, "mgda", out, small)
    assert e.value.code == bk.BKMOO_ERR_WORKSPACE
    ok = torch.empty(need, dtype=torch.uint8, device=DEV)
    res.resolve_host(host, "mgda", out, ok)
    torch.cuda.synchronize()
    assert res.status() == 0 and torch.count_nonzero(out).item() == 0
