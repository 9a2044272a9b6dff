"""The allocation-free Gram entry point (bkmoo_gram_noalloc).

Some callers hold their gradient and output buffers but cannot obtain more
device memory -- a hook running inside a training framework whose device
memory all belongs to the framework's caching allocator, or a C caller in a
process where another component owns allocation.  bkmoo_gram_noalloc serves
them by keeping its scratch in a static device array of the library.  This
test calls it through the C ABI twice in a row, with different plans and
inputs, and checks each result against bkmoo_gram (which uses a caller
workspace) within the Gram tolerance of the parity tests.  The file sorts
last so that a run stopping at the first failure has run everything else.
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2606_05613_gb300 import build as nb
from paper_2606_05613_gb300 import inputs
from paper_2606_05613_gb300 import native as bk
from tests.parity_util import gram_close

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")


def _case(K, dt, sizes, bucket_elems, seed):
    import dataclasses
    eb = 4 if dt == "f32" else 2
    w = inputs.scaled(inputs.gpt2_small(), "noalloc", sizes, bucket_elems * eb)
    w = dataclasses.replace(w, K=K, dtype=dt, seed=seed)
    off = bk.bkmoo_plan(w.param_sizes, w.elem_bytes, w.bucket_bytes)
    return off, inputs.generate(w, off, DEV)


def _noalloc_c_abi(grads, off, out):
    lib = bk.load()
    ptrs = (ctypes.c_void_p * len(grads))(*[g.data_ptr() for g in grads])
    offs = np.ascontiguousarray(off, dtype=np.int64)
    dt = bk.BKMOO_F32 if grads[0].dtype == torch.float32 else bk.BKMOO_BF16
    stream = ctypes.c_void_p(torch.cuda.current_stream(DEV).cuda_stream)
    return lib.bkmoo_gram_noalloc(ptrs, len(grads), dt, offs.ctypes.data, len(offs) - 1,
                                  ctypes.c_void_p(out.data_ptr()), stream)


def test_gram_noalloc_matches_gram_twice():
    nb.build()
    cases = [(4, "bf16", [70001, 3, 131071, 5, 65536, 99999, 17, 40000], 150000, 1),
             (8, "f32", [300000, 7, 123457, 1, 98765], 100000, 2)]
    for K, dt, sizes, be, seed in cases:
        off, grads = _case(K, dt, sizes, be, seed)
        B = len(off) - 1
        got = torch.full((B, K, K), float("nan"), dtype=torch.float64, device=DEV)
        assert _noalloc_c_abi(grads, off, got) == bk.BKMOO_OK
        ref = torch.empty(B, K, K, dtype=torch.float64, device=DEV)
        bk.Resolver(K, grads[0].dtype, off, DEV).gram(grads, ref)
        torch.cuda.synchronize()
        g, r = got.cpu().numpy(), ref.cpu().numpy()
        for b in range(B):
            ok, err = gram_close(g[b], r[b])
            assert ok, (K, dt, b, err)


def test_gram_noalloc_rejects_too_large():
    nb.build()
    lib = bk.load()
    K = 16
    g = [torch.empty(16, dtype=torch.float32, device=DEV) for _ in range(K)]
    ptrs = (ctypes.c_void_p * K)(*[t.data_ptr() for t in g])
    too_many = np.arange(0, bk.BKMOO_NOALLOC_MAX_BUCKETS + 2, dtype=np.int64)
    out = torch.empty(1, dtype=torch.float64, device=DEV)
    r = lib.bkmoo_gram_noalloc(ptrs, K, bk.BKMOO_F32, too_many.ctypes.data, len(too_many) - 1,
                               ctypes.c_void_p(out.data_ptr()), None)
    assert r == bk.BKMOO_ERR_WORKSPACE
    huge = np.array([0, 10**10], dtype=np.int64)      # needs far more than the array
    r = lib.bkmoo_gram_noalloc(ptrs, K, bk.BKMOO_F32, huge.ctypes.data, 1,
                               ctypes.c_void_p(out.data_ptr()), None)
    assert r == bk.BKMOO_ERR_WORKSPACE
