"""The allocation-free Gram entry point (bkmoo_gram_noalloc).

Some callers hold their gradient and output buffers but cannot obtain more
device memory -- a hook running inside a training framework whose device
memory all belongs to the framework's caching allocator, or a C caller in a
process where another component owns allocation.  bkmoo_gram_noalloc serves
them by keeping its scratch in a static device array of the library.

This test calls it through the C ABI several times in a row, with different
plans and inputs, and checks each result bit for bit against bkmoo_gram
(which runs the same kernels on a caller workspace, so the results must be
identical) and against the oracle's fp64 Gram within the Gram tolerance of
the parity tests.  The cases cover several bucket-table slices (more than
224 buckets) and a bucket of more than 1024 chunks (the group pre-reduction
of the chunk partials).  Argument and size rejections are tested on the CPU
(tests/test_abi_cpu.py).  The file sorts last so that a run stopping at the
first failure has run everything else.
"""
import ctypes

import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2606_05613_gb300 import build as nb
from paper_2606_05613_gb300 import inputs
from paper_2606_05613_gb300 import native as bk
from tests.parity_util import gram_close

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")


def _case(K, dt, sizes, bucket_elems, seed, one_per_tensor=False):
    import dataclasses
    eb = 4 if dt == "f32" else 2
    w = inputs.scaled(inputs.gpt2_small(), "noalloc", sizes, bucket_elems * eb)
    w = dataclasses.replace(w, K=K, dtype=dt, seed=seed)
    if one_per_tensor:
        off = np.concatenate([[0], np.cumsum(list(reversed(sizes)))]).astype(np.int64)
    else:
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


def test_gram_noalloc_matches_gram_and_oracle():
    nb.build()
    orc.build()
    ch_bf16 = 32768
    cases = [
        (4, "bf16", [70001, 3, 131071, 5, 65536, 99999, 17, 40000], 150000, 1, False),
        (8, "f32", [300000, 7, 123457, 1, 98765], 100000, 2, False),
        # about 600 small buckets: three bucket-table slices
        (3, "f32", [997 + 13 * (i % 37) for i in range(600)], 1, 3, True),
        # one bucket of 1100 chunks between two small ones (group pre-reduction)
        (2, "bf16", [5000, 1100 * ch_bf16 - 77, 9999], 1, 4, True),
    ]
    for K, dt, sizes, be, seed, one in cases:
        off, grads = _case(K, dt, sizes, be, seed, one)
        B = len(off) - 1
        ref = torch.empty(B, K, K, dtype=torch.float64, device=DEV)
        bk.Resolver(K, grads[0].dtype, off, DEV).gram(grads, ref)
        for _ in range(2):                 # two calls in a row on the same array
            got = torch.full((B, K, K), float("nan"), dtype=torch.float64, device=DEV)
            assert _noalloc_c_abi(grads, off, got) == bk.BKMOO_OK
            torch.cuda.synchronize()
            assert torch.equal(got, ref), (K, dt, B)
        g = got.cpu().numpy()
        hv = [inputs.host_view(t) for t in grads]
        for b in range(B):
            ok, err = gram_close(g[b], orc.gram(hv, int(off[b]), int(off[b + 1] - off[b])))
            assert ok, (K, dt, b, err)
