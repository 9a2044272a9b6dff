"""ctypes binding of the C ABI in include/bkmoo.h.

Argument marshalling only: every step of the resolve runs in the CUDA library
(libbkmoo.so, built in-tree by paper_2606_05613_gb300.build).  There is no
CPU or PyTorch fallback; if the library is missing or cannot be loaded, every
call raises.  Functions carry the C names; torch tensors supply device
pointers and the current CUDA stream.
"""
from __future__ import annotations

import ctypes
import os
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libbkmoo.so")

BKMOO_OK = 0
BKMOO_ERR_INVALID = 1
BKMOO_ERR_CUDA = 2
BKMOO_ERR_NONFINITE = 3
BKMOO_ERR_WORKSPACE = 4
BKMOO_ERR_TIMEOUT = 5
BKMOO_ERR_BUFFER_TOO_SMALL = 6
BKMOO_ERR_NOT_CONVERGED = 7

BKMOO_MGDA, BKMOO_PCGRAD, BKMOO_CAGRAD, BKMOO_MEAN = 0, 1, 2, 3
BKMOO_F32, BKMOO_BF16 = 0, 1
BKMOO_FLAG_CLOSED_FORM_K2 = 0x1
BKMOO_FLAG_POLISH = 0x2
BKMOO_FLAG_FUSED = 0x4
BKMOO_FLAG_THREE_PASS = 0x8
BKMOO_FLAG_TEST_WITHHOLD = 0x100
BKMOO_FLAG_TEST_WITHHOLD_EXCHANGE = 0x200
BKMOO_NOALLOC_SCRATCH_BYTES = 32 << 20
BKMOO_NOALLOC_MAX_BUCKETS = 4096

RULES = {"mgda": BKMOO_MGDA, "pcgrad": BKMOO_PCGRAD, "cagrad": BKMOO_CAGRAD, "mean": BKMOO_MEAN}

_lock = threading.Lock()
_lib = None


class BkmooError(RuntimeError):
    def __init__(self, code: int, where: str):
        self.code = code
        super().__init__("%s failed: %s (%d)" % (where, bkmoo_status_string(code), code))


class bkmoo_params(ctypes.Structure):
    _fields_ = [
        ("max_iter", ctypes.c_int32),
        ("tol", ctypes.c_double),
        ("cagrad_c", ctypes.c_double),
        ("seed", ctypes.c_uint64),
        ("step", ctypes.c_uint64),
        ("flags", ctypes.c_uint32),
        ("events", ctypes.c_void_p),
    ]


def load():
    """Load libbkmoo.so (raises if it is missing: there is no fallback)."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        if not os.path.exists(LIB_PATH):
            raise RuntimeError("libbkmoo.so is not built (%s); run "
                               "paper_2606_05613_gb300.build.build()" % LIB_PATH)
        lib = ctypes.CDLL(LIB_PATH)
        i32, i64, sz, vp = ctypes.c_int32, ctypes.c_int64, ctypes.c_size_t, ctypes.c_void_p
        lib.bkmoo_default_params.restype = None
        lib.bkmoo_default_params.argtypes = [ctypes.POINTER(bkmoo_params)]
        lib.bkmoo_plan.restype = ctypes.c_int
        lib.bkmoo_plan.argtypes = [vp, i32, i32, i64, vp, i64, ctypes.POINTER(i64)]
        lib.bkmoo_workspace_size.restype = ctypes.c_int
        lib.bkmoo_workspace_size.argtypes = [i32, i32, vp, i64, ctypes.POINTER(sz)]
        lib.bkmoo_workspace_init.restype = ctypes.c_int
        lib.bkmoo_workspace_init.argtypes = [i32, i32, vp, i64, vp, sz, vp]
        lib.bkmoo_gram.restype = ctypes.c_int
        lib.bkmoo_gram.argtypes = [vp, i32, i32, vp, i64, vp, vp, sz, vp]
        lib.bkmoo_conflicts.restype = ctypes.c_int
        lib.bkmoo_conflicts.argtypes = [vp, i32, i64, vp, vp, vp, vp]
        lib.bkmoo_gram_noalloc.restype = ctypes.c_int
        lib.bkmoo_gram_noalloc.argtypes = [vp, i32, i32, vp, i64, vp, vp]
        lib.bkmoo_resolve.restype = ctypes.c_int
        lib.bkmoo_resolve.argtypes = [vp, i32, i32, vp, i64, i32, ctypes.POINTER(bkmoo_params),
                                      vp, i32, vp, vp, vp, sz, vp]
        lib.bkmoo_resolve_buckets.restype = ctypes.c_int
        lib.bkmoo_resolve_buckets.argtypes = [vp, i32, i32, vp, i64, i64, i64, i32,
                                              ctypes.POINTER(bkmoo_params), vp, i32, vp, vp, vp,
                                              sz, vp]
        lib.bkmoo_host_staging_size.restype = ctypes.c_int
        lib.bkmoo_host_staging_size.argtypes = [i32, i32, i32, vp, i64, i64, ctypes.POINTER(sz)]
        lib.bkmoo_resolve_host.restype = ctypes.c_int
        lib.bkmoo_resolve_host.argtypes = [vp, i32, i32, vp, i64, i32,
                                           ctypes.POINTER(bkmoo_params), vp, i32, vp, vp, vp, sz,
                                           vp, sz, vp]
        lib.bkmoo_workspace_status.restype = ctypes.c_int
        lib.bkmoo_workspace_status.argtypes = [vp, vp, ctypes.POINTER(i32)]
        lib.bkmoo_status_string.restype = ctypes.c_char_p
        lib.bkmoo_status_string.argtypes = [i32]
        lib.bkmoo_version.restype = i32
        lib.bkmoo_version.argtypes = []
        lib.bkmoo_resolve_path.restype = ctypes.c_int
        lib.bkmoo_resolve_path.argtypes = [i32, i32, i32, vp, i64, ctypes.c_uint32,
                                           ctypes.POINTER(ctypes.c_int32)]
        lib.bkmoo_selftest_fp64.restype = ctypes.c_int
        lib.bkmoo_selftest_fp64.argtypes = [i32, vp, vp, vp, i64, vp]
        _lib = lib
        return lib


def _check(code: int, where: str):
    if code != BKMOO_OK:
        raise BkmooError(code, where)


def _dtype_code(t) -> int:
    import torch
    if t.dtype == torch.float32:
        return BKMOO_F32
    if t.dtype == torch.bfloat16:
        return BKMOO_BF16
    raise TypeError("gradients must be float32 or bfloat16, got %s" % t.dtype)


def _stream_handle(stream, device):
    import torch
    if stream is None:
        stream = torch.cuda.current_stream(device)
    return ctypes.c_void_p(stream.cuda_stream)


def _offsets_array(offsets) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(offsets, dtype=np.int64))


def _grad_ptrs(grads):
    if not grads:
        raise ValueError("need at least one gradient")
    for g in grads:
        if not g.is_cuda or not g.is_contiguous():
            raise ValueError("gradients must be contiguous CUDA tensors")
    return (ctypes.c_void_p * len(grads))(*[g.data_ptr() for g in grads])


def bkmoo_default_params() -> bkmoo_params:
    p = bkmoo_params()
    load().bkmoo_default_params(ctypes.byref(p))
    return p


def bkmoo_plan(param_sizes, elem_bytes: int, bucket_bytes: int) -> np.ndarray:
    lib = load()
    sizes = np.ascontiguousarray(np.asarray(param_sizes, dtype=np.int64))
    nb = ctypes.c_int64(0)
    _check(lib.bkmoo_plan(sizes.ctypes.data, len(sizes), elem_bytes, bucket_bytes, None, 0,
                          ctypes.byref(nb)), "bkmoo_plan")
    out = np.zeros(nb.value + 1, dtype=np.int64)
    _check(lib.bkmoo_plan(sizes.ctypes.data, len(sizes), elem_bytes, bucket_bytes,
                          out.ctypes.data, len(out), ctypes.byref(nb)), "bkmoo_plan")
    return out


def bkmoo_workspace_size(K: int, in_dtype: int, offsets) -> int:
    off = _offsets_array(offsets)
    n = ctypes.c_size_t(0)
    _check(load().bkmoo_workspace_size(K, in_dtype, off.ctypes.data, len(off) - 1,
                                       ctypes.byref(n)), "bkmoo_workspace_size")
    return int(n.value)


def bkmoo_workspace_init(K: int, in_dtype: int, offsets, ws, stream=None):
    off = _offsets_array(offsets)
    _check(load().bkmoo_workspace_init(K, in_dtype, off.ctypes.data, len(off) - 1,
                                       ws.data_ptr(), ws.numel() * ws.element_size(),
                                       _stream_handle(stream, ws.device)),
           "bkmoo_workspace_init")


def bkmoo_gram(grads, offsets, out_gram, ws, stream=None):
    off = _offsets_array(offsets)
    ptrs = _grad_ptrs(grads)
    _check(load().bkmoo_gram(ptrs, len(grads), _dtype_code(grads[0]), off.ctypes.data,
                             len(off) - 1, out_gram.data_ptr(), ws.data_ptr(),
                             ws.numel() * ws.element_size(),
                             _stream_handle(stream, grads[0].device)), "bkmoo_gram")


def bkmoo_conflicts(gram, out_cos=None, out_stats=None, out_conflict=None, stream=None):
    """Figure 1's conflict statistics from Gram matrices [B, K, K] (fp64, CUDA)."""
    B, K = int(gram.shape[0]), int(gram.shape[1])
    _check(load().bkmoo_conflicts(gram.data_ptr(), K, B,
                                  out_cos.data_ptr() if out_cos is not None else None,
                                  out_stats.data_ptr() if out_stats is not None else None,
                                  out_conflict.data_ptr() if out_conflict is not None else None,
                                  _stream_handle(stream, gram.device)), "bkmoo_conflicts")


def bkmoo_gram_noalloc(grads, offsets, out_gram, stream=None):
    """bkmoo_gram for callers that cannot allocate device memory: no
    workspace; the scratch is a static device array of the library (see
    include/bkmoo.h for its limits and the rule that overlapping calls race)."""
    off = _offsets_array(offsets)
    ptrs = _grad_ptrs(grads)
    _check(load().bkmoo_gram_noalloc(ptrs, len(grads), _dtype_code(grads[0]), off.ctypes.data,
                                     len(off) - 1, out_gram.data_ptr(),
                                     _stream_handle(stream, grads[0].device)),
           "bkmoo_gram_noalloc")


def bkmoo_resolve(grads, offsets, rule, out_dir, ws, params=None, out_weights=None,
                  out_status=None, stream=None):
    if isinstance(rule, str):
        rule = RULES[rule]
    off = _offsets_array(offsets)
    ptrs = _grad_ptrs(grads)
    p = params if params is not None else bkmoo_default_params()
    _check(load().bkmoo_resolve(ptrs, len(grads), _dtype_code(grads[0]), off.ctypes.data,
                                len(off) - 1, rule, ctypes.byref(p), out_dir.data_ptr(),
                                _dtype_code(out_dir),
                                out_weights.data_ptr() if out_weights is not None else None,
                                out_status.data_ptr() if out_status is not None else None,
                                ws.data_ptr(), ws.numel() * ws.element_size(),
                                _stream_handle(stream, grads[0].device)), "bkmoo_resolve")


def bkmoo_resolve_buckets(grads, offsets, b_lo, b_hi, rule, out_dir, ws, params=None,
                          out_weights=None, out_status=None, stream=None):
    if isinstance(rule, str):
        rule = RULES[rule]
    off = _offsets_array(offsets)
    ptrs = _grad_ptrs(grads)
    p = params if params is not None else bkmoo_default_params()
    _check(load().bkmoo_resolve_buckets(ptrs, len(grads), _dtype_code(grads[0]), off.ctypes.data,
                                        len(off) - 1, b_lo, b_hi, rule, ctypes.byref(p),
                                        out_dir.data_ptr(), _dtype_code(out_dir),
                                        out_weights.data_ptr() if out_weights is not None
                                        else None,
                                        out_status.data_ptr() if out_status is not None else None,
                                        ws.data_ptr(), ws.numel() * ws.element_size(),
                                        _stream_handle(stream, grads[0].device)),
           "bkmoo_resolve_buckets")


def bkmoo_host_staging_size(K: int, in_dtype: int, out_dtype: int, offsets,
                            window_elems: int = 0) -> int:
    off = _offsets_array(offsets)
    n = ctypes.c_size_t(0)
    _check(load().bkmoo_host_staging_size(K, in_dtype, out_dtype, off.ctypes.data, len(off) - 1,
                                          window_elems, ctypes.byref(n)),
           "bkmoo_host_staging_size")
    return int(n.value)


def bkmoo_resolve_host(host_grads, offsets, rule, host_out, ws, staging, params=None,
                       out_weights=None, out_status=None, stream=None):
    """host_grads / host_out: contiguous CPU tensors (page-locked for overlap);
    ws, staging, out_weights, out_status: CUDA tensors."""
    if isinstance(rule, str):
        rule = RULES[rule]
    if not host_grads:
        raise ValueError("need at least one gradient")
    for g in list(host_grads) + [host_out]:
        if g.is_cuda or not g.is_contiguous():
            raise ValueError("host_grads and host_out must be contiguous CPU tensors")
    off = _offsets_array(offsets)
    ptrs = (ctypes.c_void_p * len(host_grads))(*[g.data_ptr() for g in host_grads])
    p = params if params is not None else bkmoo_default_params()
    _check(load().bkmoo_resolve_host(ptrs, len(host_grads), _dtype_code(host_grads[0]),
                                     off.ctypes.data, len(off) - 1, rule, ctypes.byref(p),
                                     host_out.data_ptr(), _dtype_code(host_out),
                                     out_weights.data_ptr() if out_weights is not None else None,
                                     out_status.data_ptr() if out_status is not None else None,
                                     ws.data_ptr(), ws.numel() * ws.element_size(),
                                     staging.data_ptr(), staging.numel() * staging.element_size(),
                                     _stream_handle(stream, ws.device)), "bkmoo_resolve_host")


def bkmoo_workspace_status(ws, stream=None) -> int:
    st = ctypes.c_int32(0)
    _check(load().bkmoo_workspace_status(ws.data_ptr(), _stream_handle(stream, ws.device),
                                         ctypes.byref(st)), "bkmoo_workspace_status")
    return int(st.value)


def bkmoo_status_string(code: int) -> str:
    return load().bkmoo_status_string(code).decode()


def bkmoo_version() -> int:
    return int(load().bkmoo_version())


def bkmoo_resolve_path(K: int, in_dtype: int, rule, offsets, flags: int) -> int:
    """0: three launches; 1: cluster-per-bucket fused kernel; 2:
    grid-synchronised fused kernel (the path bkmoo_resolve takes)."""
    if isinstance(rule, str):
        rule = RULES[rule]
    off = _offsets_array(offsets)
    out = ctypes.c_int32(-1)
    _check(load().bkmoo_resolve_path(K, in_dtype, rule, off.ctypes.data, len(off) - 1, flags,
                                     ctypes.byref(out)), "bkmoo_resolve_path")
    return int(out.value)


def bkmoo_selftest_fp64(op: int, a, b, out, stream=None):
    """The solvers' fp64 division (op 0, out = a / b) or square root (op 1,
    out = sqrt(a)) element-wise on the device (fp64 CUDA tensors)."""
    _check(load().bkmoo_selftest_fp64(op, a.data_ptr(), b.data_ptr() if b is not None else None,
                                      out.data_ptr(), int(out.numel()),
                                      _stream_handle(stream, out.device)), "bkmoo_selftest_fp64")


class Resolver:
    """Holds the plan and the workspace of one (K, dtype, offsets) triple.

    Allocates the workspace once (torch, on `device`) and initialises it; each
    call to resolve() then queues Gram -> solve -> combine on the current
    stream without further allocation."""

    def __init__(self, K: int, in_dtype, offsets, device):
        import torch
        self.K = K
        self.in_dtype = in_dtype if isinstance(in_dtype, int) else (
            BKMOO_F32 if in_dtype == torch.float32 else BKMOO_BF16)
        self.offsets = _offsets_array(offsets)
        self.n_buckets = len(self.offsets) - 1
        self.device = torch.device(device)
        nbytes = bkmoo_workspace_size(K, self.in_dtype, self.offsets)
        self.ws = torch.empty(nbytes, dtype=torch.uint8, device=self.device)
        bkmoo_workspace_init(K, self.in_dtype, self.offsets, self.ws)

    def resolve(self, grads, rule, out_dir, params=None, out_weights=None, out_status=None,
                stream=None):
        bkmoo_resolve(grads, self.offsets, rule, out_dir, self.ws, params, out_weights,
                      out_status, stream)

    def resolve_buckets(self, grads, b_lo, b_hi, rule, out_dir, params=None, out_weights=None,
                        out_status=None, stream=None):
        bkmoo_resolve_buckets(grads, self.offsets, b_lo, b_hi, rule, out_dir, self.ws, params,
                              out_weights, out_status, stream)

    def resolve_host(self, host_grads, rule, host_out, staging, params=None, out_weights=None,
                     out_status=None, stream=None):
        bkmoo_resolve_host(host_grads, self.offsets, rule, host_out, self.ws, staging, params,
                           out_weights, out_status, stream)

    def staging_size(self, out_dtype: int, window_elems: int = 0) -> int:
        return bkmoo_host_staging_size(self.K, self.in_dtype, out_dtype, self.offsets,
                                       window_elems)

    def gram(self, grads, out_gram, stream=None):
        bkmoo_gram(grads, self.offsets, out_gram, self.ws, stream)

    def status(self, stream=None) -> int:
        return bkmoo_workspace_status(self.ws, stream)
