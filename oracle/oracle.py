"""fp64 CPU oracle for Bucket-Level MOO -- TEST INFRASTRUCTURE.

Only the test-suite, ``__graft_entry__.smoke()`` and the benchmark's
``cpu_baseline`` / ``--impl reference`` legs may import this module.  It wraps
``bkmoo_oracle.c`` (plain C, double precision, sequential sums) through
ctypes and never touches the CUDA library.

Arrays are numpy: gradients are ``float32`` arrays, or ``uint16`` arrays
holding bf16 bit patterns (pass ``dtype="bf16"``).  Every function cites the
paper section, equation or algorithm that it restates (see the C source).

Parity unpinned (definitions of this library, not of the paper): the bucket
rule R1 for multi-tensor models, the PCGrad order generator, the Frank-Wolfe
initialisation and tie-breaks, and the non-finite policy.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "bkmoo_oracle.c")
_LIB = os.path.join(_HERE, "_build", "libbkmoo_oracle.so")
_lock = threading.Lock()
_lib = None

F32, BF16 = 0, 1
MGDA, PCGRAD, CAGRAD, MEAN = 0, 1, 2, 3
MGDA_EXACT, MGDA_FW, MGDA_ENUM = 0, 1, 2


class Params(ctypes.Structure):
    _fields_ = [
        ("mgda_mode", ctypes.c_int32),
        ("max_iter", ctypes.c_int32),
        ("tol", ctypes.c_double),
        ("cagrad_c", ctypes.c_double),
        ("seed", ctypes.c_uint64),
        ("step", ctypes.c_uint64),
    ]


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (OpenMP over buckets when available)."""
    os.makedirs(os.path.dirname(_LIB), exist_ok=True)
    if not force and os.path.exists(_LIB) and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC):
        return _LIB
    tmp = _LIB + ".tmp.%d" % os.getpid()
    base = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-o", tmp, _SRC, "-lm"]
    try:
        subprocess.run(base[:4] + ["-fopenmp"] + base[4:], check=True,
                       capture_output=True)
    except subprocess.CalledProcessError:
        subprocess.run(base, check=True, capture_output=True)
    os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        lib = ctypes.CDLL(build())
        i32, i64, u64, dbl = ctypes.c_int32, ctypes.c_int64, ctypes.c_uint64, ctypes.c_double
        vp, dp = ctypes.c_void_p, ctypes.POINTER(ctypes.c_double)
        lib.bko_plan.restype = i64
        lib.bko_plan.argtypes = [vp, i32, i32, i64, vp, i64]
        lib.bko_gram.restype = None
        lib.bko_gram.argtypes = [i32, i32, vp, i64, i64, vp]
        lib.bko_mgda_k2.restype = None
        lib.bko_mgda_k2.argtypes = [vp, vp]
        lib.bko_mgda_wolfe.restype = ctypes.c_int
        lib.bko_mgda_wolfe.argtypes = [i32, vp, vp]
        lib.bko_mgda_enum.restype = None
        lib.bko_mgda_enum.argtypes = [i32, vp, vp]
        lib.bko_mgda_fw.restype = ctypes.c_int
        lib.bko_mgda_fw.argtypes = [i32, vp, i32, dbl, vp]
        lib.bko_pcgrad_order.restype = None
        lib.bko_pcgrad_order.argtypes = [u64, u64, i64, i32, i32, vp]
        lib.bko_pcgrad.restype = None
        lib.bko_pcgrad.argtypes = [i32, vp, u64, u64, i64, vp, vp]
        lib.bko_pcgrad_alternatives.restype = i32
        lib.bko_pcgrad_alternatives.argtypes = [i32, vp, u64, u64, i64, i32, vp]
        lib.bko_cagrad.restype = None
        lib.bko_cagrad.argtypes = [i32, vp, dbl, vp, vp]
        lib.bko_conflicts.restype = None
        lib.bko_conflicts.argtypes = [i32, vp, vp, vp, vp]
        lib.bko_combine.restype = None
        lib.bko_combine.argtypes = [i32, i32, vp, i64, i64, vp, vp]
        lib.bko_resolve.restype = ctypes.c_int
        lib.bko_resolve.argtypes = [i32, i32, vp, vp, i64, i64, i32,
                                    ctypes.POINTER(Params), vp, vp, vp, vp, i32]
        lib.bko_max_threads.restype = i32
        lib.bko_max_threads.argtypes = []
        _lib = lib
        return lib


def _ptr(a: np.ndarray) -> int:
    return a.ctypes.data


def _dtype_code(xs) -> int:
    kinds = {x.dtype for x in xs}
    if kinds == {np.dtype(np.float32)}:
        return F32
    if kinds == {np.dtype(np.uint16)}:
        return BF16
    raise TypeError("gradients must all be float32, or all uint16 bf16 bit patterns")


def _ptr_array(xs):
    for x in xs:
        if not x.flags.c_contiguous:
            raise ValueError("gradients must be contiguous")
    arr = (ctypes.c_void_p * len(xs))(*[_ptr(x) for x in xs])
    return arr


def max_threads() -> int:
    return int(_load().bko_max_threads())


def plan(param_sizes, elem_bytes: int, bucket_bytes: int) -> np.ndarray:
    """Bucket offsets by rule R1 over the reverse registration order."""
    lib = _load()
    sizes = np.ascontiguousarray(np.asarray(param_sizes, dtype=np.int64))
    nb = lib.bko_plan(_ptr(sizes), len(sizes), elem_bytes, bucket_bytes, None, 0)
    if nb < 0:
        raise ValueError("invalid plan arguments")
    out = np.zeros(nb + 1, dtype=np.int64)
    r = lib.bko_plan(_ptr(sizes), len(sizes), elem_bytes, bucket_bytes, _ptr(out), nb + 1)
    assert r == nb
    return out


def gram(xs, begin: int = 0, n: int | None = None) -> np.ndarray:
    lib = _load()
    K = len(xs)
    if n is None:
        n = xs[0].size - begin
    G = np.zeros((K, K), dtype=np.float64)
    lib.bko_gram(K, _dtype_code(xs), _ptr_array(xs), begin, n, _ptr(G))
    return G


def _as_G(G) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(G, dtype=np.float64))


def mgda_k2(G) -> np.ndarray:
    G = _as_G(G)
    a = np.zeros(2)
    _load().bko_mgda_k2(_ptr(G), _ptr(a))
    return a


def mgda_wolfe(G) -> np.ndarray:
    G = _as_G(G)
    K = G.shape[0]
    a = np.zeros(K)
    _load().bko_mgda_wolfe(K, _ptr(G), _ptr(a))
    return a


def mgda_enum(G) -> np.ndarray:
    G = _as_G(G)
    K = G.shape[0]
    a = np.zeros(K)
    _load().bko_mgda_enum(K, _ptr(G), _ptr(a))
    return a


def mgda_fw(G, max_iter: int, tol: float):
    """Frank-Wolfe replay; returns (alpha, completed steps)."""
    G = _as_G(G)
    K = G.shape[0]
    a = np.zeros(K)
    it = _load().bko_mgda_fw(K, _ptr(G), max_iter, tol, _ptr(a))
    return a, it


def pcgrad_order(seed: int, step: int, bucket: int, K: int, t: int) -> list[int]:
    o = np.zeros(max(K - 1, 1), dtype=np.int32)
    _load().bko_pcgrad_order(seed, step, bucket, K, t, _ptr(o))
    return [int(v) for v in o[: K - 1]]


def pcgrad(G, seed: int, step: int, bucket: int):
    """PCGrad coefficients beta (d = sum_j beta_j g_j); returns (beta, near_ties)."""
    G = _as_G(G)
    K = G.shape[0]
    b = np.zeros(K)
    ties = np.zeros(1, dtype=np.int32)
    _load().bko_pcgrad(K, _ptr(G), seed, step, bucket, _ptr(b), _ptr(ties))
    return b, int(ties[0])


def pcgrad_alternatives(G, seed: int, step: int, bucket: int, cap: int = 256) -> np.ndarray:
    """Every PCGrad result when each near-tie conflict test may go either way
    (n x K array of beta; one row, equal to pcgrad()'s, when there is no near
    tie).  Raises when there are more than `cap` results."""
    G = _as_G(G)
    K = G.shape[0]
    out = np.zeros((cap, K))
    n = _load().bko_pcgrad_alternatives(K, _ptr(G), seed, step, bucket, cap, _ptr(out))
    if n < 0:
        raise ValueError("more than %d PCGrad alternatives" % cap)
    return out[:n].copy()


def cagrad(G, c: float):
    """CAGrad coefficients; returns (beta, w) with w the simplex minimiser of the dual."""
    G = _as_G(G)
    K = G.shape[0]
    b = np.zeros(K)
    w = np.zeros(K)
    _load().bko_cagrad(K, _ptr(G), c, _ptr(b), _ptr(w))
    return b, w


def conflicts(G):
    """Figure 1 statistics of one bucket: (cos matrix, (mean, std, min), conflict flag)."""
    G = _as_G(G)
    K = G.shape[0]
    cos = np.zeros((K, K))
    stats = np.zeros(3)
    flag = np.zeros(1, dtype=np.int32)
    _load().bko_conflicts(K, _ptr(G), _ptr(cos), _ptr(stats), _ptr(flag))
    return cos, stats, int(flag[0])


def combine(xs, beta, begin: int = 0, n: int | None = None) -> np.ndarray:
    lib = _load()
    K = len(xs)
    if n is None:
        n = xs[0].size - begin
    beta = np.ascontiguousarray(np.asarray(beta, dtype=np.float64))
    d = np.zeros(n, dtype=np.float64)
    lib.bko_combine(K, _dtype_code(xs), _ptr_array(xs), begin, n, _ptr(beta), _ptr(d))
    return d


def resolve(xs, offsets, rule: int, *, b0: int = 0, b1: int | None = None,
            mgda_mode: int = MGDA_EXACT, max_iter: int = 256, tol: float = 1e-12,
            cagrad_c: float = 0.5, seed: int = 0, step: int = 0,
            want_d: bool = True, want_gram: bool = False, n_threads: int = 0):
    """Whole path over buckets [b0, b1); returns dict(beta, d, gram, status)."""
    lib = _load()
    K = len(xs)
    offsets = np.ascontiguousarray(np.asarray(offsets, dtype=np.int64))
    if b1 is None:
        b1 = len(offsets) - 1
    nb = b1 - b0
    beta = np.zeros((nb, K), dtype=np.float64)
    d = np.zeros(int(offsets[b1] - offsets[b0]), dtype=np.float64) if want_d else None
    G = np.zeros((nb, K, K), dtype=np.float64) if want_gram else None
    status = np.zeros(nb, dtype=np.int32)
    p = Params(mgda_mode, max_iter, tol, cagrad_c, seed, step)
    r = lib.bko_resolve(K, _dtype_code(xs), _ptr_array(xs), _ptr(offsets), b0, b1, rule,
                        ctypes.byref(p), _ptr(beta), _ptr(d) if d is not None else None,
                        _ptr(G) if G is not None else None, _ptr(status), n_threads)
    if r != 0:
        raise ValueError("invalid resolve arguments")
    return {"beta": beta, "d": d, "gram": G, "status": status}


def bf16_to_f64(bits: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns (uint16) to float64."""
    return (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
