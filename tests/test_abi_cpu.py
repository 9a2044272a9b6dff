"""CPU-side checks of the C ABI: the library loads, exports every declared
symbol, its host-only plan is bit-exact against the oracle, and argument
errors are rejected synchronously (no GPU needed, no kernel launched)."""
import ctypes
import os
import re

import numpy as np
import pytest

from oracle import oracle as orc
from paper_2606_05613_gb300 import build as nb
from paper_2606_05613_gb300 import inputs
from paper_2606_05613_gb300 import native as bk

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module", autouse=True)
def _built():
    nb.build()
    bk.load()


def _declared_symbols():
    hdrs = [os.path.join(ROOT, "include", f) for f in os.listdir(os.path.join(ROOT, "include"))
            if f.endswith(".h")]
    names = set()
    for h in hdrs:
        src = open(h).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        for m in re.finditer(r"\b(bkmoo_[a-z0-9_]+)\s*\(", src):
            names.add(m.group(1))
    return sorted(names)


def test_library_exports_every_declared_symbol():
    names = _declared_symbols()
    assert "bkmoo_resolve" in names and "bkmoo_plan" in names and "bkmoo_gram" in names
    lib = ctypes.CDLL(bk.LIB_PATH)
    for n in names:
        assert hasattr(lib, n), n


def test_binding_constants_match_the_header():
    """Every enumerator and integer #define of include/bkmoo.h has the same
    value in the binding (the binding restates them; nothing else ties the
    two together)."""
    import os
    h = os.path.join(os.path.dirname(bk.LIB_PATH), "..", "include", "bkmoo.h")
    src = re.sub(r"/\*.*?\*/", "", open(h).read(), flags=re.S)
    consts = {}
    for m in re.finditer(r"#define\s+(BKMOO_[A-Z0-9_]+)\s+\(?\s*(0x[0-9a-fA-F]+|\d+)u?"
                         r"(?:\s*<<\s*(\d+)\s*\))?", src):
        v = int(m.group(2), 0)
        consts[m.group(1)] = v << int(m.group(3)) if m.group(3) else v
    for body in re.findall(r"enum\s*\{(.*?)\}", src, flags=re.S):
        for m in re.finditer(r"(BKMOO_[A-Z0-9_]+)\s*=\s*(\d+)", body):
            consts[m.group(1)] = int(m.group(2))
    assert len(consts) >= 20, sorted(consts)
    for name, v in consts.items():
        assert hasattr(bk, name), name
        assert getattr(bk, name) == v, (name, getattr(bk, name), v)


def test_version_and_status_strings():
    assert bk.bkmoo_version() == 200
    for code in range(8):
        assert bk.bkmoo_status_string(code) != "unknown status"
    assert bk.bkmoo_status_string(99) == "unknown status"


def test_default_params():
    p = bk.bkmoo_default_params()
    assert p.max_iter == 256 and p.tol == 1e-12 and p.cagrad_c == 0.5
    assert p.flags == bk.BKMOO_FLAG_CLOSED_FORM_K2 | bk.BKMOO_FLAG_POLISH


def test_plan_bit_exact_vs_oracle_models():
    for sizes, eb in [(inputs.gpt2_small_sizes(), 4), (inputs.llama32_1b_sizes(), 2),
                      (inputs.qwen3_8b_sizes(), 2)]:
        for bb in (inputs.MiB, 25 * inputs.MiB, 100 * inputs.MiB, 3 * 10**6 + 7):
            np.testing.assert_array_equal(bk.bkmoo_plan(sizes, eb, bb), orc.plan(sizes, eb, bb))
    for mib in inputs.SWEEP_BUCKET_MIB:
        np.testing.assert_array_equal(bk.bkmoo_plan([10**9], 4, mib * inputs.MiB),
                                      orc.plan([10**9], 4, mib * inputs.MiB))


def test_plan_bit_exact_vs_oracle_random_and_golden():
    import json
    g = json.load(open(os.path.join(ROOT, "tests", "golden", "plan_cases.json")))
    for c in g["cases"]:
        assert bk.bkmoo_plan(c["sizes"], c["elem_bytes"], c["bucket_bytes"]).tolist() == c["offsets"]
    rng = np.random.default_rng(0)
    for _ in range(2000):
        sizes = rng.integers(0, 100, size=int(rng.integers(0, 15))).tolist()
        eb = int(rng.integers(1, 5))
        bb = int(rng.integers(1, 300))
        if bb // eb < 1:
            continue
        np.testing.assert_array_equal(bk.bkmoo_plan(sizes, eb, bb), orc.plan(sizes, eb, bb))


def test_plan_buffer_too_small_and_invalid():
    lib = bk.load()
    sizes = np.array([10, 10, 10], dtype=np.int64)
    nb_ = ctypes.c_int64(0)
    out = np.zeros(2, dtype=np.int64)
    r = lib.bkmoo_plan(sizes.ctypes.data, 3, 1, 10, out.ctypes.data, 2, ctypes.byref(nb_))
    assert r == bk.BKMOO_ERR_BUFFER_TOO_SMALL and nb_.value == 3
    assert lib.bkmoo_plan(sizes.ctypes.data, 3, 4, 3, None, 0, ctypes.byref(nb_)) == bk.BKMOO_ERR_INVALID
    assert lib.bkmoo_plan(sizes.ctypes.data, 3, 0, 3, None, 0, ctypes.byref(nb_)) == bk.BKMOO_ERR_INVALID
    bad = np.array([3, -1], dtype=np.int64)
    assert lib.bkmoo_plan(bad.ctypes.data, 2, 1, 3, None, 0, ctypes.byref(nb_)) == bk.BKMOO_ERR_INVALID
    assert lib.bkmoo_plan(sizes.ctypes.data, 3, 1, 3, None, 0, None) == bk.BKMOO_ERR_INVALID


def test_workspace_size_layout():
    off = orc.plan(inputs.qwen3_8b_sizes(), 2, 25 * inputs.MiB)
    n4 = bk.bkmoo_workspace_size(4, bk.BKMOO_BF16, off)
    n8 = bk.bkmoo_workspace_size(8, bk.BKMOO_BF16, off)
    assert n8 > n4 > 0 and n4 % 256 == 0
    # partials dominate: one fp64 triangle per 32768-element bf16 chunk
    chunks = sum((int(off[b + 1] - off[b]) + 32767) // 32768 for b in range(len(off) - 1))
    assert n4 >= chunks * 10 * 8
    with pytest.raises(bk.BkmooError):
        bk.bkmoo_workspace_size(0, bk.BKMOO_F32, off)
    with pytest.raises(bk.BkmooError):
        bk.bkmoo_workspace_size(17, bk.BKMOO_F32, off)
    with pytest.raises(bk.BkmooError):
        bk.bkmoo_workspace_size(4, 7, off)
    with pytest.raises(bk.BkmooError):
        bk.bkmoo_workspace_size(4, bk.BKMOO_F32, [0, 5, 5, 9])   # empty bucket
    with pytest.raises(bk.BkmooError):
        bk.bkmoo_workspace_size(4, bk.BKMOO_F32, [1, 5])          # must start at 0


def test_resolve_rejects_bad_arguments_without_launch():
    """Every check below fails before any CUDA call (fake, aligned addresses)."""
    lib = bk.load()
    off = np.array([0, 1000, 2500], dtype=np.int64)
    base = 1 << 40
    grads = (ctypes.c_void_p * 4)(*[base + i * (1 << 20) for i in range(4)])
    ws = ctypes.c_void_p(base + (1 << 30))
    out = ctypes.c_void_p(base + (1 << 31))
    p = bk.bkmoo_default_params()

    def call(**kw):
        a = dict(grads=grads, K=4, dt=0, off=off.ctypes.data, B=2, rule=0, p=ctypes.byref(p),
                 out=out, odt=0, w=None, st=None, ws=ws, wsb=1 << 30)
        a.update(kw)
        return lib.bkmoo_resolve(a["grads"], a["K"], a["dt"], a["off"], a["B"], a["rule"], a["p"],
                                 a["out"], a["odt"], a["w"], a["st"], a["ws"], a["wsb"], None)

    assert call(K=0) == bk.BKMOO_ERR_INVALID
    assert call(K=17) == bk.BKMOO_ERR_INVALID
    assert call(dt=2) == bk.BKMOO_ERR_INVALID
    assert call(odt=5) == bk.BKMOO_ERR_INVALID
    assert call(rule=4) == bk.BKMOO_ERR_INVALID
    assert call(out=None) == bk.BKMOO_ERR_INVALID
    assert call(out=ctypes.c_void_p(base + (1 << 31) + 4)) == bk.BKMOO_ERR_INVALID   # unaligned
    assert call(ws=ctypes.c_void_p(base + (1 << 30) + 16)) == bk.BKMOO_ERR_INVALID  # ws not 256-B
    assert call(wsb=64) == bk.BKMOO_ERR_WORKSPACE
    bad = np.array([0, 1000, 900], dtype=np.int64)
    assert call(off=bad.ctypes.data) == bk.BKMOO_ERR_INVALID
    g2 = (ctypes.c_void_p * 4)(base, base + 8, base + (2 << 20), base + (3 << 20))
    assert call(grads=g2) == bk.BKMOO_ERR_INVALID                                  # unaligned grad
    # out overlapping a gradient without being exactly it
    assert call(out=ctypes.c_void_p(base + 256)) == bk.BKMOO_ERR_INVALID
    # in place over a gradient with another dtype
    assert call(out=ctypes.c_void_p(base), odt=1) == bk.BKMOO_ERR_INVALID
    q = bk.bkmoo_default_params()
    q.cagrad_c = 1.0
    assert call(p=ctypes.byref(q)) == bk.BKMOO_ERR_INVALID
    q = bk.bkmoo_default_params()
    q.max_iter = -1
    assert call(p=ctypes.byref(q)) == bk.BKMOO_ERR_INVALID


def test_host_staging_size():
    """Three slots, each K input regions and one output region of the largest
    of (window, longest bucket) elements plus 16 bytes, 256-byte aligned."""
    off = np.array([0, 1000, 2500, 2600], dtype=np.int64)

    def expect(K, ei, eo, n):
        r = lambda e: (n * e + 16 + 255) // 256 * 256
        return 3 * (K * r(ei) + r(eo))

    assert bk.bkmoo_host_staging_size(4, bk.BKMOO_BF16, bk.BKMOO_BF16, off) == expect(4, 2, 2, 1500)
    assert bk.bkmoo_host_staging_size(3, bk.BKMOO_F32, bk.BKMOO_BF16, off, 10**6) == \
        expect(3, 4, 2, 10**6)
    with pytest.raises(bk.BkmooError):
        bk.bkmoo_host_staging_size(0, bk.BKMOO_F32, bk.BKMOO_F32, off)
    with pytest.raises(bk.BkmooError):
        bk.bkmoo_host_staging_size(4, bk.BKMOO_F32, 3, off)
    with pytest.raises(bk.BkmooError):
        bk.bkmoo_host_staging_size(4, bk.BKMOO_F32, bk.BKMOO_F32, off, -1)


def test_resolve_host_rejects_bad_arguments_without_launch():
    """Argument errors of bkmoo_resolve_host are returned before any CUDA
    call (fake, aligned addresses)."""
    lib = bk.load()
    off = np.array([0, 1000, 2500], dtype=np.int64)
    base = 1 << 40
    grads = (ctypes.c_void_p * 4)(*[base + i * (1 << 20) for i in range(4)])
    ws = ctypes.c_void_p(base + (1 << 30))
    out = ctypes.c_void_p(base + (1 << 31))
    stg = ctypes.c_void_p(base + (1 << 32))
    p = bk.bkmoo_default_params()
    need = bk.bkmoo_host_staging_size(4, 0, 0, off)

    def call(**kw):
        a = dict(grads=grads, K=4, dt=0, off=off.ctypes.data, B=2, rule=0, p=ctypes.byref(p),
                 out=out, odt=0, ws=ws, wsb=1 << 30, stg=stg, stgb=need)
        a.update(kw)
        return lib.bkmoo_resolve_host(a["grads"], a["K"], a["dt"], a["off"], a["B"], a["rule"],
                                      a["p"], a["out"], a["odt"], None, None, a["ws"], a["wsb"],
                                      a["stg"], a["stgb"], None)

    assert call(K=0) == bk.BKMOO_ERR_INVALID
    assert call(rule=4) == bk.BKMOO_ERR_INVALID
    assert call(odt=2) == bk.BKMOO_ERR_INVALID
    assert call(out=None) == bk.BKMOO_ERR_INVALID
    assert call(stg=None) == bk.BKMOO_ERR_INVALID
    assert call(stg=ctypes.c_void_p(base + (1 << 32) + 128)) == bk.BKMOO_ERR_INVALID  # 256-B
    assert call(wsb=64) == bk.BKMOO_ERR_WORKSPACE
    assert call(stgb=need - 512) == bk.BKMOO_ERR_WORKSPACE        # a bucket does not fit a slot
    assert call(out=ctypes.c_void_p(base + 256)) == bk.BKMOO_ERR_INVALID     # partial overlap
    assert call(out=ctypes.c_void_p(base), odt=1) == bk.BKMOO_ERR_INVALID    # in place, other dtype
    q = bk.bkmoo_default_params()
    q.cagrad_c = -0.5
    assert call(p=ctypes.byref(q)) == bk.BKMOO_ERR_INVALID


def test_resolve_buckets_rejects_bad_ranges_without_launch():
    """bkmoo_resolve_buckets checks its bucket range before any CUDA call;
    an empty range queues nothing (fake, aligned addresses)."""
    lib = bk.load()
    off = np.array([0, 1000, 2500, 4000], dtype=np.int64)
    base = 1 << 40
    grads = (ctypes.c_void_p * 2)(base, base + (1 << 20))
    ws = ctypes.c_void_p(base + (1 << 30))
    out = ctypes.c_void_p(base + (1 << 31))
    p = bk.bkmoo_default_params()

    def call(lo, hi, **kw):
        a = dict(wsb=1 << 30)
        a.update(kw)
        return lib.bkmoo_resolve_buckets(grads, 2, 0, off.ctypes.data, 3, lo, hi, 0,
                                         ctypes.byref(p), out, 0, None, None, ws, a["wsb"],
                                         None)

    assert call(-1, 2) == bk.BKMOO_ERR_INVALID
    assert call(0, 4) == bk.BKMOO_ERR_INVALID
    assert call(2, 1) == bk.BKMOO_ERR_INVALID
    assert call(1, 1) == bk.BKMOO_OK            # empty range: nothing queued
    assert call(0, 3, wsb=64) == bk.BKMOO_ERR_WORKSPACE


def test_plan_one_bucket_global_variant():
    """The conventional (global) MOO is the one-bucket plan: a bucket size
    larger than the model puts every tensor into one bucket."""
    sizes = inputs.gpt2_small_sizes()
    off = bk.bkmoo_plan(sizes, 4, 1 << 62)
    np.testing.assert_array_equal(off, [0, sum(sizes)])
    np.testing.assert_array_equal(off, orc.plan(sizes, 4, 1 << 62))


def test_bench_workload_names():
    import sys
    sys.path.insert(0, ROOT)
    import bench
    w = bench.workload("qwen3-8b-global")
    assert w.bucket_bytes == 1 << 62 and w.K == 4 and w.dtype == "bf16"
    w = bench.workload("sweep-16-1-64M")
    assert w.K == 16 and w.bucket_bytes == 1 << 20 and sum(w.param_sizes) == 64_000_000
    assert bench.workload("sweep-2-100").param_sizes == (1_000_000_000,)


def _aligned_dummies(n):
    """n distinct 16-byte-aligned host addresses (never dereferenced: every
    call below must be rejected before any launch, and on a machine without
    a GPU a launch would fail with a CUDA error rather than read memory)."""
    buf = np.zeros(64 * (n + 1), dtype=np.uint8)
    base = (buf.ctypes.data + 15) & ~15
    return buf, [base + 64 * i for i in range(n)]


def test_gram_noalloc_rejects_bad_arguments_without_launch():
    lib = bk.load()
    keep, ptrs_l = _aligned_dummies(17)
    out = ctypes.c_void_p(ptrs_l[16])

    def call(K, dt, offs, grads=None, out_gram=out, n_buckets=None):
        ptrs = (ctypes.c_void_p * max(K, 1))(*(grads or ptrs_l[:max(K, 1)]))
        offs = np.ascontiguousarray(offs, dtype=np.int64)
        nb_ = len(offs) - 1 if n_buckets is None else n_buckets
        return lib.bkmoo_gram_noalloc(ptrs, K, dt, offs.ctypes.data, nb_, out_gram, None)

    ok_off = [0, 1000, 2500]
    # sizes beyond the static scratch: too many buckets, too many elements
    too_many = np.arange(0, bk.BKMOO_NOALLOC_MAX_BUCKETS + 2, dtype=np.int64)
    assert call(16, bk.BKMOO_F32, too_many) == bk.BKMOO_ERR_WORKSPACE
    assert call(16, bk.BKMOO_F32, [0, 10**10]) == bk.BKMOO_ERR_WORKSPACE
    assert call(4, bk.BKMOO_BF16, [0, 10**11]) == bk.BKMOO_ERR_WORKSPACE
    # invalid arguments
    assert call(0, bk.BKMOO_F32, ok_off) == bk.BKMOO_ERR_INVALID
    assert call(17, bk.BKMOO_F32, ok_off) == bk.BKMOO_ERR_INVALID
    assert call(4, 7, ok_off) == bk.BKMOO_ERR_INVALID
    assert call(4, bk.BKMOO_F32, [0, 1000, 1000]) == bk.BKMOO_ERR_INVALID
    assert call(4, bk.BKMOO_F32, [0, 1000, 900]) == bk.BKMOO_ERR_INVALID
    assert call(4, bk.BKMOO_F32, [5, 1000, 2500]) == bk.BKMOO_ERR_INVALID
    assert call(4, bk.BKMOO_F32, ok_off, n_buckets=-1) == bk.BKMOO_ERR_INVALID
    assert call(4, bk.BKMOO_F32, ok_off, out_gram=None) == bk.BKMOO_ERR_INVALID
    misaligned = list(ptrs_l[:4])
    misaligned[2] += 4
    assert call(4, bk.BKMOO_F32, ok_off, grads=misaligned) == bk.BKMOO_ERR_INVALID
    nulls = list(ptrs_l[:4])
    nulls[1] = None
    assert call(4, bk.BKMOO_F32, ok_off, grads=nulls) == bk.BKMOO_ERR_INVALID
    assert lib.bkmoo_gram_noalloc(None, 4, bk.BKMOO_F32, np.array(ok_off).ctypes.data, 2, out,
                                  None) == bk.BKMOO_ERR_INVALID
    # no bucket: nothing to do, nothing launched
    assert call(4, bk.BKMOO_F32, [0]) == bk.BKMOO_OK
    del keep


def test_selftest_fp64_rejects_bad_arguments_without_launch():
    lib = bk.load()
    keep, p = _aligned_dummies(3)
    assert lib.bkmoo_selftest_fp64(2, p[0], p[1], p[2], 4, None) == bk.BKMOO_ERR_INVALID
    assert lib.bkmoo_selftest_fp64(0, p[0], None, p[2], 4, None) == bk.BKMOO_ERR_INVALID
    assert lib.bkmoo_selftest_fp64(1, None, None, p[2], 4, None) == bk.BKMOO_ERR_INVALID
    assert lib.bkmoo_selftest_fp64(1, p[0], None, p[2], -1, None) == bk.BKMOO_ERR_INVALID
    assert lib.bkmoo_selftest_fp64(1, p[0], None, p[2], 0, None) == bk.BKMOO_OK
    del keep


def test_resolve_path_choice():
    """The per-plan path rule (measured on GB300): the cluster-per-bucket
    fused kernel for K = 2..4 with buckets of at least 2 MiB whose K
    gradients take at most 12 MiB (bf16: 6..12 MiB; CAGrad: fp32 and at
    least 8 MiB), and for tiny plans; the three launches otherwise; the
    flags force either path."""
    F32, BF16 = bk.BKMOO_F32, bk.BKMOO_BF16
    MiB = inputs.MiB

    def plan(n, bucket_bytes, eb):
        return bk.bkmoo_plan([n], eb, bucket_bytes)

    def path(K, dt, rule, mib, eb):
        return bk.bkmoo_resolve_path(K, dt, rule, plan(10**9, int(mib * MiB), eb), 0)

    sweep4 = plan(10**9, 2 * MiB, 4)
    for rule in ("mgda", "pcgrad", "mean"):
        assert bk.bkmoo_resolve_path(4, F32, rule, sweep4, 0) == 1
    # CAGrad: fp32 with at least 8 MiB of gradients per bucket
    assert bk.bkmoo_resolve_path(4, F32, "cagrad", sweep4, 0) == 1
    assert bk.bkmoo_resolve_path(2, F32, "cagrad", sweep4, 0) == 0
    assert bk.bkmoo_resolve_path(3, F32, "cagrad", sweep4, 0) == 0
    assert path(2, F32, "cagrad", 4, 4) == 1
    assert path(3, F32, "cagrad", 4, 4) == 1
    assert path(4, BF16, "cagrad", 2, 2) == 0
    assert bk.bkmoo_resolve_path(8, F32, "mgda", sweep4, 0) == 0
    assert bk.bkmoo_resolve_path(1, F32, "mgda", sweep4, 0) == 0
    # fp32: buckets >= 2 MiB, K x bucket <= 12 MiB
    fp32 = {(2, 1): 0, (2, 2): 1, (2, 4): 1, (2, 6): 1, (2, 8): 0,
            (3, 1): 0, (3, 2): 1, (3, 4): 1, (3, 8): 0,
            (4, 1): 0, (4, 2): 1, (4, 3): 1, (4, 4): 0}
    for (K, mib), want in fp32.items():
        assert path(K, F32, "mgda", mib, 4) == want, (K, mib)
    # bf16: buckets >= 2 MiB, K x bucket in 6..12 MiB
    bf16 = {(2, 2): 0, (2, 4): 1, (2, 8): 0, (3, 2): 1, (3, 4): 1, (3, 8): 0,
            (4, 1): 0, (4, 2): 1, (4, 4): 0}
    for (K, mib), want in bf16.items():
        assert path(K, BF16, "mgda", mib, 2) == want, (K, mib)
    # tiny plans: one launch (K <= 2, at most 8 buckets and 4 Mi elements)
    assert bk.bkmoo_resolve_path(2, F32, "mgda", plan(1 << 20, MiB, 4), 0) == 1
    assert bk.bkmoo_resolve_path(2, F32, "cagrad", plan(1 << 21, MiB, 4), 0) == 1
    assert bk.bkmoo_resolve_path(2, F32, "mgda", plan(1 << 23, MiB, 4), 0) == 0
    assert bk.bkmoo_resolve_path(4, F32, "mgda", plan(1 << 20, MiB, 4), 0) == 0
    # the benchmark's model workloads keep the three launches
    for sizes, eb, K, dt in [(inputs.qwen3_8b_sizes(), 2, 4, BF16),
                             (inputs.gpt2_small_sizes(), 4, 4, F32),
                             (inputs.llama32_1b_sizes(), 2, 8, BF16)]:
        off = bk.bkmoo_plan(sizes, eb, 25 * MiB)
        assert bk.bkmoo_resolve_path(K, dt, "mgda", off, 0) == 0
    # one bucket in range and a third of the elements in small buckets: not
    # chosen; with the small buckets under a tenth of the elements: chosen
    mixed = np.array([0, 2**19] + [2**19 + 3000 * (i + 1) for i in range(100)],
                     dtype=np.int64)
    assert bk.bkmoo_resolve_path(4, F32, "mgda", mixed, 0) == 0
    mostly = np.array([0, 2**19] + [2**19 + 300 * (i + 1) for i in range(100)],
                      dtype=np.int64)
    assert bk.bkmoo_resolve_path(4, F32, "mgda", mostly, 0) == 1
    # flags
    assert bk.bkmoo_resolve_path(4, F32, "mgda", sweep4, bk.BKMOO_FLAG_THREE_PASS) == 0
    assert bk.bkmoo_resolve_path(2, F32, "mgda", sweep4, bk.BKMOO_FLAG_FUSED) == 1
    assert bk.bkmoo_resolve_path(8, F32, "mgda", sweep4, bk.BKMOO_FLAG_FUSED) == 2
    assert bk.bkmoo_resolve_path(16, F32, "mgda", sweep4, bk.BKMOO_FLAG_FUSED) == 0
    assert bk.bkmoo_resolve_path(
        4, F32, "mgda", sweep4, bk.BKMOO_FLAG_FUSED | bk.BKMOO_FLAG_TEST_WITHHOLD) == 2
    assert bk.bkmoo_resolve_path(
        4, F32, "mgda", sweep4, bk.BKMOO_FLAG_FUSED | bk.BKMOO_FLAG_TEST_WITHHOLD_EXCHANGE) == 1
    with pytest.raises(bk.BkmooError):
        bk.bkmoo_resolve_path(0, F32, "mgda", sweep4, 0)
