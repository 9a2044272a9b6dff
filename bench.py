#!/usr/bin/env python
"""Benchmark of the bucket-level MOO resolve on GB300.

One step = one full resolve (Gram -> per-bucket solve -> combination) over
every bucket of a K-language gradient set, through the C ABI.  Default
workload: Qwen3-8B-shaped, K = 4 languages, bf16 gradients of 8,190,735,360
parameters each (65.5 GB resident), 25 MiB buckets (672), MGDA.

Prints ONE JSON line (rank 0).  `value` is the throughput in GB/s of
K-language gradient bytes resolved (K * N * 2 bytes per step) over all ranks;
`ms_per_step` the device time of one step.  Timed with CUDA events on the
stream the kernels run on, after warm-up; the inputs (65.5 GB) are far larger
than L2, so no flush is needed between steps.

--impl reference times the fp64 CPU oracle (the only reference this method
has: the paper ships no implementation) on a bounded sample of the same
workload's buckets, on the host cores.
"""
from __future__ import annotations

import argparse
import ctypes
import hashlib
import json
import os
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

GB = 1e9


def _args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="qwen3-8b",
                    help="qwen3-8b | llama3.2-1b | gpt2-small | tiny | sweep-K-MiB[-<n>M]; "
                         "append -global for one bucket over every parameter")
    ap.add_argument("--rule", default="mgda", choices=["mgda", "pcgrad", "cagrad", "mean"])
    ap.add_argument("--path", default="auto", choices=["auto", "fused", "3pass"],
                    help="auto: the library's per-plan choice; fused: one launch per step "
                         "(re-read from L2); 3pass: Gram, solve and combination launches")
    ap.add_argument("--hook", action="store_true",
                    help="time a synthetic training step of a GPT-2-small-shaped transformer "
                         "with the per-bucket resolve inside the backward pass (BucketMOO) "
                         "against plain gradient accumulation")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--e2e-steps", type=int, default=6)
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    return ap.parse_args()


def workload(name):
    from paper_2606_05613_gb300 import inputs
    if name == "qwen3-8b":
        return inputs.qwen3_8b()
    if name == "llama3.2-1b":
        return inputs.llama32_1b()
    if name == "gpt2-small":
        return inputs.gpt2_small()
    if name == "tiny":
        return inputs.tiny()
    if name.startswith("qwen3-8b-") and name.endswith("layers"):
        return inputs.qwen3_8b_layers(int(name[len("qwen3-8b-"):-len("layers")]))
    if name.endswith("-global"):
        # the conventional (global) MOO of the paper's Table 2: one bucket
        # holding every parameter
        import dataclasses
        w = workload(name[: -len("-global")])
        return dataclasses.replace(w, name=w.name + "-global", bucket_bytes=1 << 62)
    if name.startswith("sweep-"):
        # sweep-K-MiB, or sweep-K-MiB-<n>M for a vector of n million elements
        parts = name.split("-")
        n = int(parts[3][:-1]) * 1_000_000 if len(parts) > 3 else 1_000_000_000
        return inputs.sweep(int(parts[1]), int(parts[2]), n)
    raise SystemExit("unknown workload " + name)


def _dist():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def _peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


def _source_digest(files):
    h = hashlib.sha256()
    for f in files:
        with open(os.path.join(ROOT, f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def _traffic_per_elem(kernel):
    """DRAM bytes per element of `kernel` from the committed ncu summary, or
    None when the summary is missing or the kernel source changed since."""
    p = os.path.join(ROOT, "profiles", "traffic_%s.txt" % kernel)
    if not os.path.exists(p):
        return None
    vals = {}
    for line in open(p):
        if ":" in line and not line.startswith("#"):
            k, v = line.split(":", 1)
            vals[k.strip()] = v.strip()
    try:
        files = vals["sources"].split()
        if _source_digest(files) != vals["source_digest"]:
            return None
        return float(vals["dram_bytes_per_elem"])
    except (KeyError, ValueError, OSError):
        return None


class ClockSampler:
    """nvidia-smi clocks / throttle reasons sampled every 200 ms."""

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(prefix="bkmoo_clocks_", suffix=".csv")
        os.close(fd)
        q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), "--query-gpu=" + q,
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        rows = []
        for line in open(self.path):
            parts = [x.strip() for x in line.split(",")]
            if len(parts) >= 9:
                rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return None
        sm = sorted(float(r[1]) for r in rows if r[1].replace(".", "").isdigit())
        mx = max(float(r[2]) for r in rows if r[2].replace(".", "").isdigit())
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({n for r in rows for n, v in zip(names, r[5:9]) if v == "Active"})
        return {"sm_mhz": sm[len(sm) // 2] if sm else None, "sm_max_mhz": mx,
                "reasons": reasons, "samples": len(rows)}


def launches_per_step(w, off, fused):
    """Kernels of this library one resolve launches: the fused kernel; or
    Gram pass, solve and combination, plus the group pre-reduction of the
    chunk partials when a bucket has more than 1024 chunks."""
    import numpy as np
    if fused and w.K <= 8:
        return 1
    ch = 16384 if w.dtype == "f32" else 32768
    longest = int(np.max(np.diff(np.asarray(off, dtype=np.int64))))
    return 3 + (1 if (longest + ch - 1) // ch > 1024 else 0)


def base_config(w, off, rule):
    """The workload description both arms print."""
    return {"workload": w.name, "K": w.K, "grad_dtype": w.dtype, "out_dtype": w.dtype,
            "rule": rule, "n_elems_per_language": int(off[-1]), "n_buckets": len(off) - 1,
            "bucket_bytes": w.bucket_bytes}


def reduce_over_ranks(ms_step, grad_bytes, device):
    """Whole-job throughput: the gradient bytes of all ranks over the slowest
    rank's time per step.  Returns (max ms per step, GB/s).  One rank: no
    collective."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return ms_step, grad_bytes / (ms_step * 1e-3) / GB
    t = torch.tensor([ms_step], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    u = torch.tensor([float(grad_bytes)], dtype=torch.float64, device=device)
    dist.all_reduce(u, op=dist.ReduceOp.SUM)
    ms = float(t.item())
    return ms, float(u.item()) / (ms * 1e-3) / GB


def cpu_sample(w, offsets, cores):
    """A bounded sample of the workload for the CPU oracle: one bucket per
    core, spread over the model, host-generated with the same generator.
    Returns (K host arrays, sample offsets, the picked bucket indices)."""
    import numpy as np
    import torch

    from paper_2606_05613_gb300 import inputs
    B = len(offsets) - 1
    n_s = min(B, max(1, cores))
    picks = sorted(set(int(round(i * (B - 1) / max(1, n_s - 1))) for i in range(n_s)))
    sub_off = [0]
    for b in picks:
        sub_off.append(sub_off[-1] + int(offsets[b + 1] - offsets[b]))
    hv = [np.empty(sub_off[-1], dtype=np.float32 if w.dtype == "f32" else np.uint16)
          for _ in range(w.K)]
    tdt = torch.float32 if w.dtype == "f32" else torch.bfloat16
    for i, b in enumerate(picks):
        lo, hi = int(offsets[b]), int(offsets[b + 1])
        bufs = [torch.empty(hi - lo, dtype=tdt) for _ in range(w.K)]
        _generate_bucket(w, offsets, b, bufs)
        for k in range(w.K):
            hv[k][sub_off[i]:sub_off[i + 1]] = inputs.host_view(bufs[k])
    return hv, np.array(sub_off, dtype=np.int64), picks


def oracle_pass(hv, sub_off, rule, cores):
    """One pass of the oracle, as it stands, over the sample; returns seconds."""
    from oracle import oracle as orc
    t0 = time.perf_counter()
    orc.resolve(hv, sub_off, getattr(orc, rule.upper()), n_threads=cores)
    return time.perf_counter() - t0


def cpu_baseline(w, offsets, seconds, n_threads=0, rule="mgda"):
    """The oracle on a bounded sample of the workload's buckets, repeated
    until about `seconds` of wall time; returns (GB/s of gradient bytes,
    cores, sample description, seconds per pass)."""
    from oracle import oracle as orc
    cores = orc.max_threads() if n_threads <= 0 else n_threads
    hv, sub_off, picks = cpu_sample(w, offsets, cores)
    dt, passes = 0.0, 0
    while True:
        dt += oracle_pass(hv, sub_off, rule, cores)
        passes += 1
        if dt >= seconds:
            break
    grad_bytes = w.K * int(sub_off[-1]) * w.elem_bytes * passes
    sample = ("%d of %d buckets (%d elements per language), %d passes, %s"
              % (len(picks), len(offsets) - 1, int(sub_off[-1]), passes, rule))
    return grad_bytes / dt / GB, cores, sample, dt / passes


def _generate_bucket(w, offsets, b, bufs):
    """Fill bufs (one CPU tensor per language, bucket length) with bucket b of
    the workload, via the shared generator."""
    import numpy as np

    from paper_2606_05613_gb300 import inputs
    lo, hi = int(offsets[b]), int(offsets[b + 1])
    # a view of the flat layout restricted to bucket b: shift offsets
    # the generator needs the full plan (draws, tensor boundaries): hand it
    # windows that store only the bucket's range
    inputs.generate(w, offsets, "cpu", buckets=[b], out=[_Window(bf, lo) for bf in bufs])


class _Window:
    """Slice-assignable stand-in for a full-length tensor that stores only
    [lo, lo + len(buf))."""

    def __init__(self, buf, lo):
        self.buf, self.lo = buf, lo

    def __getitem__(self, sl):
        return self.buf[sl.start - self.lo: sl.stop - self.lo]


def run_reference(a):
    """Reference arm: the fp64 CPU oracle on the host cores."""
    ws, rank, _ = _dist()
    if rank != 0:
        return
    from oracle import oracle as orc
    from paper_2606_05613_gb300 import inputs  # noqa: F401
    orc.build()
    w = workload(a.workload)
    off = orc.plan(w.param_sizes, w.elem_bytes, w.bucket_bytes)
    # each step: one oracle pass over a sample of one bucket per core (the
    # sample is generated once, outside the timed passes)
    cores = orc.max_threads()
    hv, sub_off, picks = cpu_sample(w, off, cores)
    for _ in range(a.warmup):
        oracle_pass(hv, sub_off, a.rule, cores)
    times = [oracle_pass(hv, sub_off, a.rule, cores) for _ in range(a.steps)]
    step_bytes = w.K * int(sub_off[-1]) * w.elem_bytes
    v = step_bytes * len(times) / sum(times) / GB
    sample = ("%d of %d buckets (%d elements per language), one pass per step, %s"
              % (len(picks), len(off) - 1, int(sub_off[-1]), a.rule))
    line = {
        "impl": "reference", "metric": "bucket-MOO resolve GB/s of K-language grads",
        "value": v, "unit": "GB/s", "n_gpus": a.gpus, "steps": a.steps, "warmup": a.warmup,
        "ms_per_step": 1e3 * sum(times) / len(times), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": dict(base_config(w, off, a.rule),
                       parallelism="host cores (OpenMP over buckets)",
                       path="fp64 CPU oracle (plain C) on a sample of buckets"),
        "cpu_baseline": {"value": v, "unit": "GB/s", "cores": cores, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": v, "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def run_hook(a):
    """One training step = K languages' forward + backward on their own
    synthetic token batches.  BucketMOO: gradients land in the bucket layout
    and each bucket is resolved (MGDA) on a side stream as soon as the last
    language's backward pass completes it (Algorithm 1); baseline: the same
    passes accumulating into .grad (the averaged update of plain fine-tuning).
    Prints one JSON line with both step times."""
    import numpy as np
    import torch

    from paper_2606_05613_gb300 import build as nb
    from paper_2606_05613_gb300 import native as bk
    from paper_2606_05613_gb300.hook import BucketMOO
    nb.build()
    bk.load()
    dev = torch.device("cuda", 0)
    torch.manual_seed(0)
    V, D, L, H, F, T, Bt, K = 50257, 768, 12, 12, 3072, 512, 8, 4

    class Model(torch.nn.Module):
        def __init__(self):
            super().__init__()
            self.emb = torch.nn.Embedding(V, D)
            self.pos = torch.nn.Embedding(T, D)
            layer = torch.nn.TransformerEncoderLayer(D, H, F, dropout=0.0, activation="gelu",
                                                     batch_first=True, norm_first=True)
            self.body = torch.nn.TransformerEncoder(layer, L, enable_nested_tensor=False)
            self.norm = torch.nn.LayerNorm(D)

        def forward(self, x):
            h = self.emb(x) + self.pos.weight[: x.shape[1]]
            mask = torch.nn.Transformer.generate_square_subsequent_mask(x.shape[1], device=x.device)
            h = self.norm(self.body(h, mask=mask, is_causal=True))
            return h @ self.emb.weight.t()          # tied head

    model = Model().to(dev)
    params = [p for p in model.parameters() if p.requires_grad]
    n_params = sum(p.numel() for p in params)
    gen = torch.Generator(device=dev).manual_seed(1)
    batches = [torch.randint(0, V, (Bt, T + 1), device=dev, generator=gen) for _ in range(K)]

    def loss_of(k):
        x = batches[k]
        logits = model(x[:, :-1])
        return torch.nn.functional.cross_entropy(logits.reshape(-1, V), x[:, 1:].reshape(-1))

    moo = BucketMOO(params, K, 25 << 20, rule=a.rule if a.rule != "mean" else "mgda")

    def step_moo():
        for k in range(K):
            moo.begin(k)
            loss_of(k).backward()
        moo.finish()

    def step_plain():
        for p in params:
            p.grad = None
        for k in range(K):
            (loss_of(k) / K).backward()

    def timed(fn):
        for _ in range(a.warmup):
            fn()
        torch.cuda.synchronize(dev)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(a.steps):
            fn()
        e1.record()
        torch.cuda.synchronize(dev)
        return e0.elapsed_time(e1) / a.steps

    t_plain = timed(step_plain)
    t_moo = timed(step_moo)
    moo.remove()
    print(json.dumps({
        "metric": "training step with per-bucket MOO resolve inside the backward pass",
        "unit": "ms", "n_gpus": 1, "steps": a.steps, "warmup": a.warmup, "data": "synthetic",
        "dtype": "f32", "higher_is_better": False,
        "config": {"model": "GPT-2-small-shaped transformer (12 x 768, tied 50257 vocab)",
                   "n_params": n_params, "K": K, "batch_per_language": Bt, "seq_len": T,
                   "rule": moo.rule, "n_buckets": moo.layout.n_buckets,
                   "bucket_bytes": 25 << 20},
        "ms_per_step_bucket_moo": t_moo, "ms_per_step_plain_accumulation": t_plain,
        "overhead": t_moo / t_plain - 1.0,
        "bucket_status_counts": {str(k): int(v) for k, v in
                                 zip(*np.unique(moo.status.cpu().numpy(), return_counts=True))},
    }), flush=True)


def main():
    a = _args()
    if a.impl == "reference":
        run_reference(a)
        return
    if a.hook:
        run_hook(a)
        return
    import numpy as np
    import torch

    from paper_2606_05613_gb300 import build as nb
    from paper_2606_05613_gb300 import inputs
    from paper_2606_05613_gb300 import native as bk

    world, rank, local = _dist()
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if rank == 0:
        nb.build()
    if world > 1:
        torch.distributed.barrier()
    bk.load()

    w = workload(a.workload)
    off = bk.bkmoo_plan(w.param_sizes, w.elem_bytes, w.bucket_bytes)
    B = len(off) - 1
    N = int(off[-1])
    tdt = torch.float32 if w.dtype == "f32" else torch.bfloat16
    grads = inputs.generate(w, off, dev)
    out = torch.empty(N, dtype=tdt, device=dev)
    beta = torch.empty(B, w.K, dtype=torch.float32, device=dev)
    status = torch.empty(B, dtype=torch.int32, device=dev)
    res = bk.Resolver(w.K, tdt, off, dev)
    stream = torch.cuda.current_stream(dev)
    params = bk.bkmoo_default_params()
    if w.max_iter != 256:
        params.max_iter = w.max_iter
    if a.path == "fused":
        params.flags |= bk.BKMOO_FLAG_FUSED
    elif a.path == "3pass":
        params.flags |= bk.BKMOO_FLAG_THREE_PASS
    path_id = bk.bkmoo_resolve_path(w.K, bk.BKMOO_F32 if tdt == torch.float32 else bk.BKMOO_BF16,
                                    a.rule, off, params.flags)
    fused = path_id != 0

    def step(evs=None):
        if evs is not None:
            arr = (ctypes.c_void_p * 4)(*[e.cuda_event for e in evs])
            params.events = ctypes.cast(arr, ctypes.c_void_p).value
            step.keep = arr
        else:
            params.events = None
        res.resolve(grads, a.rule, out, params=params, out_weights=beta, out_status=status)

    for _ in range(a.warmup):
        step()
    torch.cuda.synchronize(dev)
    if res.status() != 0:
        raise SystemExit("resolve failed: " + bk.bkmoo_status_string(res.status()))
    st = status.cpu().numpy()

    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(a.steps)]
    for e4 in evs:           # create the underlying CUDA events before timing
        for e in e4:
            e.record(stream)
    torch.cuda.synchronize(dev)
    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.3)
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize(dev)
    t0 = time.perf_counter()
    for i in range(a.steps):
        step(evs[i])
    torch.cuda.synchronize(dev)
    wall = time.perf_counter() - t0
    if world > 1:
        torch.distributed.barrier()
    clk = clocks.stop()

    total_ms = evs[0][0].elapsed_time(evs[-1][3])
    per = np.array([[e4[0].elapsed_time(e4[1]), e4[1].elapsed_time(e4[2]),
                     e4[2].elapsed_time(e4[3])] for e4 in evs])
    grad_bytes = w.K * N * w.elem_bytes
    ms_step, value = reduce_over_ranks(total_ms / a.steps, grad_bytes, dev)

    peak, peak_kind = _peaks()
    e_in = w.elem_bytes
    e_out = out.element_size()
    if fused:   # one launch: Gram + solve + combination, re-read from L2
        kern = {"fused": (per[:, 0].mean(), (w.K * e_in + e_out) * N, "fused")}
        dom = "fused"
    else:
        kern = {"gram": (per[:, 0].mean(), w.K * e_in * N, "gram"),
                "solve": (per[:, 1].mean(), None, "solve"),
                "combine": (per[:, 2].mean(), (w.K * e_in + e_out) * N, "combine")}
        dom = max(("gram", "combine"), key=lambda k: kern[k][0])
    dms, dbytes, _ = kern[dom]
    achieved = dbytes / (dms * 1e-3) / GB
    tpe = _traffic_per_elem("%s_%s_k%d" % (dom, w.dtype, w.K))
    roofline = {"bound": "hbm", "kernel": dom, "achieved": achieved, "peak": peak,
                "unit": "GB/s", "frac": achieved / peak, "peak_kind": peak_kind,
                "traffic": (tpe * N if tpe is not None else None),
                "algorithmic_bytes": dbytes,
                "avg_ms": {"gram": float(per[:, 0].mean()), "solve": float(per[:, 1].mean()),
                           "combine": float(per[:, 2].mean())}}
    step_bytes_2k1 = (2 * w.K * e_in + e_out) * N
    step_bytes_k1 = (w.K * e_in + e_out) * N

    line = {
        "metric": "bucket-MOO resolve GB/s of K-language grads",
        "value": value, "unit": "GB/s", "n_gpus": world, "steps": a.steps, "warmup": a.warmup,
        "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f32" if w.dtype == "f32" else "bf16",
        "data": "synthetic",
        "config": dict(base_config(w, off, a.rule),
                       l2=("inputs (%.1f GB) >> L2, no flush" % (grad_bytes / GB)
                           if grad_bytes > 4 * 126e6 else
                           "inputs (%.3f GB) fit in L2 and are not flushed: L2-resident "
                           "timing" % (grad_bytes / GB)),
                       parallelism="replicas" if world > 1 else "1 GPU",
                       path=({1: "fused: one launch, a thread-block cluster per bucket, "
                                    "combination re-reads each bucket from L2",
                              2: "fused: one persistent launch, groups of CTAs per bucket, "
                                 "combination re-reads each bucket from L2"}.get(
                                  path_id, "gram -> solve -> combine (3 launches)")
                             + (" (chosen per plan)" if a.path == "auto" else ""))),
        "roofline": roofline,
        "step_roofline": {"bytes_2k1": step_bytes_2k1, "bytes_k1": step_bytes_k1,
                          "frac_2k1_of_measured": step_bytes_2k1 / (ms_step * 1e-3) / GB / peak,
                          "frac_k1_of_measured": step_bytes_k1 / (ms_step * 1e-3) / GB / peak,
                          "frac_2k1_of_8tbs": step_bytes_2k1 / (ms_step * 1e-3) / GB / 8000.0},
        "gpu_launches": launches_per_step(w, off, fused) * a.steps,
        "clocks": clk,
        "bucket_status_counts": {str(k): int((st == k).sum()) for k in sorted(set(st.tolist()))},
        "host_wall_ms_per_step": 1e3 * wall / a.steps,
    }

    # end to end through the public API with host buffers (pinned)
    if not a.no_e2e:
        line["e2e"] = e2e_measure(a, w, off, grads, res, params, dev, tdt)
    if rank == 0 and world == 1 and not a.no_cpu_baseline:
        del grads
        torch.cuda.empty_cache()
        v, cores, sample, _ = cpu_baseline(w, off, a.cpu_seconds, rule=a.rule)
        line["cpu_baseline"] = {"value": v, "unit": "GB/s", "cores": cores, "kind": "oracle",
                                "sample": sample}
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()


def e2e_measure(a, w, off, grads, res, params, dev, tdt):
    """End to end through the public host-memory entry point
    (bkmoo_resolve_host): page-locked host gradients in, page-locked host
    direction out, every byte crossing the host link inside the timed region
    (the call overlaps the copies with the resolve)."""
    import torch

    from paper_2606_05613_gb300 import native as bk
    # Page-locked host memory per rank: at most half of the available host
    # memory shared by the ranks on this node; when the whole gradient set
    # does not fit, the measurement covers the longest prefix of whole
    # buckets that does (and says so).
    N_all = int(off[-1])
    e_el = w.elem_bytes
    avail = _mem_available_bytes()
    local_ranks = int(os.environ.get("LOCAL_WORLD_SIZE", os.environ.get("WORLD_SIZE", "1")))
    budget = 0.5 * avail / max(1, local_ranks) if avail else float("inf")
    B_all = len(off) - 1
    B_e2e = B_all
    while B_e2e > 1 and (w.K + 1) * int(off[B_e2e]) * e_el > budget:
        B_e2e -= 1
    N = int(off[B_e2e])
    sample = None if B_e2e == B_all else "first %d of %d buckets (%d of %d elements per language)" % (
        B_e2e, B_all, N, N_all)
    if B_e2e < B_all:
        off = off[:B_e2e + 1]
        res = bk.Resolver(w.K, tdt, off, dev)
    try:
        host = [torch.empty(N, dtype=tdt, pin_memory=True) for _ in range(w.K)]
        host_out = torch.empty(N, dtype=tdt, pin_memory=True)
    except RuntimeError as e:
        return {"value": None, "unit": "GB/s", "error": "pinned host allocation failed: %s"
                % str(e)[:120]}
    for k in range(w.K):
        host[k].copy_(grads[k][:N])
    torch.cuda.synchronize(dev)
    out_dt = bk.BKMOO_F32 if tdt == torch.float32 else bk.BKMOO_BF16
    # windows of about an eighth of the model, at most 64 Mi elements per
    # language, never shorter than the longest bucket
    longest = int((off[1:] - off[:-1]).max())
    window = max(longest, min(1 << 26, N // 8))
    staging = torch.empty(res.staging_size(out_dt, window), dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream(dev)
    params.events = None

    def one():
        res.resolve_host(host, a.rule, host_out, staging, params=params)
        stream.synchronize()

    one()
    if res.status() != 0:
        raise SystemExit("host resolve failed: " + bk.bkmoo_status_string(res.status()))
    t0 = time.perf_counter()
    for _ in range(a.e2e_steps):
        one()
    dt = (time.perf_counter() - t0) / a.e2e_steps
    gb = w.K * N * w.elem_bytes
    gbo = N * host_out.element_size()
    r = {"value": gb / dt / GB, "unit": "GB/s", "ms_per_step": dt * 1e3,
         "h2d_bytes_per_step": gb, "d2h_bytes_per_step": gbo,
         "steps": a.e2e_steps, "api": "bkmoo_resolve_host",
         "window_elems": window, "staging_bytes": staging.numel(),
         "link_GBps": (gb + gbo) / dt / GB}
    del staging
    link = link_bound(host, host_out, window, dev, reps=max(2, a.e2e_steps // 2))
    r["link_bound"] = link
    r["ms_over_link_bound"] = dt * 1e3 / link["both_ms"]
    r["ms_over_one_way_h2d"] = dt * 1e3 / link["h2d_only_ms"]
    if sample:
        r["sample"] = sample
    return r


def link_bound(host, host_out, window, dev, reps=2):
    """What the host link itself allows for the end-to-end step, measured on
    the same page-locked buffers with the same window length: every input
    window copied host -> device into one of two device slots (one stream),
    every output window copied device -> host (another stream), each alone
    and both at once (window w's input beside window w-1's output).  No
    kernel runs; the slots' contents are discarded."""
    import torch

    K, N = len(host), host[0].numel()
    slots = [[torch.empty(window, dtype=host[0].dtype, device=dev) for _ in range(K)]
             for _ in range(2)]
    outs = [torch.empty(window, dtype=host_out.dtype, device=dev) for _ in range(2)]
    s_in, s_out = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
    wins = [(lo, min(lo + window, N)) for lo in range(0, N, window)]

    def h2d(i, lo, hi):
        with torch.cuda.stream(s_in):
            for k in range(K):
                slots[i % 2][k][:hi - lo].copy_(host[k][lo:hi], non_blocking=True)

    def d2h(i, lo, hi):
        with torch.cuda.stream(s_out):
            host_out[lo:hi].copy_(outs[i % 2][:hi - lo], non_blocking=True)

    def timed(fn):
        best = None
        for _ in range(reps):
            torch.cuda.synchronize(dev)
            t0 = time.perf_counter()
            fn()
            torch.cuda.synchronize(dev)
            t = time.perf_counter() - t0
            best = t if best is None else min(best, t)
        return best * 1e3

    def only_in():
        for i, (lo, hi) in enumerate(wins):
            h2d(i, lo, hi)

    def only_out():
        for i, (lo, hi) in enumerate(wins):
            d2h(i, lo, hi)

    def both():
        for i, (lo, hi) in enumerate(wins):
            h2d(i, lo, hi)
            if i:
                d2h(i - 1, *wins[i - 1])
        d2h(len(wins) - 1, *wins[-1])

    r = {"h2d_only_ms": timed(only_in), "d2h_only_ms": timed(only_out), "both_ms": timed(both)}
    gb_in = sum(t.numel() * t.element_size() for t in host)
    r["h2d_GBps"] = gb_in / r["h2d_only_ms"] * 1e3 / GB
    r["d2h_GBps"] = host_out.numel() * host_out.element_size() / r["d2h_only_ms"] * 1e3 / GB
    r["reps"] = reps
    del slots, outs
    return r


def _mem_available_bytes():
    """MemAvailable of /proc/meminfo in bytes, or None."""
    try:
        with open("/proc/meminfo") as f:
            for line in f:
                if line.startswith("MemAvailable:"):
                    return int(line.split()[1]) * 1024
    except OSError:
        pass
    return None


if __name__ == "__main__":
    main()
