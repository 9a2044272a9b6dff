"""Per-bucket resolve inside the backward pass (Algorithm 1, Figure 4).

The method intercepts gradients bucket by bucket during the backward pass
("when bucket k is full") and resolves each bucket's conflict before the next
one arrives.  On one GPU the K languages' gradients come from K backward
passes of the same model.  BucketMOO lays them out as K flat buffers in the
bucket order of the method -- tensors in reverse registration order, which is
the order backward produces them, cut into buckets by bkmoo_plan -- and makes
every parameter's .grad a view into the buffer of the language whose backward
pass runs (autograd then accumulates straight into it, no copy).  During the
last language's backward pass a post-accumulate hook counts the tensors of
each bucket; once a bucket is complete its resolve (bkmoo_resolve_buckets) is
queued on a side stream behind an event on the backward stream, so it
overlaps the rest of the backward pass.  finish() resolves what is left
(buckets whose tensors got no gradient), joins the side stream and points
every .grad at the resolved direction d for the optimizer step.

Argument marshalling and bookkeeping only: the resolve runs in the CUDA
library through its C ABI.
"""
from __future__ import annotations

from dataclasses import dataclass
from typing import List, Sequence

import numpy as np

from . import native


@dataclass
class BucketLayout:
    """Flat layout of a model's gradient in bucket order.

    offsets: bucket boundaries (elements) from bkmoo_plan.
    starts[i]: flat position of parameter i (registration order); parameters
      are laid out last-registered first.
    first[i], last[i]: the buckets parameter i spans (last inclusive; a
      parameter larger than a bucket spans several); -1 for empty ones.
    need[b]: number of parameters that touch bucket b.
    """
    offsets: np.ndarray
    starts: List[int]
    first: List[int]
    last: List[int]
    need: List[int]

    @property
    def n_elems(self) -> int:
        return int(self.offsets[-1])

    @property
    def n_buckets(self) -> int:
        return len(self.offsets) - 1


def bucket_layout(sizes: Sequence[int], elem_bytes: int, bucket_bytes: int) -> BucketLayout:
    offsets = native.bkmoo_plan(list(sizes), elem_bytes, bucket_bytes)
    starts = [0] * len(sizes)
    pos = 0
    for i in reversed(range(len(sizes))):
        starts[i] = pos
        pos += int(sizes[i])
    assert pos == int(offsets[-1])
    B = len(offsets) - 1
    first, last = [-1] * len(sizes), [-1] * len(sizes)
    need = [0] * B
    for i, n in enumerate(sizes):
        if n == 0:
            continue
        first[i] = int(np.searchsorted(offsets, starts[i], side="right")) - 1
        last[i] = int(np.searchsorted(offsets, starts[i] + int(n) - 1, side="right")) - 1
        for b in range(first[i], last[i] + 1):
            need[b] += 1
    return BucketLayout(offsets, starts, first, last, need)


class BucketMOO:
    """K per-language gradients of `params`, resolved bucket by bucket.

    Use:
        moo = BucketMOO(model.parameters(), K, bucket_bytes, rule="mgda")
        for k in range(K):
            moo.begin(k)
            loss_k(model, batch_k).backward()
        d = moo.finish()        # every p.grad is now a view of d
        optimizer.step()

    All parameters that require gradients must share one device and one
    dtype, float32 or bfloat16.  The buffers (K gradients, the direction, the
    workspace) are allocated once, here.
    """

    def __init__(self, params, K: int, bucket_bytes: int, rule: str = "mgda",
                 moo_params: "native.bkmoo_params | None" = None):
        import torch
        self.params = [p for p in params if p.requires_grad]
        if not self.params:
            raise ValueError("no parameter requires a gradient")
        dev, dt = self.params[0].device, self.params[0].dtype
        if dt not in (torch.float32, torch.bfloat16):
            raise TypeError("parameters must be float32 or bfloat16, got %s" % dt)
        for p in self.params:
            if p.device != dev or p.dtype != dt:
                raise TypeError("all parameters must share one device and dtype")
        if not 1 <= K <= 16:
            raise ValueError("K must be in [1, 16]")
        self.K, self.rule, self.device, self.dtype = K, rule, dev, dt
        self.moo_params = moo_params if moo_params is not None else native.bkmoo_default_params()
        sizes = [p.numel() for p in self.params]
        self.layout = bucket_layout(sizes, 4 if dt == torch.float32 else 2, bucket_bytes)
        N, B = self.layout.n_elems, self.layout.n_buckets
        self.grads = [torch.zeros(N, dtype=dt, device=dev) for _ in range(K)]
        self.direction = torch.zeros(N, dtype=dt, device=dev)
        self.weights = torch.zeros(B, K, dtype=torch.float32, device=dev)
        self.status = torch.zeros(B, dtype=torch.int32, device=dev)
        self.resolver = native.Resolver(K, dt, self.layout.offsets, dev)
        self.side = torch.cuda.Stream(device=dev)
        self._lang = None
        self._left = list(self.layout.need)
        self._done = [False] * B
        self._hooks = [p.register_post_accumulate_grad_hook(self._make_hook(i))
                       for i, p in enumerate(self.params)]

    def _view(self, buf, i):
        p = self.params[i]
        s = self.layout.starts[i]
        return buf[s:s + p.numel()].view_as(p)

    def begin(self, k: int) -> None:
        """Zero language k's buffer and make every .grad a view into it."""
        if not 0 <= k < self.K:
            raise ValueError("language %d out of range" % k)
        import torch
        # language k's buffer may still be read by last step's resolves
        torch.cuda.current_stream(self.device).wait_stream(self.side)
        self.grads[k].zero_()
        for i, p in enumerate(self.params):
            p.grad = self._view(self.grads[k], i)
        self._lang = k
        if k == self.K - 1:
            self._left = list(self.layout.need)
            self._done = [False] * self.layout.n_buckets

    def _make_hook(self, i):
        def hook(p):
            if self._lang != self.K - 1:
                return
            for b in range(self.layout.first[i], self.layout.last[i] + 1):
                self._left[b] -= 1
                if self._left[b] == 0:
                    self._resolve(b, b + 1)
        return hook

    def _resolve(self, b_lo: int, b_hi: int) -> None:
        import torch
        ev = torch.cuda.Event()
        ev.record(torch.cuda.current_stream(self.device))
        self.side.wait_event(ev)
        self.resolver.resolve_buckets(self.grads, b_lo, b_hi, self.rule, self.direction,
                                      params=self.moo_params, out_weights=self.weights,
                                      out_status=self.status, stream=self.side)
        for b in range(b_lo, b_hi):
            self._done[b] = True

    def finish(self):
        """Resolve the buckets not resolved yet, join the side stream and
        point every .grad at the direction.  Returns the flat direction."""
        import torch
        if self._lang != self.K - 1:
            raise RuntimeError("finish() before the last language's backward pass")
        b = 0
        B = self.layout.n_buckets
        while b < B:                        # runs of unresolved buckets
            if self._done[b]:
                b += 1
                continue
            e = b
            while e < B and not self._done[e]:
                e += 1
            self._resolve(b, e)
            b = e
        torch.cuda.current_stream(self.device).wait_stream(self.side)
        for i, p in enumerate(self.params):
            p.grad = self._view(self.direction, i)
        self._lang = None
        return self.direction

    def remove(self) -> None:
        for h in self._hooks:
            h.remove()
        self._hooks = []
