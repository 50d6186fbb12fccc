"""Sample-sharded FlipFlop fit: the calibration samples of one layer split over ranks.

Section 5 writes both flip-flop updates as expectations over the samples, so with the
samples split into disjoint shards S_1..S_R (one per rank: process / GPU),

    B = 1/(N n) sum_r P_r,   P_r = sum_{k in S_r} (x_k^T A^-1 x_k) g_k g_k^T,
    A = 1/(N m) sum_r Q_r,   Q_r = sum_{k in S_r} (g_k^T B^-1 g_k) x_k x_k^T,

with N = sum_r |S_r|.  Per half-step every rank forms its unscaled partial Gram with
libffh (Cholesky of the replicated factor, the quadratic forms and the weighted Gram of
its shard), the d x d fp32 partial Grams are summed over ranks by the caller's
`reduce_sum` (torch.distributed.all_reduce over NCCL in a multi-GPU run: the one data
exchange of the method), and every rank finishes the update identically: scale, damping,
the tr(A) = n rescale and the stopping statistic delta_t.  The Cholesky factorisations are
replicated, so no factor is ever broadcast.  A process may hold several shards; their
partial Grams are added on the device before the reduction.

Every step of the path runs in libffh kernels; this module only sequences the calls and
the reduction.  The log-likelihood trace of ffh_fit is not kept here.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Callable, List, Optional, Sequence, Tuple

import torch

from . import Handle


@dataclasses.dataclass
class ShardedResult:
    A: torch.Tensor
    B: torch.Tensor
    iters_done: int
    deltas: List[float]
    scales: List[float]


class LibffhSteps:
    """The four steps of a sharded half-step, on the GPU through the libffh C ABI."""

    def __init__(self, handle: Handle):
        self.h = handle

    def partial_gram(self, shards: Sequence[Tuple[torch.Tensor, torch.Tensor]],
                     F: Optional[torch.Tensor]) -> torch.Tensor:
        P = None
        for i, (U, V) in enumerate(shards):
            if i == 0:
                P, _ = self.h.partial_gram(U, V, F)
            else:
                self.h.partial_gram(U, V, F, P_out=P, accumulate=True)
        return P

    def update_from_sum(self, P: torch.Tensor, scale: float) -> torch.Tensor:
        return self.h.update_from_sum(P, scale, F_out=P)

    def normalize_pair(self, A: torch.Tensor, B: torch.Tensor) -> float:
        return self.h.normalize_pair(A, B)

    def relative_change(self, F: torch.Tensor, Fprev: torch.Tensor) -> float:
        return self.h.relative_change(F, Fprev)


def fit_sharded(shards: Sequence[Tuple[torch.Tensor, torch.Tensor]], iters: int,
                tol: float = 0.0, reduce_sum: Optional[Callable[[torch.Tensor], None]] = None,
                n_total: Optional[int] = None, steps=None, handle: Optional[Handle] = None,
                dtype: str = "bf16", damping: float = 0.0) -> ShardedResult:
    """FlipFlop fit of A (n x n) and B (m x m) to the samples of all ranks.

    shards      this rank's (X_r, G_r) pairs (rows x_k^T, g_k^T), usually one pair
    iters, tol  as ffh_fit: A_0 = I, one iteration = B-update then A-update, stop after
                iteration t when delta_t < tol (tol = 0: exactly `iters` iterations)
    reduce_sum  in-place sum of a tensor over all ranks (None: this process holds every
                shard); every rank must call fit_sharded with the same iters and tol
    n_total     total sample count over all ranks (None: summed with reduce_sum)
    steps       the step implementation (default: libffh on the handle `handle`)
    """
    if not shards:
        raise ValueError("no samples on this rank")
    n = shards[0][0].shape[1]
    m = shards[0][1].shape[1]
    own = None
    if steps is None:
        own = handle is None
        handle = handle or Handle(dtype=dtype, damping=damping)
        steps = LibffhSteps(handle)
    reduce = reduce_sum or (lambda t: None)
    try:
        if n_total is None:
            cnt = torch.tensor([float(sum(X.shape[0] for X, _ in shards))], dtype=torch.float64,
                               device=shards[0][0].device)
            reduce(cnt)
            n_total = int(round(float(cnt.item())))
        x_side = [(X, G) for X, G in shards]   # weights from x, Gram of g: the B-update
        g_side = [(G, X) for X, G in shards]   # weights from g, Gram of x: the A-update
        A: Optional[torch.Tensor] = None       # None: A_0 = I (weights ||x_k||^2)
        A_prev = B_prev = None
        deltas, scales = [], []
        t_done = 0
        B = None
        for t in range(1, iters + 1):
            P = steps.partial_gram(x_side, A)
            reduce(P)
            B = steps.update_from_sum(P, 1.0 / (n_total * n))
            Q = steps.partial_gram(g_side, B)
            reduce(Q)
            A = steps.update_from_sum(Q, 1.0 / (n_total * m))
            scales.append(steps.normalize_pair(A, B))
            if A_prev is None:
                delta = math.inf
            else:
                delta = max(steps.relative_change(A, A_prev), steps.relative_change(B, B_prev))
            deltas.append(delta)
            A_prev, B_prev = A.clone(), B.clone()
            t_done = t
            if tol > 0.0 and delta < tol:
                break
        return ShardedResult(A=A, B=B, iters_done=t_done, deltas=deltas, scales=scales)
    finally:
        if own:
            handle.close()
