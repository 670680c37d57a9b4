"""Several GPUs, one process each: which traces a rank simulates and the
small cross-rank reductions of the benchmark and of the global best point.

Simulations are independent, so ranks share nothing while they run.  After a
run each rank holds per-point partial sums over its own traces
(`Sim.point_sums`); adding them up over the ranks and handing the totals to
`hxsim.best_of_sums` gives the best point of the whole grid (Sec. 4.3's
argmin over every trace).  Works with any torch.distributed backend (NCCL on
GPUs, gloo on CPUs).
"""
from __future__ import annotations

import os
from typing import Tuple

import numpy as np


def env() -> Tuple[int, int, int]:
    """(world size, rank, local rank) from the torchrun environment."""
    return (int(os.environ.get("WORLD_SIZE", "1")), int(os.environ.get("RANK", "0")),
            int(os.environ.get("LOCAL_RANK", "0")))


def first_trace(rank: int, traces_per_rank: int) -> int:
    """Index of the first trace seed of a rank's shard (weak scaling: every
    rank simulates its own `traces_per_rank` traces)."""
    return rank * traces_per_rank


def _device():
    import torch
    import torch.distributed as d
    return torch.device("cuda", torch.cuda.current_device()) if d.get_backend() == "nccl" else torch.device("cpu")


def max_over_ranks(x: float) -> float:
    import torch
    import torch.distributed as d
    if not d.is_initialized() or d.get_world_size() == 1:
        return float(x)
    t = torch.tensor([float(x)], dtype=torch.float64, device=_device())
    d.all_reduce(t, op=d.ReduceOp.MAX)
    return float(t.item())


def sum_over_ranks(v: np.ndarray) -> np.ndarray:
    """Element-wise int64 sum of a vector over all ranks."""
    import torch
    import torch.distributed as d
    v = np.ascontiguousarray(v, dtype=np.int64)
    if not d.is_initialized() or d.get_world_size() == 1:
        return v.copy()
    t = torch.from_numpy(v.copy()).to(_device())
    d.all_reduce(t, op=d.ReduceOp.SUM)
    return t.cpu().numpy()


def global_point_sums(sum_p95: np.ndarray, sum_slo: np.ndarray, n_failed: np.ndarray, n_queries: int):
    """Add every rank's per-point partial sums and query count."""
    packed = np.concatenate([np.asarray(sum_p95, np.int64), np.asarray(sum_slo, np.int64),
                             np.asarray(n_failed, np.int64), np.array([n_queries], np.int64)])
    tot = sum_over_ranks(packed)
    P = len(sum_p95)
    return tot[:P], tot[P:2 * P], tot[2 * P:3 * P].astype(np.int32), int(tot[-1])
