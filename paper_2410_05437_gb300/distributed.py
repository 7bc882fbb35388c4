"""Data-parallel calibration across processes (one GPU per rank).

The projected forward needs no communication: tokens are independent and every rank holds
the same P^T and W'^T (Sec. 2.2 notes that the method adds no dependency across
mini-batches). Calibration has one exchange step: the ranks' autocorrelation sums S_r and
token counts n_r are added before the eigen-solve, so that C = (sum_r S_r) / (sum_r n_r)
is the estimate over all calibration tokens (Eq. 4).

The sums are reduced in fp64 on the host with torch.distributed (any backend that reduces
CPU tensors, e.g. gloo), then written back into the handle.
"""
from __future__ import annotations

import numpy as np
import torch
import torch.distributed as dist


def allreduce_sum_and_count(S: np.ndarray, n: int, group=None) -> tuple[np.ndarray, int]:
    """Sum of the ranks' autocorrelation sums and token counts (fp64)."""
    t = torch.from_numpy(np.ascontiguousarray(S, dtype=np.float64))
    dist.all_reduce(t, op=dist.ReduceOp.SUM, group=group)
    c = torch.tensor([int(n)], dtype=torch.int64)
    dist.all_reduce(c, op=dist.ReduceOp.SUM, group=group)
    return t.numpy(), int(c.item())


def calib_allreduce(h: int, K: int, group=None, stream=None) -> int:
    """Replaces the accumulator of every rank with the sum over all ranks; returns the
    total token count. Call it on every rank after the local espace_calib_accumulate calls
    and before espace_build_projection."""
    from . import espace_calib_export, espace_calib_import
    S, n = espace_calib_export(h, K, stream)
    S_sum, n_sum = allreduce_sum_and_count(np.triu(S.astype(np.float64)), n, group)
    espace_calib_import(h, S_sum.astype(np.float32), n_sum, stream)
    return n_sum
