"""Sharded PTF calibration over torch.distributed ranks.

The calibration batch of Eqs. 8-10 is split by rows, one shard per rank.
The range needs every row (Eqs. 8-9) and the error of Eq. 10 sums over every
row, so the ranks exchange twice:

  1. each rank's exact (min, max)            -> all-reduce MIN / MAX
  2. each rank's Eq. 10 sums for that range  -> all-gather
  3. every rank adds the gathered sums in rank order and takes the argmin
     (fqvit_calibrate_combine, host code of libfqvit)

All ranks end with the same s, zp and alpha.  Inference after calibration is
independent per token, batch and head, so it needs no exchange at all; this
is the only collective of the path.

The per-rank stages default to the CUDA library on this rank's GPU
(``DeviceCalibOps``).  ``ops`` may be any object with the same two methods,
which is how the exchange protocol is exercised with CPU ranks.
"""
from __future__ import annotations

import torch
import torch.distributed as dist

from . import fqvit


class DeviceCalibOps:
    """Per-rank calibration stages on this process's GPU (libfqvit)."""

    def minmax(self, x: torch.Tensor) -> torch.Tensor:
        return fqvit.calibrate_minmax(x)

    def sse_partial(self, x: torch.Tensor, K: int, mnmx: torch.Tensor) -> torch.Tensor:
        return fqvit.calibrate_sse_partial(x, K, mnmx)


def calibrate_ptf_sharded(x_local: torch.Tensor, K: int = 3, group=None, ops=None):
    """Eqs. 8-10 over the union of every rank's ``x_local`` [rows_r, C] (rows_r may be 0).

    Returns (s float, zp int, alpha uint8[C] CPU tensor, sse_total float64 [C, K+1] CPU
    tensor), identical on every rank of ``group``.
    """
    ops = ops if ops is not None else DeviceCalibOps()
    world = dist.get_world_size(group)
    rows, C = x_local.shape
    dev = x_local.device
    if rows > 0:
        mnmx = ops.minmax(x_local).to(torch.float32)
    else:  # an empty shard contributes nothing to the range
        mnmx = torch.tensor([float("inf"), float("-inf")], dtype=torch.float32, device=dev)
    mn = mnmx[0:1].clone()
    mx = mnmx[1:2].clone()
    dist.all_reduce(mn, op=dist.ReduceOp.MIN, group=group)
    dist.all_reduce(mx, op=dist.ReduceOp.MAX, group=group)
    if not bool(torch.isfinite(mn).item() and torch.isfinite(mx).item()):
        raise ValueError("calibrate_ptf_sharded: no calibration rows on any rank")
    if rows > 0:
        part = ops.sse_partial(x_local, K, torch.cat([mn, mx])).to(torch.float64)
    else:
        part = torch.zeros(C, K + 1, dtype=torch.float64, device=dev)
    parts = [torch.empty_like(part) for _ in range(world)]
    dist.all_gather(parts, part.contiguous(), group=group)
    stacked = torch.stack([p.cpu() for p in parts])
    return fqvit.calibrate_combine(stacked, float(mn.item()), float(mx.item()), K)
