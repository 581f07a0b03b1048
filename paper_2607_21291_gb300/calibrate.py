"""Similarity-driven retention plan across data-parallel replicas (Sec. 3.3).

Each replica runs the dense calibration forward on its own shard of the
calibration subset and accumulates, per layer, the Eq. 4 partial sums
(sum of per-token cosines, token count) on its device. The only exchange of
the whole path is one sum over replicas of these 2L doubles; every replica
then evaluates Eqs. 5-8 on the host (adadsf_alloc_ratios) and obtains the
same kept counts K_l. The sparse forward itself needs no communication.
"""
from __future__ import annotations

from typing import Optional

import numpy as np
import torch
import torch.distributed as dist

from . import adadsf as A


def allreduce_stats(acc: torch.Tensor, group: Optional[dist.ProcessGroup] = None) -> torch.Tensor:
    """Sum of the per-layer Eq. 4 partial sums over the replicas of `group`
    (identity without an initialised process group). NCCL reduces the device
    tensor in place; other backends reduce a host copy."""
    if not dist.is_available() or not dist.is_initialized() or dist.get_world_size(group) == 1:
        return acc
    if dist.get_backend(group) == "nccl" and acc.is_cuda:
        dist.all_reduce(acc, op=dist.ReduceOp.SUM, group=group)
        return acc
    host = acc.detach().to("cpu", torch.float64).clone()
    dist.all_reduce(host, op=dist.ReduceOp.SUM, group=group)
    return host.to(acc.device)


def similarity_of(acc) -> np.ndarray:
    """s_l = (sum of cosines) / (token count) for acc laid out [L, 2]
    (Eq. 4, evaluated by the library's adadsf_similarity)."""
    return A.adadsf_similarity(acc, A.STATS_TOKEN)


def retention_plan(acc, T: int, t: float, tau: float = 0.05, beta: float = 10.0, flags: int = 0):
    """(s, r, K) from accumulated statistics: Eqs. 5-8 (clamped) and K_l = floor(r_l T)."""
    s = similarity_of(acc)
    r, K = A.adadsf_alloc_ratios(s, t, tau, beta, T, flags)
    return s, r, K


def calibrate(model: "A.DeviceModel", ids: torch.Tensor, t: float, tau: float = 0.05, beta: float = 10.0,
              group: Optional[dist.ProcessGroup] = None, ws: Optional[torch.Tensor] = None, stream=None):
    """Dense forward with statistics on this replica's calibration ids, sum over
    replicas, allocation. Returns (s, r, K) -- identical on every replica."""
    B, T = ids.shape
    L = model.cfg.n_layers
    acc = torch.zeros(2 * L, dtype=torch.float64, device=ids.device)
    out = torch.empty((B, T, model.cfg.d), device=ids.device,
                      dtype=torch.bfloat16 if model.cfg.dtype == A.BF16 else torch.float32)
    A.adadsf_sparse_model_forward(model, ids, [T] * L, out, stats_acc=acc, ws=ws, stream=stream)
    acc = allreduce_stats(acc, group)
    return retention_plan(acc, T, t, tau, beta)
