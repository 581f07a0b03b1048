"""The N > 1 path on CPU: two gloo ranks each hold the Eq. 4 partial sums of
their own shard of the calibration rows; after the exchange both derive the
same retention plan, equal to the single-process plan on all rows."""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from oracle import adadsf_oracle as O


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, shards, T, t, out_q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    from paper_2607_21291_gb300 import calibrate as C
    L = len(shards[rank])
    acc = torch.zeros(2 * L, dtype=torch.float64)
    for l, (a, b) in enumerate(shards[rank]):
        acc[2 * l:2 * l + 2] = torch.tensor(O.cos_sim_stat(a, b), dtype=torch.float64)
    acc = C.allreduce_stats(acc)
    s, r, K = C.retention_plan(acc, T, t)
    out_q.put((rank, s.tolist(), r.tolist(), K.tolist()))
    dist.barrier()
    dist.destroy_process_group()


def test_two_rank_calibration_plan():
    from paper_2607_21291_gb300 import build as B
    B.build()
    g = np.random.default_rng(0)
    L, T, t, d = 6, 512, 0.5, 32
    rows = [g.normal(size=(40, d)) for _ in range(L)]
    outs = [r + g.normal(scale=0.2 + 0.3 * l, size=r.shape) for l, r in enumerate(rows)]
    shards = [[(rows[l][:13], outs[l][:13]) for l in range(L)],
              [(rows[l][13:], outs[l][13:]) for l in range(L)]]
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, shards, T, t, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    s_ref = np.array([O.similarity(O.cos_sim_stat(rows[l], outs[l])) for l in range(L)])
    r_ref, _ = O.allocate_ratios(s_ref, t)
    K_ref = O.kept_counts(r_ref, T)
    for _, s, r, K in res:
        assert np.allclose(s, s_ref, rtol=1e-12)
        assert np.allclose(r, r_ref, rtol=1e-10)
        assert K == K_ref.tolist()
    assert res[0][3] == res[1][3]


def test_single_process_is_identity():
    from paper_2607_21291_gb300 import calibrate as C
    acc = torch.tensor([3.0, 4.0, 1.5, 2.0], dtype=torch.float64)
    assert C.allreduce_stats(acc) is acc
    assert C.similarity_of(acc).tolist() == [0.75, 0.75]
