"""Full-size parity in the benchmark's launch configuration: one layer of each
bf16 workload shape at its full (B, T) with r = 0.5, checked against the fp64
oracle on sampled sequences (sequences are independent, so one sequence is a
complete check of itself), plus whole-batch properties that hold at any size:
skipped rows bit-identical and kept sets identical to the oracle's Top-K of
the GPU scores."""
import numpy as np
import pytest
import torch

from oracle import adadsf_oracle as O
from paper_2607_21291_gb300 import synth as S
from tests import helpers as H

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def A():
    from paper_2607_21291_gb300 import adadsf
    adadsf.lib()
    return adadsf


@pytest.mark.parametrize("key,samples", [("c2", (0, 3)), ("c3", (0, 7)), ("c4", (0, 7)), ("c5", (15,))])
def test_fullsize_layer(A, key, samples):
    wl = S.WORKLOADS[key]
    shape, B, T = wl.shape, wl.B, wl.T
    K = T // 2
    td = H.tdtype(shape)
    W = H.host_layer(shape, 11, 0, gain_std=0.1)
    x = S.round_to(S.hidden(11, B, T, shape.d), shape.dtype)
    xd = H.to_dev(x, td)
    x0 = xd.clone()
    idx = torch.empty((B, K), dtype=torch.int32, device="cuda")
    sc = torch.empty((B, T), dtype=torch.float32, device="cuda")
    cfg = A.make_cfg(shape)
    ws = A.workspace(A.adadsf_layer_workspace_size(cfg, B, T, K))
    A.adadsf_sparse_layer_forward(cfg, A.to_device(W, td), xd, K, idx, sc, ws)
    assert A.adadsf_sync_check(ws) == A.OK
    gi = idx.cpu().numpy()
    gs = sc.cpu().numpy()
    # whole batch: kept sets are the Top-K of the GPU scores; skipped rows untouched
    keep = torch.zeros((B, T), dtype=torch.bool, device="cuda")
    keep.scatter_(1, idx.long(), True)
    assert torch.equal(xd[~keep], x0[~keep])
    for b in range(B):
        assert O.topk_keep(gs[b], K).tolist() == gi[b].tolist()
    # sampled sequences against the oracle
    W64 = H.f64(W)
    p = O.params_of(shape)
    got = xd.float().cpu().numpy()
    for b in samples:
        xb = x[b:b + 1].astype(np.float64)
        ref_sc = O.router_scores(xb, W64)
        H.check_kept_sets(gs[b:b + 1], gi[b:b + 1], ref_sc, K)
        ref, _, _ = O.sparse_layer_forward(xb, W64, p, K, idx=gi[b:b + 1])
        assert H.max_rel(got[b:b + 1], ref) <= H.BF16_TOL
