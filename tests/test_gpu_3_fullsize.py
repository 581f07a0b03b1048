"""Full-size parity in the benchmark's launch configuration: one layer of each
bf16 workload shape at its full (B, T), with the first, a middle and the last
layer's weights, and kept counts from the retention sweep (r = 0.25 / 0.5 /
0.75, and r = 1 from the t = 1 allocation, which clamps every layer to dense).
Each layer gets the same input on both sides (teacher forcing: the GPU's
earlier layers do not feed it). The oracle checks sampled sequences (sequences
are independent, so one sequence is a complete check of itself); properties
that hold at any size are checked on the whole batch: skipped rows
bit-identical and kept sets identical to the oracle's Top-K of the GPU scores."""
import functools

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


@functools.lru_cache(maxsize=2)
def _weights(key, layer):
    return H.host_layer(S.WORKLOADS[key].shape, 11, layer, gain_std=0.1)


def _mid(key):
    return S.WORKLOADS[key].shape.n_layers // 2


def _last(key):
    return S.WORKLOADS[key].shape.n_layers - 1


CASES = [("c2", 0, 0.5), ("c2", _mid("c2"), 0.5), ("c2", _last("c2"), 0.5),
         ("c3", 0, 0.5), ("c3", _mid("c3"), 0.5), ("c3", _mid("c3"), 0.25), ("c3", _mid("c3"), 0.75),
         ("c3", _last("c3"), 0.5),
         ("c4", 0, 0.5), ("c4", _mid("c4"), 0.5), ("c4", _last("c4"), 0.5),
         ("c5", 0, 0.5), ("c5", _mid("c5"), 0.5), ("c5", _mid("c5"), 0.75), ("c5", _last("c5"), 0.5),
         ("c5", _last("c5"), 0.25), ("c5", _last("c5"), 1.0)]


@pytest.mark.parametrize("key,layer,r", CASES)
def test_fullsize_layer(A, key, layer, r):
    wl = S.WORKLOADS[key]
    shape, B, T = wl.shape, wl.B, wl.T
    if r == 1.0:
        # t = 1: Eq. 8 gives some r_l > 1 on an uneven similarity vector; the
        # clamp makes every layer dense
        s = np.linspace(0.80, 0.99, shape.n_layers)
        r_raw, _ = A.adadsf_alloc_ratios(s, 1.0, 0.05, 10.0, T, A.ALLOC_RAW)
        assert r_raw.max() > 1.0
        _, Ks = A.adadsf_alloc_ratios(s, 1.0, 0.05, 10.0, T)
        assert Ks.tolist() == [T] * shape.n_layers
        K = int(Ks[layer])
    else:
        K = int(np.floor(r * T))
    td = H.tdtype(shape)
    W = _weights(key, layer)
    x = S.round_to(S.hidden(11 + layer, B, T, shape.d), shape.dtype)
    xd = H.to_dev(x, td)
    x0 = xd.clone()
    idx = torch.empty((B, K), dtype=torch.int32, device="cuda")
    sc = torch.full((B, T), float("nan"), dtype=torch.float32, device="cuda")
    cfg = A.make_cfg(shape)
    ws = A.workspace(A.adadsf_layer_workspace_size(cfg, B, T, K))
    A.adadsf_sparse_layer_forward(cfg, A.to_device(W, td), xd, K, idx, sc, ws)
    assert A.adadsf_sync_check(ws) == A.OK
    gi = idx.cpu().numpy()
    gs = sc.cpu().numpy()
    if K < T:
        # whole batch: kept sets are the Top-K of the GPU scores; skipped rows untouched
        keep = torch.zeros((B, T), dtype=torch.bool, device="cuda")
        keep.scatter_(1, idx.long(), True)
        assert torch.equal(xd[~keep], x0[~keep])
        for b in range(B):
            assert O.topk_keep(gs[b], K).tolist() == gi[b].tolist()
    else:
        assert (gi == np.arange(T)[None, :]).all()
    # two sampled sequences (the first and the last) against the oracle
    W64 = H.f64(W)
    p = O.params_of(shape)
    got = xd.float().cpu().numpy()
    for b in (0, B - 1):
        xb = x[b:b + 1].astype(np.float64)
        if K < T:
            H.check_kept_sets(gs[b:b + 1], gi[b:b + 1], O.router_scores(xb, W64), K)
        ref, _, _ = O.sparse_layer_forward(xb, W64, p, K, idx=gi[b:b + 1])
        H.assert_close(got[b:b + 1], ref, H.BF16_TOL, f"{key} layer {layer} K {K} seq {b}")


FOLDED_CASES = [("c4", _mid("c4"), 0.5), ("c5", 0, 0.5), ("c5", _mid("c5"), 0.75), ("c5", _last("c5"), 0.25)]


@pytest.mark.parametrize("key,layer,r", FOLDED_CASES)
def test_fullsize_layer_gathered_qkv(A, key, layer, r):
    """Qwen shapes with folded norm gains and FLAG_GATHERED_QKV at full size:
    the first RMSNorm runs inside the QKV projection (the router's per-token sums of squares, the
    kept rows gathered from x by the projection's loads), so no gather + norm
    launch remains; sampled sequences against the oracle on the unfolded
    weights, skipped rows bit-identical. Token rows carry a spread of scales,
    so that a row norm dropped or taken from another row shows."""
    wl = S.WORKLOADS[key]
    shape, B, T = wl.shape, wl.B, wl.T
    K = int(np.floor(r * T))
    td = H.tdtype(shape)
    W = _weights(key, layer)
    x = S.round_to(H.row_spread(S.hidden(11 + layer, B, T, shape.d), 11 + layer), shape.dtype)
    xd = H.to_dev(x, td)
    x0 = xd.clone()
    wd = A.to_device(W, td)
    A.adadsf_fold_norms(A.make_cfg(shape.replace(n_layers=1)), wd)
    idx = torch.empty((B, K), dtype=torch.int32, device="cuda")
    sc = torch.empty((B, T), dtype=torch.float32, device="cuda")
    cfg = A.make_cfg(shape, A.FLAG_FOLDED_NORMS | A.FLAG_GATHERED_QKV)
    ws = A.workspace(A.adadsf_layer_workspace_size(cfg, B, T, K))
    A.adadsf_profile_begin(256)
    A.adadsf_sparse_layer_forward(cfg, wd, xd, K, idx, sc, ws)
    kinds = {rec[0] for rec in A.adadsf_profile_end(256)}
    assert A.adadsf_sync_check(ws) == A.OK
    assert not kinds & {"gather_norm", "topk_gather_norm"}, kinds
    keep = torch.zeros((B, T), dtype=torch.bool, device="cuda")
    keep.scatter_(1, idx.long(), True)
    assert torch.equal(xd[~keep], x0[~keep])
    gi = idx.cpu().numpy()
    gs = sc.cpu().numpy()
    W64 = H.f64(W)
    p = O.params_of(shape)
    got = xd.float().cpu().numpy()
    for b in (0, B - 1):
        xb = x[b:b + 1].astype(np.float64)
        H.check_kept_sets(gs[b:b + 1], gi[b:b + 1], O.router_scores(xb, W64), K)
        ref, _, _ = O.sparse_layer_forward(xb, W64, p, K, idx=gi[b:b + 1])
        H.assert_close(got[b:b + 1], ref, H.BF16_TOL, f"{key} folded layer {layer} K {K} seq {b}")
