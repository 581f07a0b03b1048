"""GPU parity of the individual steps against the fp64 oracle, through the C ABI.
Sizes span several tiles with ragged tails; edge cases include K = 0, 1, T-1, T,
ties, NaN and signed zeros."""
import numpy as np
import pytest
import torch

from oracle import adadsf_oracle as O
from paper_2607_21291_gb300 import synth as S
from tests import helpers as H

pytestmark = pytest.mark.gpu
SYNC_BYTES = 16384   # arrival counters right after the device error word


@pytest.fixture(scope="module")
def A():
    from paper_2607_21291_gb300 import adadsf
    adadsf.lib()
    torch.cuda.init()
    return adadsf


# ---------------------------------------------------------------- failure channel
def test_bounded_wait_gives_up_cleanly(A):
    ws = A.workspace(256)
    A.adadsf_selftest_bounded_wait(ws, 2000)
    assert A.adadsf_sync_check(ws) == A.ERR_DEVICE_TIMEOUT
    assert A.adadsf_sync_check(ws) == A.OK              # cleared by the read
    x = torch.ones(16, device="cuda")
    assert float((x * 2).sum()) == 32.0                 # context still usable



def test_timeout_clears_sync_area(A):
    """A kernel that gives up waiting may leave cross-CTA arrival counters
    part-way. After a timeout, adadsf_sync_check zeroes the synchronisation
    area, so the same workspace then gives correct router scores on a shape
    whose tiles are split along d (counters in use)."""
    shape = S.QWEN25_7B.replace(ffn=256)
    n = 25600 - 77                                          # 200 tiles: split past one wave
    cfg = A.make_cfg(shape)
    ws = A.workspace(A.adadsf_router_select_workspace_size(cfg, 1, 1))
    ws[256:256 + SYNC_BYTES].view(torch.int32)[::7] = 3     # counters left part-way
    A.adadsf_selftest_bounded_wait(ws, 2000)
    assert A.adadsf_sync_check(ws) == A.ERR_DEVICE_TIMEOUT
    assert int(ws[256:256 + SYNC_BYTES].view(torch.int32).abs().sum()) == 0
    W = H.host_layer(shape, 3)
    x = S.round_to(np.random.default_rng(n + 1).standard_normal((n, shape.d)).astype(np.float32), shape.dtype)
    sc = torch.empty(n, dtype=torch.float32, device="cuda")
    A.adadsf_router_scores(cfg, A.to_device(W, H.tdtype(shape)), H.to_dev(x, H.tdtype(shape)), sc, ws=ws)
    assert A.adadsf_sync_check(ws) == A.OK
    ref = O.router_scores(x.astype(np.float64), H.f64(W))
    assert np.max(np.abs(sc.cpu().numpy() - ref)) / np.max(np.abs(ref)) < 5e-3

# ---------------------------------------------------------------- Top-K (Sec. 3.4)
@pytest.mark.parametrize("B,T,K", [(1, 1, 1), (3, 7, 3), (2, 128, 64), (4, 512, 256), (2, 1000, 1),
                                   (2, 1000, 999), (2, 1000, 1000), (5, 2048, 1024), (16, 4096, 2048),
                                   (1, 16384, 5000)])
def test_topk_random(A, B, T, K):
    g = np.random.default_rng(B * 100003 + T * 7 + K)
    s = g.standard_normal((B, T)).astype(np.float32)
    s[:, ::5] = np.round(s[:, ::5], 1)                 # plenty of exact ties
    sd = torch.from_numpy(s).cuda()
    idx = torch.full((B, K), -1, dtype=torch.int32, device="cuda")
    rows = torch.full((B, K), -1, dtype=torch.int32, device="cuda")
    A.adadsf_topk_select(sd, K, idx, rows)
    gi, gr = idx.cpu().numpy(), rows.cpu().numpy()
    for b in range(B):
        ref = O.topk_keep(s[b], K)
        assert gi[b].tolist() == ref.tolist()
        assert gr[b].tolist() == (b * T + ref).tolist()


def test_topk_special_values(A):
    s = np.array([[1.0, 3.0, 3.0, 2.0, 3.0, -0.0, 0.0, np.nan, -np.inf, np.inf, np.nan, -1.0]],
                 dtype=np.float32)
    sd = torch.from_numpy(s).cuda()
    for K in range(0, 13):
        idx = torch.full((1, max(K, 1)), -1, dtype=torch.int32, device="cuda")
        A.adadsf_topk_select(sd, K, idx)
        if K:
            assert idx[0].cpu().tolist() == O.topk_keep(s[0], K).tolist(), K
    allnan = torch.full((2, 33), float("nan"), device="cuda")
    idx = torch.empty((2, 5), dtype=torch.int32, device="cuda")
    A.adadsf_topk_select(allnan, 5, idx)
    assert idx.cpu().tolist() == [[0, 1, 2, 3, 4]] * 2


# ---------------------------------------------------------------- projections (Eq. 2)
@pytest.mark.parametrize("M,N,Kd", [(1, 64, 64), (127, 128, 64), (129, 256, 128), (300, 384, 192),
                                    (1024, 2304, 768), (2050, 512, 2048), (4099, 3072, 768),
                                    # CTA-pair 256x256 tiles (large M, N % 256 == 0)
                                    (8192, 2048, 512), (2600, 4608, 320), (10000, 4096, 1024)])
@pytest.mark.parametrize("act", [0, 1])
def test_linear_bf16(A, M, N, Kd, act):
    g = np.random.default_rng(M + N + Kd + act)
    x = S.round_to(g.standard_normal((M, Kd)).astype(np.float32), "bf16")
    w = S.round_to((0.05 * g.standard_normal((N, Kd))).astype(np.float32), "bf16")
    b = S.round_to((0.1 * g.standard_normal(N)).astype(np.float32), "bf16")
    out = torch.empty((M, N), dtype=torch.bfloat16, device="cuda")
    A.adadsf_linear(H.to_dev(x, torch.bfloat16), H.to_dev(w, torch.bfloat16),
                    H.to_dev(b, torch.bfloat16), out, act=act)
    ref = O.linear(x, w, b, "gelu" if act else None)
    assert H.max_rel(H.to_np(out), ref) < 8e-3


@pytest.mark.parametrize("M,N,Kd,act", [(1, 64, 3072, 0), (300, 768, 3072, 1), (1384, 768, 3072, 0),
                                        (128, 256, 2048, 0), (777, 2304, 768, 1), (1000, 384, 1024, 0),
                                        (1024, 768, 768, 1), (1024, 768, 3072, 0), (333, 640, 960, 1),
                                        (129, 128, 192, 0),
                                        # fewer than 128 rows: a stage loads only them, rounded up to 8
                                        (5, 512, 3584, 0), (13, 4608, 3584, 1), (16, 3584, 18944, 0),
                                        (17, 1024, 2048, 1), (100, 640, 1536, 0)])
def test_linear_bf16_small_m(A, M, N, Kd, act):
    """Small-M projections of the sparse layers: one wave of tiles, long K
    (with room for scratch most of these run split along K over clusters of 2
    or 4 CTAs, with ragged M, N and K tails and uneven K ranges per CTA; with
    the minimum workspace they do not); two launches in a row agree bit for
    bit (the partial tiles are summed in a fixed order)."""
    g = np.random.default_rng(M * 7 + N + Kd)
    x = S.round_to(g.standard_normal((M, Kd)).astype(np.float32), "bf16")
    w = S.round_to((0.05 * g.standard_normal((N, Kd))).astype(np.float32), "bf16")
    b = S.round_to((0.1 * g.standard_normal(N)).astype(np.float32), "bf16")
    ref = O.linear(x, w, b, "gelu" if act else None)
    for ws_bytes in (A.LINEAR_SPLIT_WS_BYTES, 256):
        ws = A.workspace(ws_bytes)
        outs = []
        for _ in range(2):
            out = torch.empty((M, N), dtype=torch.bfloat16, device="cuda")
            A.adadsf_linear(H.to_dev(x, torch.bfloat16), H.to_dev(w, torch.bfloat16),
                            H.to_dev(b, torch.bfloat16), out, act=act, ws=ws)
            assert A.adadsf_sync_check(ws) == A.OK
            assert H.max_rel(H.to_np(out), ref) < 8e-3
            outs.append(out)
        assert torch.equal(outs[0], outs[1])


@pytest.mark.parametrize("M,N,Kd", [(1, 4, 4), (65, 132, 68), (200, 2048, 512)])
def test_linear_f32(A, M, N, Kd):
    g = np.random.default_rng(M * N)
    x = g.standard_normal((M, Kd)).astype(np.float32)
    w = (0.05 * g.standard_normal((N, Kd))).astype(np.float32)
    out = torch.empty((M, N), dtype=torch.float32, device="cuda")
    A.adadsf_linear(H.to_dev(x, torch.float32), H.to_dev(w, torch.float32), None, out, act=1)
    assert H.max_rel(H.to_np(out), O.linear(x, w, None, "gelu")) < 1e-5


# ---------------------------------------------------------------- router (Sec. 3.4)
@pytest.mark.parametrize("shape,n", [(S.PYTHIA_160M, 1), (S.PYTHIA_160M, 2048), (S.QWEN25_1_5B, 333),
                                     (S.PYTHIA_70M, 128), (S.PYTHIA_160M, 777), (S.PYTHIA_1_4B, 16384)])
def test_router(A, shape, n):
    W = H.host_layer(shape, 3)
    x = S.round_to(np.random.default_rng(n).standard_normal((n, shape.d)).astype(np.float32), shape.dtype)
    w = A.to_device(W, H.tdtype(shape))
    sc = torch.empty(n, dtype=torch.float32, device="cuda")
    A.adadsf_router_scores(A.make_cfg(shape), w, H.to_dev(x, H.tdtype(shape)), sc)
    ref = O.router_scores(x.astype(np.float64), H.f64(W))
    err = np.max(np.abs(sc.cpu().numpy() - ref)) / np.max(np.abs(ref))
    assert err < (5e-3 if shape.dtype == "bf16" else 1e-5)


@pytest.mark.parametrize("shape,n", [(S.PYTHIA_160M, 2048), (S.PYTHIA_1_4B, 16384), (S.QWEN25_1_5B, 999),
                                     (S.QWEN25_7B.replace(ffn=256), 4096),
                                     (S.QWEN25_7B.replace(ffn=256), 25600 - 77)])
def test_router_split(A, shape, n):
    """Router with room for scratch. Up to one wave of 128-token tiles every
    CTA takes whole tiles; past it (the last case: 200 tiles of d = 3584 on
    the GPU's ~150 SMs) the CTAs take equal ranges of k-blocks, tiles are
    split along d and the last CTA of a tile sums the partials in a fixed
    order. Either way two calls agree bit for bit and the counters end at
    zero."""
    W = H.host_layer(shape, 3)
    x = S.round_to(np.random.default_rng(n + 1).standard_normal((n, shape.d)).astype(np.float32), shape.dtype)
    w = A.to_device(W, H.tdtype(shape))
    cfg = A.make_cfg(shape)
    ws = A.workspace(A.adadsf_router_select_workspace_size(cfg, 1, 1))
    ref = O.router_scores(x.astype(np.float64), H.f64(W))
    outs = []
    for _ in range(2):
        sc = torch.empty(n, dtype=torch.float32, device="cuda")
        A.adadsf_router_scores(cfg, w, H.to_dev(x, H.tdtype(shape)), sc, ws=ws)
        assert A.adadsf_sync_check(ws) == A.OK
        err = np.max(np.abs(sc.cpu().numpy() - ref)) / np.max(np.abs(ref))
        assert err < 5e-3
        outs.append(sc)
    assert torch.equal(outs[0], outs[1])
    assert int(ws[256:256 + SYNC_BYTES].view(torch.int32).abs().sum()) == 0


@pytest.mark.parametrize("shape,B,T,K", [(S.PYTHIA_70M, 2, 128, 64),
                                         (S.PYTHIA_160M, 4, 512, 256), (S.PYTHIA_1_4B, 8, 2048, 1024),
                                         (S.QWEN25_1_5B, 3, 333, 100), (S.PYTHIA_160M, 2, 100, 1),
                                         (S.PYTHIA_160M, 5, 64, 64), (S.PYTHIA_160M, 300, 1, 1),
                                         (S.QWEN25_7B.replace(ffn=256), 2, 4096, 2000), (S.PYTHIA_160M, 1, 16384, 777)])
def test_router_select(A, shape, B, T, K):
    """Router scores and the per-sequence Top-K in one launch (Sec. 3.4):
    scores within the router tolerance of the oracle, and the kept positions
    bit-exact against the oracle's Top-K of the GPU's own scores; the
    counters in the workspace end at zero, so a second call selects the same."""
    W = H.host_layer(shape, 5)
    g = np.random.default_rng(B * 1000 + T + K)
    x = S.round_to(g.standard_normal((B * T, shape.d)).astype(np.float32), shape.dtype)
    w = A.to_device(W, H.tdtype(shape))
    cfg = A.make_cfg(shape)
    ws = A.workspace(A.adadsf_router_select_workspace_size(cfg, B, T))
    ref = O.router_scores(x.astype(np.float64), H.f64(W))
    xd = H.to_dev(x, H.tdtype(shape))
    first = None
    for rep in range(2):
        sc = torch.empty(B * T, dtype=torch.float32, device="cuda")
        idx = torch.full((B, K), -1, dtype=torch.int32, device="cuda")
        rows = torch.full((B, K), -1, dtype=torch.int32, device="cuda")
        A.adadsf_router_select(cfg, w, xd, B, T, K, sc, idx, rows, ws=ws)
        assert A.adadsf_sync_check(ws) == A.OK
        s = sc.cpu().numpy()
        assert np.max(np.abs(s - ref)) / np.max(np.abs(ref)) < 5e-3
        gi, gr = idx.cpu().numpy(), rows.cpu().numpy()
        for b in range(B):
            kept = O.topk_keep(s[b * T:(b + 1) * T], K)
            assert gi[b].tolist() == kept.tolist(), b
            assert gr[b].tolist() == (b * T + kept).tolist(), b
        if first is None:
            first = (sc, idx)
        else:
            assert torch.equal(first[0], sc) and torch.equal(first[1], idx)
    assert int(ws[256:256 + SYNC_BYTES].view(torch.int32).abs().sum()) == 0


# ---------------------------------------------------------------- attention (Eq. 1)
@pytest.mark.parametrize("hq,hkv,hd", [(12, 12, 64), (12, 2, 128), (4, 4, 128)])
@pytest.mark.parametrize("B,K", [(1, 1), (2, 63), (2, 64), (3, 130), (1, 257)])
@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_attention(A, hq, hkv, hd, B, K, dtype):
    shape = S.PYTHIA_160M.replace(n_heads=hq, n_kv_heads=hkv, head_dim=hd, d=hq * hd if hq * hd % 64 == 0 else 768,
                                  dtype=dtype)
    width = (hq + 2 * hkv) * hd
    g = np.random.default_rng(B * K + hq + hd)
    qkv = S.round_to(g.standard_normal((B * K, width)).astype(np.float32), dtype)
    out = torch.empty((B * K, hq * hd), dtype=H.tdtype(shape), device="cuda")
    A.adadsf_causal_attention(A.make_cfg(shape), H.to_dev(qkv, H.tdtype(shape)), B, K, out)
    got = H.to_np(out)
    q64 = qkv.astype(np.float64)
    for b in range(B):
        blk = q64[b * K:(b + 1) * K]
        ref = O.causal_attention(blk[:, :hq * hd], blk[:, hq * hd:(hq + hkv) * hd], blk[:, (hq + hkv) * hd:],
                                 hq, hkv, hd)
        assert H.max_rel(got[b * K:(b + 1) * K], ref) < (2e-2 if dtype == "bf16" else 1e-5)


@pytest.mark.parametrize("hq,hkv,hd,B,K", [(12, 12, 64, 7, 520), (12, 12, 64, 7, 300), (12, 2, 128, 5, 520),
                                          (4, 4, 128, 20, 300), (28, 4, 128, 2, 1100)])
def test_attention_paired_tiles(A, hq, hkv, hd, B, K):
    """Enough (query-block pair, head, sequence) work units to fill the GPU:
    the kernel runs two query tiles per CTA (with an odd number of query
    blocks the last pair has one tile), bf16 against the oracle."""
    shape = S.PYTHIA_160M.replace(n_heads=hq, n_kv_heads=hkv, head_dim=hd, d=hq * hd, dtype="bf16")
    width = (hq + 2 * hkv) * hd
    g = np.random.default_rng(B * K + hq + hd + 7)
    qkv = S.round_to(g.standard_normal((B * K, width)).astype(np.float32), "bf16")
    out = torch.empty((B * K, hq * hd), dtype=torch.bfloat16, device="cuda")
    A.adadsf_causal_attention(A.make_cfg(shape), H.to_dev(qkv, torch.bfloat16), B, K, out)
    got = H.to_np(out)
    q64 = qkv.astype(np.float64)
    for b in range(B):
        blk = q64[b * K:(b + 1) * K]
        ref = O.causal_attention(blk[:, :hq * hd], blk[:, hq * hd:(hq + hkv) * hd], blk[:, (hq + hkv) * hd:],
                                 hq, hkv, hd)
        assert H.max_rel(got[b * K:(b + 1) * K], ref) < 2e-2


# ---------------------------------------------------------------- Eq. 4 statistics
@pytest.mark.parametrize("n,d,dtype", [(1, 64, "f32"), (37, 768, "bf16"), (5000, 1536, "bf16"),
                                       (3000, 512, "f32")])
def test_layer_stats(A, n, d, dtype):
    g = np.random.default_rng(n + d)
    a = S.round_to(g.standard_normal((n, d)).astype(np.float32), dtype)
    b = S.round_to((a + 0.7 * g.standard_normal((n, d))).astype(np.float32), dtype)
    td = torch.bfloat16 if dtype == "bf16" else torch.float32
    ad, bd = H.to_dev(a, td), H.to_dev(b, td)
    acc = torch.zeros(2, dtype=torch.float64, device="cuda")
    A.adadsf_layer_stats(ad, bd, acc)
    A.adadsf_layer_stats(ad, ad, acc)                    # accumulates: + n rows of cos = 1
    ref, cnt = O.cos_sim_stat(a.astype(np.float64), b.astype(np.float64))
    got = acc.cpu().numpy()
    assert got[1] == 2 * n
    assert got[0] == pytest.approx(ref + n, rel=1e-5)
    flat = torch.zeros(3, dtype=torch.float64, device="cuda")
    A.adadsf_layer_stats(ad, bd, flat, mode=A.STATS_FLAT)
    assert flat.cpu().numpy() == pytest.approx(O.cos_sim_stat(a.astype(np.float64), b.astype(np.float64), "flat"),
                                               rel=1e-5)
    again = torch.zeros(2, dtype=torch.float64, device="cuda")
    A.adadsf_layer_stats(ad, bd, again)
    A.adadsf_layer_stats(ad, ad, again)
    assert again.cpu().numpy().tolist() == got.tolist()  # bit-reproducible
