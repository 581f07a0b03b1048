"""GPU parity of generation with a kept-token cache (adadsf_prefill, then
adadsf_decode_step) against the oracle's sparse_prefill / decode_step,
through the C ABI.

The GPU's prompt kept sets are given to the oracle (kept-set rules as for the
sparse forward), and so are its per-step keep decisions; each decision must
equal the oracle's own wherever the oracle's score is more than 1e-3 away
from its threshold. Hidden states within the parity tolerance; cached counts
follow the decisions; the cache's thresholds match the oracle's."""
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


QWEN_SMALL = S.QWEN25_1_5B.replace(d=1024, n_heads=8, n_kv_heads=2, ffn=1536, n_layers=3, vocab=500)
NEOX_SMALL = S.PYTHIA_160M.replace(n_layers=3, vocab=500)
NEOX_F32 = S.PYTHIA_70M.replace(n_layers=2, vocab=500)
# the Qwen2.5-7B attention geometry (28 query heads on 4 key/value heads,
# head_dim 128) with a narrow MLP: caches of several hundred keys spread over
# several splits, some of them empty
QWEN7_ATTN = S.QWEN25_7B.replace(ffn=2048, n_layers=2, vocab=500)
# 16 query heads on one key/value head, head_dim 64: every row of the tensor
# core tile is a real head
QWEN_G16 = QWEN_SMALL.replace(n_heads=16, n_kv_heads=1, head_dim=64, rotary_dim=64, n_layers=2)

CASES = [
    # (shape, B, T0, K per layer, steps, C_max, gated, element-wise tolerance)
    (NEOX_SMALL, 3, 64, [64, 20, 40], 5, 80, False, None),
    (QWEN_SMALL, 2, 100, [50, 100, 0], 4, 128, False, None),
    (QWEN_SMALL, 2, 96, [48, 30, 96], 3, 100, True, None),
    (NEOX_F32, 2, 40, [20, 40], 4, 48, False, None),
    (QWEN7_ATTN, 2, 700, [350, 700], 3, 720, False, H.BF16_DEEP_ELEM_TOL),
    (QWEN_G16, 3, 200, [131, 64], 3, 216, True, None),
]


def _cache_counts(A, cache, L, B):
    """Per-layer kept counts and thresholds from the cache header area
    ([L][B] int32 at byte 256, then [L][B] fp32 256-aligned)."""
    lens = cache[256:256 + 4 * L * B].view(torch.int32).view(L, B).cpu().numpy()
    off = 256 + ((4 * L * B + 255) // 256) * 256
    thr = cache[off:off + 4 * L * B].view(torch.float32).view(L, B).cpu().numpy()
    return lens, thr


@pytest.mark.parametrize("shape,B,T0,K,steps,C_max,gated,etol", CASES)
def test_prefill_then_decode(A, shape, B, T0, K, steps, C_max, gated, etol):
    _prefill_then_decode(A, shape, B, T0, K, steps, C_max, gated, etol)


@pytest.mark.parametrize("gated", [False, True])
def test_prefill_then_decode_folded_norms(A, gated):
    """The same check on weights with the norm gains folded in
    (adadsf_fold_norms, FLAG_FOLDED_NORMS): the decode step's post-attention
    RMSNorm then runs inside the output and gate / up projections."""
    _prefill_then_decode(A, QWEN_SMALL, 2, 96, [48, 30, 96], 3, 100, gated, None, folded=True)


def _prefill_then_decode(A, shape, B, T0, K, steps, C_max, gated, etol, folded=False):
    L = shape.n_layers
    td = H.tdtype(shape)
    flags = (A.FLAG_GATE_SIGMOID if gated else 0) | (A.FLAG_FOLDED_NORMS if folded else 0)
    hostL = [H.host_layer(shape, 13, l) for l in range(L)]
    extra = H.host_extra(shape, 13)
    layers = [A.to_device(w, td) for w in hostL]
    if folded:
        for w in layers:
            A.adadsf_fold_norms(A.make_cfg(shape.replace(n_layers=1)), w)
    model = A.DeviceModel(A.make_cfg(shape, flags), layers, A.to_device(extra, td))
    ids = S.token_ids(14, B, T0 + steps, shape.vocab)
    ids_d = torch.from_numpy(ids).cuda()
    cache = A.kv_cache(model.cfg, B, C_max)
    hidden = torch.empty((B, T0, shape.d), dtype=td, device="cuda")
    idx = torch.full((B * sum(K),), -1, dtype=torch.int32, device="cuda")
    ws = A.workspace(A.adadsf_model_workspace_size(model.cfg, B, T0, K, False))
    A.adadsf_prefill(model, ids_d[:, :T0].contiguous(), K, hidden, cache, C_max, idx_out=idx, ws=ws)
    assert A.adadsf_sync_check(ws) == A.OK
    gi, off, kept_sets = idx.cpu().numpy(), 0, []
    for k in K:
        kept_sets.append(gi[off:off + B * k].reshape(B, k))
        off += B * k
    p = dict(O.params_of(shape), gate="sigmoid") if gated else O.params_of(shape)
    W64 = [H.f64(w) for w in hostL]
    E64 = H.f64(extra)
    ref, st = O.sparse_prefill(ids[:, :T0], E64, W64, p, K, idx_force=kept_sets)
    H.assert_close(H.to_np(hidden), ref, H.tol(shape), "prefill", etol)
    lens, thr = _cache_counts(A, cache, L, B)
    assert lens.tolist() == [[k] * B for k in K]
    thr_ref = np.array(st["thr"])
    finite = np.isfinite(thr_ref)
    assert (np.isinf(thr) == ~finite).all() and (thr[~finite] > 0).all()   # K = 0: +inf
    sc_tol = 5e-3 if shape.dtype == "bf16" else 1e-5
    assert np.abs(thr[finite] - thr_ref[finite]).max(initial=0) <= sc_tol * max(1.0, np.abs(thr_ref[finite]).max(initial=0))

    dws = A.workspace(A.adadsf_decode_workspace_size(model.cfg, B, C_max))
    counts = np.array(lens, dtype=np.int64)
    n_checked = 0
    for step in range(steps):
        h = torch.empty((B, shape.d), dtype=td, device="cuda")
        kept = torch.full((L, B), -1, dtype=torch.int32, device="cuda")
        A.adadsf_decode_step(model, ids_d[:, T0 + step].contiguous(), h, cache, C_max, kept_out=kept, ws=dws)
        assert A.adadsf_sync_check(dws) == A.OK
        kg = kept.cpu().numpy().astype(bool)
        href, kown, sref = O.decode_step(ids[:, T0 + step], E64, W64, p, st, kept_force=kg)
        margin = np.abs(sref - thr_ref) > 1e-3 * np.maximum(1.0, np.abs(thr_ref))
        assert (kg[margin] == kown[margin]).all(), (step, kg, kown)
        n_checked += int(margin.sum())
        H.assert_close(H.to_np(h), href, H.tol(shape), f"decode step {step}", etol)
        counts += kg
        lens, _ = _cache_counts(A, cache, L, B)
        assert (lens == counts).all()
    assert n_checked > 0
    # a layer that kept no prompt token keeps no generated token
    for l, k in enumerate(K):
        if k == 0:
            assert (counts[l] == 0).all()


def test_decode_step_in_a_cuda_graph(A):
    """A decode step reads its position and counts from the cache, so one
    captured graph replays step after step: the same outputs as eager steps."""
    shape = NEOX_SMALL
    B, T0, C_max, K = 2, 48, 64, [24, 48, 12]
    td = H.tdtype(shape)
    hostL = [H.host_layer(shape, 21, l) for l in range(shape.n_layers)]
    model = A.DeviceModel(A.make_cfg(shape), [A.to_device(w, td) for w in hostL],
                          A.to_device(H.host_extra(shape, 21), td))
    ids = torch.from_numpy(S.token_ids(22, B, T0 + 4, shape.vocab)).cuda()
    outs = []
    for use_graph in (False, True):
        cache = A.kv_cache(model.cfg, B, C_max)
        A.adadsf_prefill(model, ids[:, :T0].contiguous(), K,
                         torch.empty((B, T0, shape.d), dtype=td, device="cuda"), cache, C_max)
        dws = A.workspace(A.adadsf_decode_workspace_size(model.cfg, B, C_max))
        tok = torch.empty(B, dtype=torch.int32, device="cuda")
        h = torch.empty((B, shape.d), dtype=td, device="cuda")
        stream = torch.cuda.Stream()
        res = []
        with torch.cuda.stream(stream):
            if use_graph:
                tok.copy_(ids[:, T0])
                A.adadsf_decode_step(model, tok, h, cache, C_max, ws=dws, stream=stream)   # warm-up step
                res.append(h.clone())
                g = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g, stream=stream):
                    A.adadsf_decode_step(model, tok, h, cache, C_max, ws=dws, stream=stream)
                for t in range(1, 4):
                    tok.copy_(ids[:, T0 + t])
                    g.replay()
                    res.append(h.clone())
            else:
                for t in range(4):
                    tok.copy_(ids[:, T0 + t])
                    A.adadsf_decode_step(model, tok, h, cache, C_max, ws=dws, stream=stream)
                    res.append(h.clone())
        torch.cuda.synchronize()
        assert A.adadsf_sync_check(dws) == A.OK
        outs.append(torch.stack(res))
    assert torch.equal(outs[0], outs[1])


def test_decode_at_bench_geometry(A):
    """A decode step at the geometry the throughput measurement replays
    (16 sequences, a 4096-token prompt, the Qwen2.5-7B attention shape, half
    the prompt kept, the same cache length and split count), one layer with a
    narrow MLP. Sequences are independent, so the oracle runs on a sample of
    two of them, with the GPU's kept sets and decisions."""
    shape = QWEN7_ATTN.replace(n_layers=1)
    B, T0, steps = 16, 4096, 2
    C_max, K = T0 + 32 + 8, [2048]
    td = H.tdtype(shape)
    hostL = [H.host_layer(shape, 31, 0)]
    extra = H.host_extra(shape, 31)
    model = A.DeviceModel(A.make_cfg(shape), [A.to_device(w, td) for w in hostL], A.to_device(extra, td))
    ids = S.token_ids(32, B, T0 + steps, shape.vocab)
    ids_d = torch.from_numpy(ids).cuda()
    cache = A.kv_cache(model.cfg, B, C_max)
    idx = torch.full((B * K[0],), -1, dtype=torch.int32, device="cuda")
    ws = A.workspace(A.adadsf_model_workspace_size(model.cfg, B, T0, K, False))
    A.adadsf_prefill(model, ids_d[:, :T0].contiguous(), K, torch.empty((B, T0, shape.d), dtype=td, device="cuda"),
                     cache, C_max, idx_out=idx, ws=ws)
    assert A.adadsf_sync_check(ws) == A.OK
    del ws
    sample = [0, B - 1]
    kept_set = idx.cpu().numpy().reshape(B, K[0])[sample]
    W64, E64 = [H.f64(hostL[0])], H.f64(extra)
    p = O.params_of(shape)
    _, st = O.sparse_prefill(ids[sample, :T0], E64, W64, p, K, idx_force=[kept_set])
    dws = A.workspace(A.adadsf_decode_workspace_size(model.cfg, B, C_max))
    for step in range(steps):
        h = torch.empty((B, shape.d), dtype=td, device="cuda")
        kept = torch.full((1, B), -1, dtype=torch.int32, device="cuda")
        A.adadsf_decode_step(model, ids_d[:, T0 + step].contiguous(), h, cache, C_max, kept_out=kept, ws=dws)
        assert A.adadsf_sync_check(dws) == A.OK
        kg = kept.cpu().numpy().astype(bool)[:, sample]
        href, _, _ = O.decode_step(ids[sample, T0 + step], E64, W64, p, st, kept_force=kg)
        H.assert_close(H.to_np(h)[sample], href, H.tol(shape), f"decode step {step}", H.BF16_DEEP_ELEM_TOL)


def _small_model(A, shape, seed):
    td = H.tdtype(shape)
    hostL = [H.host_layer(shape, seed, l) for l in range(shape.n_layers)]
    return A.DeviceModel(A.make_cfg(shape), [A.to_device(w, td) for w in hostL],
                         A.to_device(H.host_extra(shape, seed), td)), td


def _decode_run(A, model, td, ids, B, T0, K, C_max, steps, stream, capture_first=False):
    """Prefill then `steps` decode steps on `stream`; with capture_first the
    steps are replayed from a graph captured before any eager step on this
    stream (the step then runs on the caller's stream alone)."""
    d = model.cfg.d
    cache = A.kv_cache(model.cfg, B, C_max)
    dws = A.workspace(A.adadsf_decode_workspace_size(model.cfg, B, C_max))
    tok = torch.empty(B, dtype=torch.int32, device="cuda")
    h = torch.empty((B, d), dtype=td, device="cuda")
    out = []
    with torch.cuda.stream(stream):
        A.adadsf_prefill(model, ids[:, :T0].contiguous(), K, torch.empty((B, T0, d), dtype=td, device="cuda"),
                         cache, C_max, stream=stream)
        if capture_first:
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                A.adadsf_decode_step(model, tok, h, cache, C_max, ws=dws, stream=stream)
            for t in range(steps):
                tok.copy_(ids[:, T0 + t])
                g.replay()
                out.append(h.clone())
        else:
            for t in range(steps):
                tok.copy_(ids[:, T0 + t])
                A.adadsf_decode_step(model, tok, h, cache, C_max, ws=dws, stream=stream)
                out.append(h.clone())
    torch.cuda.synchronize()
    assert A.adadsf_sync_check(dws) == A.OK
    return torch.stack(out)


def test_decode_captured_before_any_eager_step(A):
    """A step captured into a graph before any uncaptured step on its stream
    runs on that stream alone (keep decision inside the norm launch); its
    outputs equal those of eager steps, which fork the router onto a second
    stream."""
    shape = QWEN_SMALL
    model, td = _small_model(A, shape, 61)
    B, T0, C_max, K = 2, 96, 112, [48, 30, 96]
    ids = torch.from_numpy(S.token_ids(62, B, T0 + 4, shape.vocab)).cuda()
    eager = _decode_run(A, model, td, ids, B, T0, K, C_max, 4, torch.cuda.Stream())
    graph = _decode_run(A, model, td, ids, B, T0, K, C_max, 4, torch.cuda.Stream(), capture_first=True)
    assert torch.equal(eager, graph)


def test_decode_on_two_streams_interleaved(A):
    """Two models decode on two streams with their steps enqueued in turn:
    each gets the outputs it gets alone (each caller stream has its own
    second stream and fork / join events)."""
    shape = NEOX_SMALL
    (m1, td), (m2, _) = _small_model(A, shape, 71), _small_model(A, shape, 72)
    B, T0, C_max, K, steps = 2, 64, 80, [40, 64, 20], 4
    ids1 = torch.from_numpy(S.token_ids(73, B, T0 + steps, shape.vocab)).cuda()
    ids2 = torch.from_numpy(S.token_ids(74, B, T0 + steps, shape.vocab)).cuda()
    alone1 = _decode_run(A, m1, td, ids1, B, T0, K, C_max, steps, torch.cuda.Stream())
    alone2 = _decode_run(A, m2, td, ids2, B, T0, K, C_max, steps, torch.cuda.Stream())
    s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()
    caches, wss, toks, hs, outs = [], [], [], [], [[], []]
    for m, ids, s in ((m1, ids1, s1), (m2, ids2, s2)):
        cache = A.kv_cache(m.cfg, B, C_max)
        with torch.cuda.stream(s):
            A.adadsf_prefill(m, ids[:, :T0].contiguous(), K, torch.empty((B, T0, shape.d), dtype=td, device="cuda"),
                             cache, C_max, stream=s)
        caches.append(cache)
        wss.append(A.workspace(A.adadsf_decode_workspace_size(m.cfg, B, C_max)))
        toks.append(torch.empty(B, dtype=torch.int32, device="cuda"))
        hs.append(torch.empty((B, shape.d), dtype=td, device="cuda"))
    torch.cuda.synchronize()
    for t in range(steps):
        for i, (m, ids, s) in enumerate(((m1, ids1, s1), (m2, ids2, s2))):
            with torch.cuda.stream(s):
                toks[i].copy_(ids[:, T0 + t])
                A.adadsf_decode_step(m, toks[i], hs[i], caches[i], C_max, ws=wss[i], stream=s)
                outs[i].append(hs[i].clone())
    torch.cuda.synchronize()
    assert A.adadsf_sync_check(wss[0]) == A.OK and A.adadsf_sync_check(wss[1]) == A.OK
    assert torch.equal(torch.stack(outs[0]), alone1)
    assert torch.equal(torch.stack(outs[1]), alone2)
