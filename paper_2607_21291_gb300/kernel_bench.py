"""Micro-benchmark of single library entry points on seeded synthetic inputs.

  python -m paper_2607_21291_gb300.kernel_bench linear --M 8192 --N 8192 --K 2048
  python -m paper_2607_21291_gb300.kernel_bench layer --workload c3 --B 2
  python -m paper_2607_21291_gb300.kernel_bench attention --workload c5 --B 1 --K 2048
  python -m paper_2607_21291_gb300.kernel_bench decode --workload c5 --B 16 --layers 2

Each case runs `--warmup` untimed calls, then `--iters` calls each bracketed by
CUDA events on the launching stream (L2 flushed between calls by a 256 MiB
write), and prints one JSON line with the mean time and the algorithmic
TFLOP/s or GB/s. This is also the command the ncu captures run.

`--graph R` also captures R back-to-back calls in one CUDA graph and reports the
replay time divided by R ("graph_ms"): the per-call cost without host work
(tensor-map encoding, launch calls), with consecutive launches overlapped by
programmatic dependent launch as in the model forward. L2 is flushed before
each replay, not between the R calls.
"""
from __future__ import annotations

import argparse
import json

import torch

from . import adadsf as A
from . import synth as S


def _time(fn, iters, warmup, stream):
    flush = torch.empty(256 << 20, dtype=torch.uint8, device="cuda")
    for _ in range(warmup):
        fn()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(iters)]
    torch.cuda.synchronize()
    for e0, e1 in ev:
        flush.zero_()
        e0.record(stream)
        fn()
        e1.record(stream)
    torch.cuda.synchronize()
    return sum(e0.elapsed_time(e1) for e0, e1 in ev) / iters


def _time_graph(fn, reps, iters, stream):
    flush = torch.empty(256 << 20, dtype=torch.uint8, device="cuda")
    fn()                                    # first call outside capture (lazy set-up)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        for _ in range(reps):
            fn()
    for _ in range(3):
        g.replay()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(iters)]
    torch.cuda.synchronize()
    for e0, e1 in ev:
        flush.zero_()
        e0.record(stream)
        g.replay()
        e1.record(stream)
    torch.cuda.synchronize()
    return sum(e0.elapsed_time(e1) for e0, e1 in ev) / (iters * reps)


def _profile(fn, stream):
    """One call under the library's per-launch timing."""
    torch.cuda.synchronize()
    A.adadsf_profile_begin(4096)
    fn()
    return A.adadsf_profile_end(4096)


def case_linear(a, stream):
    g = torch.Generator(device="cuda").manual_seed(0)
    dt = torch.bfloat16 if a.dtype == "bf16" else torch.float32
    x = torch.randn(a.M, a.K, generator=g, device="cuda").to(dt)
    w = (0.02 * torch.randn(a.N, a.K, generator=g, device="cuda")).to(dt)
    b = (0.02 * torch.randn(a.N, generator=g, device="cuda")).to(dt)
    out = torch.empty(a.M, a.N, device="cuda", dtype=dt)
    ws = A.workspace(A.LINEAR_SPLIT_WS_BYTES)
    fn = lambda: A.adadsf_linear(x, w, b, out, act=a.act, ws=ws, stream=stream)
    flops = 2.0 * a.M * a.N * a.K
    return fn, flops, (a.M * a.K + a.N * a.K + a.M * a.N) * x.element_size(), ws


def case_layer(a, stream):
    wl = S.WORKLOADS[a.workload]
    shape = wl.shape.replace(n_layers=1)
    B = a.B or wl.B
    T = a.T or wl.T
    K = a.K if a.K is not None else T // 2
    dt = torch.bfloat16 if shape.dtype == "bf16" else torch.float32
    g = torch.Generator(device="cuda").manual_seed(0)
    w = {n: (0.02 * torch.randn(shp, generator=g, device="cuda")).to(dt)
         for n, shp in S.layer_weight_shapes(shape).items()}
    for n in ("ln1_w", "ln2_w"):
        w[n] = torch.ones_like(w[n])
    x = torch.randn(B, T, shape.d, generator=g, device="cuda").to(dt)
    fold = a.fold or a.gathered
    flags = ((A.FLAG_FOLDED_NORMS if fold else 0) | (A.FLAG_GATE_SIGMOID if a.gate else 0)
             | (A.FLAG_GATHERED_QKV if a.gathered else 0))
    cfg = A.make_cfg(shape, flags)
    if fold:
        A.adadsf_fold_norms(cfg, w, stream)
    ws = A.workspace(A.adadsf_layer_workspace_size(cfg, B, T, K))
    fn = lambda: A.adadsf_sparse_layer_forward(cfg, w, x, K, ws=ws, stream=stream)
    per_tok = 2.0 * (shape.qkv_dim * shape.d + shape.d * shape.q_dim
                     + (3 if shape.arch == S.QWEN else 2) * shape.d * shape.ffn)
    flops = B * K * per_tok + 2.0 * B * shape.n_heads * shape.head_dim * K * (K + 1)
    return fn, flops, 0.0, ws


def case_attention(a, stream):
    wl = S.WORKLOADS[a.workload]
    shape = wl.shape
    B = a.B or wl.B
    K = a.K or wl.T // 2
    dt = torch.bfloat16 if shape.dtype == "bf16" else torch.float32
    g = torch.Generator(device="cuda").manual_seed(0)
    qkv = torch.randn(B * K, shape.qkv_dim, generator=g, device="cuda").to(dt)
    out = torch.empty(B * K, shape.q_dim, device="cuda", dtype=dt)
    cfg = A.make_cfg(shape)
    ws = A.workspace(A.adadsf_attention_workspace_size(cfg, B, K))
    fn = lambda: A.adadsf_causal_attention(cfg, qkv, B, K, out, ws=ws, stream=stream)
    flops = 2.0 * B * shape.n_heads * shape.head_dim * K * (K + 1)
    return fn, flops, (qkv.numel() + out.numel()) * qkv.element_size(), ws


def case_router(a, stream):
    wl = S.WORKLOADS[a.workload]
    shape = wl.shape.replace(n_layers=1)
    B = a.B or wl.B
    T = a.T or wl.T
    dt = torch.bfloat16 if shape.dtype == "bf16" else torch.float32
    g = torch.Generator(device="cuda").manual_seed(0)
    w = {n: (0.02 * torch.randn(shp, generator=g, device="cuda")).to(dt)
         for n, shp in S.layer_weight_shapes(shape).items()}
    x = torch.randn(B * T, shape.d, generator=g, device="cuda").to(dt)
    scores = torch.empty(B * T, device="cuda", dtype=torch.float32)
    cfg = A.make_cfg(shape)
    if a.case == "router_select":
        K = a.K if a.K is not None else T // 2
        idx = torch.empty(B, K, device="cuda", dtype=torch.int32)
        rows = torch.empty(B, K, device="cuda", dtype=torch.int32)
        ws = A.workspace(A.adadsf_router_select_workspace_size(cfg, B, T))
        fn = lambda: A.adadsf_router_select(cfg, w, x, B, T, K, scores, idx, rows, ws=ws, stream=stream)
    else:
        ws = A.workspace(A.adadsf_router_select_workspace_size(cfg, 1, 1))
        fn = lambda: A.adadsf_router_scores(cfg, w, x, scores, ws=ws, stream=stream)
    flops = 2.0 * B * T * shape.d * shape.router_hidden
    return fn, flops, x.numel() * x.element_size(), ws


def case_decode(a, stream):
    """Decode steps (adadsf_decode_step) of a model of the workload's layer
    shape with --layers layers and a small vocabulary, after a prefill of B
    sequences of T tokens at K kept per layer; gbs counts the step's weights
    and the cached keys and values at K per layer."""
    wl = S.WORKLOADS[a.workload]
    shape = wl.shape.replace(n_layers=a.layers, vocab=1024)
    B = a.B or wl.B
    T = a.T or wl.T
    K = a.K if a.K is not None else T // 2
    dt = torch.bfloat16 if shape.dtype == "bf16" else torch.float32
    g = torch.Generator(device="cuda").manual_seed(0)
    layers = []
    for _ in range(shape.n_layers):
        w = {n: (0.02 * torch.randn(shp, generator=g, device="cuda")).to(dt)
             for n, shp in S.layer_weight_shapes(shape).items()}
        for n in ("ln1_w", "ln2_w"):
            w[n] = torch.ones_like(w[n])
        layers.append(w)
    extra = {"embed": (0.02 * torch.randn(shape.vocab, shape.d, generator=g, device="cuda")).to(dt),
             "final_w": torch.ones(shape.d, device="cuda", dtype=dt)}
    if shape.arch == S.NEOX:
        extra["final_b"] = torch.zeros(shape.d, device="cuda", dtype=dt)
    model = A.DeviceModel(A.make_cfg(shape), layers, extra)
    Ks = [K] * shape.n_layers
    steps = (a.warmup + a.iters + 4) * (1 + a.graph)   # every call advances the position
    C_max = T + steps + 8
    cache = A.kv_cache(model.cfg, B, C_max)
    ids = torch.randint(0, shape.vocab, (B, T), generator=g, device="cuda", dtype=torch.int32)
    hid = torch.empty((B, T, shape.d), dtype=dt, device="cuda")
    pws = A.workspace(A.adadsf_model_workspace_size(model.cfg, B, T, Ks, False))
    A.adadsf_prefill(model, ids, Ks, hid, cache, C_max, ws=pws, stream=stream)
    del hid, pws
    ws = A.workspace(A.adadsf_decode_workspace_size(model.cfg, B, C_max))
    tok = torch.randint(0, shape.vocab, (B,), generator=g, device="cuda", dtype=torch.int32)
    h = torch.empty((B, shape.d), dtype=dt, device="cuda")
    fn = lambda: A.adadsf_decode_step(model, tok, h, cache, C_max, ws=ws, stream=stream)
    es = 2 if dt == torch.bfloat16 else 4
    w_bytes = sum(v.numel() for w in layers for v in w.values()) * es
    kv_bytes = shape.n_layers * B * K * 2 * shape.kv_dim * es
    return fn, 0.0, w_bytes + kv_bytes, ws


def case_topk(a, stream):
    wl = S.WORKLOADS[a.workload]
    B = a.B or wl.B
    T = a.T or wl.T
    K = a.K if a.K is not None else T // 2
    g = torch.Generator(device="cuda").manual_seed(0)
    scores = torch.randn(B, T, generator=g, device="cuda")
    idx = torch.empty(B, K, device="cuda", dtype=torch.int32)
    rows = torch.empty(B, K, device="cuda", dtype=torch.int32)
    fn = lambda: A.adadsf_topk_select(scores, K, idx, rows, stream=stream)
    return fn, 0.0, scores.numel() * 4 + 2 * idx.numel() * 4, None


def main():
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("case", choices=("linear", "layer", "attention", "router", "router_select", "topk", "decode"))
    ap.add_argument("--M", type=int, default=8192)
    ap.add_argument("--N", type=int, default=8192)
    ap.add_argument("--K", type=int, default=None)
    ap.add_argument("--T", type=int, default=None)
    ap.add_argument("--B", type=int, default=None)
    ap.add_argument("--act", type=int, default=0)
    ap.add_argument("--dtype", default="bf16")
    ap.add_argument("--workload", default="c3")
    ap.add_argument("--iters", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--profile", action="store_true", help="also report the library's per-launch events")
    ap.add_argument("--fold", action="store_true", help="layer: fold the norms (FLAG_FOLDED_NORMS)")
    ap.add_argument("--gate", action="store_true", help="layer: the score-gated variant")
    ap.add_argument("--gathered", action="store_true",
                    help="layer: folded norms and the first RMSNorm inside the QKV projection (FLAG_GATHERED_QKV)")
    ap.add_argument("--graph", type=int, default=0, help="also time R calls replayed from one CUDA graph")
    ap.add_argument("--layers", type=int, default=2, help="decode: layers of the model")
    a = ap.parse_args()
    if a.case == "linear" and a.K is None:
        a.K = 2048
    A.lib()
    stream = torch.cuda.Stream()
    with torch.cuda.stream(stream):
        fn, flops, nbytes, ws = {"linear": case_linear, "layer": case_layer, "attention": case_attention,
                            "router": case_router, "router_select": case_router,
                            "topk": case_topk, "decode": case_decode}[a.case](a, stream)
        ms = _time(fn, a.iters, a.warmup, stream)
        out = {"case": a.case, "ms": ms}
        if flops:
            out["tflops"] = flops / (ms * 1e9)
        if nbytes:
            out["gbs"] = nbytes / (ms * 1e6)
        if a.graph:
            gms = _time_graph(fn, a.graph, a.iters, stream)
            out["graph_ms"] = gms
            if flops:
                out["graph_tflops"] = flops / (gms * 1e9)
        if a.profile:
            out["launches"] = [(n, ms_, fl / max(ms_, 1e-9) / 1e9) for n, _, ms_, fl, _ in _profile(fn, stream)]
        if ws is not None:
            out["device_status"] = A.adadsf_sync_check(ws, stream)
    print(json.dumps(out))


if __name__ == "__main__":
    main()
