#!/usr/bin/env python
"""Benchmark of the AdaDSF depth-sparse forward on GB300.

One step = one sparse model forward (router, Top-K, gather + norm, QKV + rotary,
attention among kept tokens, output projection, MLP, residual scatter, for
every layer, then the final norm) over one batch of synthetic tokens, at the
per-layer kept counts K_l that the similarity-driven allocation (Eqs. 4-8)
assigns from a dense calibration pass. The calibration pass and the
allocation run once before timing (the retention is fixed across steps) and
are reported separately.

Prints ONE JSON line on rank 0. Default workload: the 12-layer Pythia-160M
shape, B=4, T=512, bf16, mean retention 0.5.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload c2|c3|c4|c5]
  python bench.py --impl reference ...   (the fp64 CPU oracle, same metric)
Multi-GPU: one process per GPU under torchrun; every rank runs its own batch
(replicas, weak scaling, no data-path collective).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

from paper_2607_21291_gb300 import synth as S  # noqa: E402

METRIC = "sparse-forward tokens/s at fixed retention; achieved TFLOP/s & HBM GB/s vs peak"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
L2_FLUSH_BYTES = 256 << 20
TAU, BETA = 0.05, 10.0


# ----------------------------------------------------------------------------- helpers
def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return p, "measured"
    except Exception:
        return dict(FALLBACK_PEAKS), "fallback"


class ClockSampler:
    """nvidia-smi clock / throttle-reason samples while the benchmark runs."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id: str):
        self.samples = []
        self.proc = None
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100", "-i", gpu_id], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) >= 9:
                self.samples.append((time.time(), parts))

    def stop(self, t0: float, t1: float) -> dict:
        if self.proc is None:
            return {"unavailable": "nvidia-smi not runnable"}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        win = [p for (t, p) in self.samples if t0 - 0.15 <= t <= t1 + 0.15] or [p for (_, p) in self.samples[-3:]]
        if not win:
            return {"unavailable": "no nvidia-smi samples"}

        def num(x):
            try:
                return float(x)
            except ValueError:
                return float("nan")
        sm = [num(p[1]) for p in win]
        reasons = set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for p in win:
            for name, v in zip(names, p[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(name)
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(num(p[2]) for p in win),
                "power_w_max": max(num(p[3]) for p in win), "samples": len(win),
                "reasons": sorted(reasons)}


def gpu_id_for_smi(dev_index: int) -> str:
    try:
        u = torch.cuda.get_device_properties(dev_index).uuid
        s = str(u)
        return s if s.startswith("GPU-") else "GPU-" + s
    except Exception:
        vis = os.environ.get("CUDA_VISIBLE_DEVICES")
        if vis:
            return vis.split(",")[dev_index]
        return str(dev_index)


# Sources that decide a kernel family's launches (tile choice, fusion) and code.
KIND_SOURCES = {
    "gemm": ("gemm_tcgen05.cu", "common.cuh", "internal.h", "api.cu"),
}


def kernel_source_hash(kind: str = "") -> str:
    h = hashlib.sha1()
    csrc = os.path.join(ROOT, "paper_2607_21291_gb300", "csrc")
    files = KIND_SOURCES.get(kind) or sorted(os.listdir(csrc))
    for f in files:
        with open(os.path.join(csrc, f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:12]


def recorded_traffic(kind: str, workload: str):
    """DRAM bytes per launch of `kind` from a committed ncu summary, if it was
    taken on the current kernel sources (line: `traffic <workload> <kind> <bytes> <hash>`)."""
    pdir = os.path.join(ROOT, "profiles")
    if not os.path.isdir(pdir):
        return None
    want = kernel_source_hash(kind)
    for f in sorted(os.listdir(pdir)):
        if not f.endswith((".md", ".txt")):
            continue
        for line in open(os.path.join(pdir, f)):
            m = re.search(r"traffic\s+(\S+)\s+(\S+)\s+([0-9.eE+]+)\s+([0-9a-f]{12})", line)
            if m and m.group(1) == workload and m.group(2) == kind and m.group(4) == want:
                return float(m.group(3))
    return None


def retention_of(args, wl):
    if args.retention is not None:
        return args.retention
    return 0.5 if 0.5 in wl.retention else wl.retention[0]


# ----------------------------------------------------------------------------- model set-up
def device_model(A, shape, seed, device):
    """Random-init weights of the backbone shape, drawn on the device (recipe of
    synth: linear weights and biases N(0, 0.02), norm gains 1, norm biases 0)."""
    td = torch.bfloat16 if shape.dtype == "bf16" else torch.float32
    gen = torch.Generator(device=device)

    def draw(tag, shp, std):
        gen.manual_seed(seed * 1000003 + tag)
        return (torch.randn(shp, generator=gen, device=device, dtype=torch.float32) * std).to(td)

    layers = []
    for l in range(shape.n_layers):
        w = {}
        for j, (name, shp) in enumerate(S.layer_weight_shapes(shape).items()):
            if name in ("ln1_w", "ln2_w"):
                w[name] = torch.ones(shp, device=device, dtype=td)
            elif name in ("ln1_b", "ln2_b"):
                w[name] = torch.zeros(shp, device=device, dtype=td)
            else:
                w[name] = draw(l * 64 + j, shp, 0.02)
        layers.append(w)
    extra = {"embed": draw(10 ** 6, (shape.vocab, shape.d), 0.02),
             "final_w": torch.ones(shape.d, device=device, dtype=td)}
    if shape.arch == S.NEOX:
        extra["final_b"] = torch.zeros(shape.d, device=device, dtype=td)
    return A.DeviceModel(A.make_cfg(shape), layers, extra)


def device_ids(seed, B, T, vocab, device):
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    return torch.randint(0, vocab, (B, T), generator=gen, device=device, dtype=torch.int32)


# ----------------------------------------------------------------------------- our arm
def run_ours(args, rank, world, local_rank):
    from paper_2607_21291_gb300 import adadsf as A
    A.lib()
    device = torch.device("cuda", local_rank)
    torch.cuda.set_device(device)
    wl = S.WORKLOADS[args.workload]
    shape, B, T = wl.shape, wl.B, wl.T
    L = shape.n_layers
    t_target = retention_of(args, wl)
    stream = torch.cuda.Stream(device)
    model = device_model(A, shape, 2, device)
    sampler = ClockSampler(gpu_id_for_smi(local_rank))

    with torch.cuda.stream(stream):
        # ---- calibration (Eq. 4, dense forward) + allocation (Eqs. 5-8), once
        ids_cal = device_ids(1 + 7919 * rank, *wl.calib, shape.vocab, device)
        Kd = [T] * L
        ws = A.workspace(max(A.adadsf_model_workspace_size(model.cfg, max(B, wl.calib[0]), T, Kd, True), 256), device)
        acc = torch.zeros(2 * L, dtype=torch.float64, device=device)
        hid_cal = torch.empty((wl.calib[0], T, shape.d), dtype=torch.bfloat16, device=device)
        A.adadsf_sparse_model_forward(model, ids_cal, Kd, hid_cal, stats_acc=acc, ws=ws, stream=stream)
        torch.cuda.synchronize()
        c0 = torch.cuda.Event(enable_timing=True)
        c1 = torch.cuda.Event(enable_timing=True)
        acc.zero_()
        c0.record(stream)
        A.adadsf_sparse_model_forward(model, ids_cal, Kd, hid_cal, stats_acc=acc, ws=ws, stream=stream)
        c1.record(stream)
        torch.cuda.synchronize()
        calib_ms = c0.elapsed_time(c1)
        # event profile of one calibration forward (the Eq. 4 statistics kernel)
        acc.zero_()
        A.adadsf_profile_begin(4 + 12 * L)
        A.adadsf_sparse_model_forward(model, ids_cal, Kd, hid_cal, stats_acc=acc, ws=ws, stream=stream)
        cal_recs = A.adadsf_profile_end(4 + 12 * L)
        torch.cuda.synchronize()
        from paper_2607_21291_gb300 import calibrate as C
        acc = C.allreduce_stats(acc)          # the one exchange: 2L doubles over replicas
        s, r, K = C.retention_plan(acc, T, t_target, TAU, BETA)
        K = [int(k) for k in K]

        # spin-up: keep the GPU busy ~1.5 s so its clocks leave the idle state
        # before anything is measured (the calibration forward, repeated)
        spin_t0 = time.time()
        spin_n = 0
        while time.time() - spin_t0 < args.spin_up:
            A.adadsf_sparse_model_forward(model, ids_cal, Kd, hid_cal, ws=ws, stream=stream)
            spin_n += 1
            if spin_n % 8 == 0:
                torch.cuda.synchronize()
        torch.cuda.synchronize()

        ids = device_ids(2 + 7919 * rank, B, T, shape.vocab, device)
        hidden = torch.empty((B, T, shape.d), dtype=torch.bfloat16, device=device)
        flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=device)

        def fwd(Ks):
            A.adadsf_sparse_model_forward(model, ids, Ks, hidden, ws=ws, stream=stream)

        # ---- per-launch profile (eager), a handful of steps
        for _ in range(2):
            fwd(K)
        torch.cuda.synchronize()
        n_prof = max(3, min(10, args.steps))
        A.adadsf_profile_begin((4 + 12 * L) * n_prof)
        for _ in range(n_prof):
            flush.zero_()
            torch.cuda.nvtx.range_push("adadsf_sparse_step")
            fwd(K)
            torch.cuda.nvtx.range_pop()
        recs = A.adadsf_profile_end((4 + 12 * L) * n_prof)
        bad = [r for r in recs if r[2] < 0]
        assert not bad, f"launch timing failed: {bad[:3]}"
        assert A.adadsf_sync_check(ws, stream) == A.OK, A.adadsf_last_error()
        launches_per_step = len(recs) // n_prof

        # ---- CUDA graphs of the sparse and the dense forward
        graphs = {}
        for name, Ks in (("sparse", K), ("dense", Kd)):
            for _ in range(max(3, args.warmup)):
                fwd(Ks)
            torch.cuda.synchronize()
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                fwd(Ks)
            graphs[name] = g
        torch.cuda.synchronize()

        def time_graph(g, steps, warmup):
            for _ in range(warmup):
                flush.zero_()
                g.replay()
            ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
            if world > 1:
                torch.distributed.barrier()
            torch.cuda.synchronize()
            t0 = time.time()
            for e0, e1 in ev:
                flush.zero_()
                e0.record(stream)
                g.replay()
                e1.record(stream)
            torch.cuda.synchronize()
            t1 = time.time()
            if world > 1:
                torch.distributed.barrier()
            return [e0.elapsed_time(e1) for e0, e1 in ev], t0, t1

        dense_ms, _, _ = time_graph(graphs["dense"], max(3, args.steps // 4), args.warmup)
        step_ms, t0, t1 = time_graph(graphs["sparse"], args.steps, args.warmup)
        assert A.adadsf_sync_check(ws, stream) == A.OK, A.adadsf_last_error()

        # ---- end to end through the public call, host buffers in and out
        ids_host = ids.cpu().pin_memory()
        out_host = torch.empty(hidden.shape, dtype=hidden.dtype, pin_memory=True)
        for _ in range(args.warmup):
            ids.copy_(ids_host, non_blocking=True)
            fwd(K)
            out_host.copy_(hidden, non_blocking=True)
        e2e_ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                  for _ in range(args.steps)]
        torch.cuda.synchronize()
        for e0, e1 in e2e_ev:
            flush.zero_()
            e0.record(stream)
            ids.copy_(ids_host, non_blocking=True)
            fwd(K)
            out_host.copy_(hidden, non_blocking=True)
            e1.record(stream)
        torch.cuda.synchronize()
        e2e_ms = [e0.elapsed_time(e1) for e0, e1 in e2e_ev]

    clocks = sampler.stop(t0, t1)
    ms = float(np.mean(step_ms))
    e2e = float(np.mean(e2e_ms))
    dense = float(np.mean(dense_ms))
    if world > 1:
        t = torch.tensor([ms, e2e, dense], device=device, dtype=torch.float64)
        torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
        ms, e2e, dense = t.tolist()
    if rank != 0:
        return

    tokens = B * T * world
    # ---- per-kernel aggregates and the roofline of the dominant kernel
    agg = {}
    for name, dense_flag, kms, fl, by in recs:
        a_ = agg.setdefault(name, {"launches": 0, "ms": 0.0, "flops": 0.0, "bytes": 0.0, "dense": dense_flag})
        a_["launches"] += 1
        a_["ms"] += kms
        a_["flops"] += fl
        a_["bytes"] += by
    tot_ms = sum(v["ms"] for v in agg.values())
    peaks, peak_src = load_peaks()
    # the HBM-bound steps before the projections (router, Top-K, gather +
    # norms) as one figure: their bytes over their time
    hbm_names = [n for n in agg if n in ("router", "topk", "gather_norm", "topk_gather_norm")]
    hbm_ms = sum(agg[n]["ms"] for n in hbm_names)
    hbm_path = None
    if hbm_ms > 0:
        gbs = sum(agg[n]["bytes"] for n in hbm_names) / (hbm_ms * 1e6)
        hbm_path = {"kernels": sorted(hbm_names), "gbs": gbs, "frac_of_hbm_peak": gbs / peaks["hbm_gbs"],
                    "ms_per_step": hbm_ms / n_prof}
    st = [r for r in cal_recs if r[0] == "stats" and r[2] > 0]
    stats_kernel = None
    if st:
        st_ms, st_bytes = sum(r[2] for r in st), sum(r[4] for r in st)
        stats_kernel = {"launches": len(st), "ms_per_launch": st_ms / len(st),
                        "gbs": st_bytes / (st_ms * 1e6), "frac_of_hbm_peak": st_bytes / (st_ms * 1e6) / peaks["hbm_gbs"]}
    long_step = ms * args.steps > 1000.0
    tc_peak = peaks["bf16_tflops_sustained" if long_step else "bf16_tflops"]
    kernels = {}
    for name, v in sorted(agg.items(), key=lambda kv: -kv[1]["ms"]):
        per = v["launches"] / n_prof
        k = {"launches_per_step": per, "ms_per_step": v["ms"] / n_prof, "share": v["ms"] / tot_ms}
        if v["dense"]:
            k["tflops"] = v["flops"] / (v["ms"] * 1e9)
            k["frac_of_bf16_peak"] = k["tflops"] / tc_peak
        else:
            k["gbs"] = v["bytes"] / (v["ms"] * 1e6)
            k["frac_of_hbm_peak"] = k["gbs"] / peaks["hbm_gbs"]
        kernels[name] = k
    # the dominant kernel binary is the tcgen05 GEMM (qkv/o/up/down/router share it)
    gemm_names = [n for n in agg if n.startswith("gemm_")]
    gemm_ms = sum(agg[n]["ms"] for n in gemm_names)
    top = max(agg, key=lambda n: agg[n]["ms"])
    if gemm_names and gemm_ms >= agg[top]["ms"]:
        launches = sum(agg[n]["launches"] for n in gemm_names)
        flops = sum(agg[n]["flops"] for n in gemm_names)
        achieved = flops / (gemm_ms * 1e9)
        roof = {"kernel": "gemm_tc_kernel (tcgen05 projections: " + ",".join(sorted(gemm_names)) + ")",
                "bound": "tensor", "achieved": achieved, "peak": tc_peak, "unit": "TFLOP/s",
                "frac": achieved / tc_peak,
                "peak_source": f"{peak_src} {'bf16_tflops_sustained' if long_step else 'bf16_tflops'}",
                "avg_launch_ms": gemm_ms / launches,
                "traffic": recorded_traffic("gemm", wl.name)}
    else:
        v = agg[top]
        if v["dense"]:
            achieved = v["flops"] / (v["ms"] * 1e9)
            roof = {"kernel": top, "bound": "tensor", "achieved": achieved, "peak": tc_peak,
                    "unit": "TFLOP/s", "frac": achieved / tc_peak}
        else:
            achieved = v["bytes"] / (v["ms"] * 1e6)
            roof = {"kernel": top, "bound": "hbm", "achieved": achieved, "peak": peaks["hbm_gbs"],
                    "unit": "GB/s", "frac": achieved / peaks["hbm_gbs"]}
        roof["peak_source"] = peak_src
        roof["avg_launch_ms"] = v["ms"] / v["launches"]
        roof["traffic"] = recorded_traffic(top, wl.name)

    sparse_flops = sum(v["flops"] for v in agg.values()) / n_prof
    out = {
        "metric": METRIC,
        "value": tokens / (ms * 1e-3),
        "unit": "tokens/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": ms,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16" if shape.dtype == "bf16" else "f32",
        "data": "synthetic (seeded token ids, random-init weights of the backbone shape)",
        "config": {"workload": wl.name, "model": shape.name, "B": B, "T": T, "layers": L,
                   "global_batch": B * world, "seq_len": T, "retention_target": t_target,
                   "K_per_layer": K, "retention_mean": float(np.mean(K)) / T,
                   "tau": TAU, "beta": BETA, "parallelism": f"replicas x{world} (batch-sharded, no collective)",
                   "l2": "flushed between timed steps (256 MiB write outside the step events)",
                   "spin_up": f"{spin_n} dense forwards over {args.spin_up:.1f} s before any measurement",
                   "timing": "CUDA graph replay of adadsf_sparse_model_forward, CUDA events per step"},
        "roofline": roof,
        "e2e": {"value": tokens / (e2e * 1e-3), "unit": "tokens/s",
                "h2d_bytes_per_step": int(ids.numel() * ids.element_size()),
                "d2h_bytes_per_step": int(hidden.numel() * hidden.element_size()),
                "how": "eager adadsf_sparse_model_forward per step with pinned-host ids in and hidden states out"},
        "gpu_launches": launches_per_step * args.steps,
        "clocks": clocks,
        "dense_same_kernels": {"ms_per_step": dense, "value": tokens / (dense * 1e-3), "unit": "tokens/s"},
        "hbm_path": hbm_path,
        "calibration": {"ms": calib_ms, "stats_kernel": stats_kernel, "batch": list(wl.calib), "similarity": [float(x) for x in s],
                        "ratios": [float(x) for x in r]},
        "normalized_flops": sparse_flops / max(1.0, sum(
            (2.0 * B * T * (shape.qkv_dim * shape.d + shape.d * shape.q_dim +
                            (3 if shape.arch == S.QWEN else 2) * shape.d * shape.ffn) +
             2.0 * B * shape.n_heads * shape.head_dim * T * (T + 1)) for _ in range(L))),
        "kernels": kernels,
    }
    if world == 1 and not args.no_cpu_baseline:
        out["cpu_baseline"] = cpu_baseline(model, shape, K, ids, budget_s=args.cpu_budget)
    print(json.dumps(out), flush=True)


def host_threads() -> int:
    """Threads the oracle's NumPy BLAS runs with: threadpoolctl's report where
    it is installed, else the CPUs this process may run on (OpenBLAS's
    default)."""
    try:
        from threadpoolctl import threadpool_info
        n = [i["num_threads"] for i in threadpool_info() if i.get("user_api") == "blas"]
        if n:
            return max(n)
    except ImportError:
        pass
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def cpu_baseline(model, shape, K, ids, budget_s=20.0):
    """The fp64 oracle as it stands on the host cores, on a bounded sample of the
    same workload: sequence after sequence, layer after layer (each layer's
    weights copied to the host when first used), until about budget_s; the
    rate is extrapolated to all layers from the mean time of one layer on one
    sequence."""
    from oracle import adadsf_oracle as O
    to = lambda t: t.float().cpu().numpy().astype(np.float64)
    p = O.params_of(shape)
    ids_h = ids.cpu().numpy()
    B, T = ids_h.shape
    L = shape.n_layers
    host = {}
    spent, n_evals, seqs = 0.0, 0, 0
    for b in range(B):
        x = to(model.extra["embed"][ids[b:b + 1].long()])
        for l in range(L):
            if l not in host:
                host[l] = {k: to(v) for k, v in model.layers[l].items()}
            t0 = time.time()
            x, _, _ = O.sparse_layer_forward(x, host[l], p, K[l])
            spent += time.time() - t0
            n_evals += 1
            if spent > budget_s:
                break
        seqs += 1
        if spent > budget_s:
            break
    per_layer_seq = spent / n_evals
    return {"value": T / (per_layer_seq * L), "unit": "tokens/s", "cores": host_threads(), "kind": "oracle",
            "sample": f"{n_evals} (sequence, layer) evaluations over {seqs} of {B} sequences x {T} tokens, "
                      f"fp64 NumPy (BLAS threads = host cores), {spent:.1f} s; rate extrapolated to all "
                      f"{L} layers"}


# ----------------------------------------------------------------------------- reference arm
def run_reference(args, rank, world):
    """The fp64 CPU oracle timed on the host cores: each step pushes one
    sequence of the workload through every sparse layer."""
    if rank != 0:
        return
    from oracle import adadsf_oracle as O
    wl = S.WORKLOADS[args.workload]
    shape, T = wl.shape, wl.T
    L = shape.n_layers
    t_target = retention_of(args, wl)
    layers = [{k: S.round_to(v, shape.dtype).astype(np.float64)
               for k, v in S.layer_weights(shape, 2, l, gain_std=0.0).items()} for l in range(L)]
    extra = {k: S.round_to(v, shape.dtype).astype(np.float64)
             for k, v in S.model_extra_weights(shape, 2, gain_std=0.0).items()}
    p = O.params_of(shape)
    ids_cal = S.token_ids(1, 1, T, shape.vocab)
    _, _, st = O.sparse_model_forward(ids_cal, extra, layers, p, [T] * L, stats_mode="token")
    s = np.array([O.similarity(a) for a in st])
    r, _ = O.allocate_ratios(s, t_target, TAU, BETA)
    K = O.kept_counts(r, T).tolist()
    ids = S.token_ids(2, args.warmup + args.steps, T, shape.vocab)
    for i in range(args.warmup):
        O.sparse_model_forward(ids[i:i + 1], extra, layers, p, K)
    t = []
    for i in range(args.steps):
        t0 = time.time()
        O.sparse_model_forward(ids[args.warmup + i:args.warmup + i + 1], extra, layers, p, K)
        t.append(time.time() - t0)
    sec = float(np.mean(t))
    v = T / sec
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": v, "unit": "tokens/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": sec * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": wl.name, "model": shape.name, "B": 1, "T": T, "layers": L,
                   "retention_target": t_target, "K_per_layer": K},
        "cpu_baseline": {"value": v, "unit": "tokens/s", "cores": host_threads(), "kind": "oracle",
                         "sample": f"1 sequence x {T} tokens per step through all {L} layers"},
        "e2e": {"value": v, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }), flush=True)


# ----------------------------------------------------------------------------- main
def main():
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--workload", choices=("c2", "c3", "c4", "c5"), default="c2")
    ap.add_argument("--retention", type=float, default=None)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-budget", type=float, default=20.0)
    ap.add_argument("--spin-up", type=float, default=1.5, help="seconds of untimed GPU work before measuring")
    args = ap.parse_args()
    args.warmup = max(3, args.warmup)

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        run_reference(args, rank, world)
        return
    if world > 1:
        torch.cuda.set_device(local_rank)
        torch.distributed.init_process_group("nccl")
    try:
        run_ours(args, rank, world, local_rank)
    finally:
        if world > 1:
            torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
