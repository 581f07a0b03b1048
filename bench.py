#!/usr/bin/env python
"""Benchmark of the AdaDSF depth-sparse forward on GB300.

One step = one sparse model forward (router, Top-K, gather + norm, QKV + rotary,
attention among kept tokens, output projection, MLP, residual scatter, for
every layer, then the final norm) over one batch of synthetic tokens, at the
per-layer kept counts K_l that the similarity-driven allocation (Eqs. 4-8)
assigns from a dense calibration pass. The calibration pass and the
allocation run once before timing (the retention is fixed across steps) and
are reported separately.

Prints ONE JSON line on rank 0. Default workload: the 28-layer Qwen2.5-7B
shape, B=16, T=4096, bf16, mean retention 0.5 (calibration over 16 x 4096
tokens), with the retention sweep 1.0 / 0.75 / 0.25 in the same line.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload c2|c3|c4|c5]
  python bench.py --impl reference ...   (the fp64 CPU oracle, same metric)
Multi-GPU: one process per GPU under torchrun; every rank runs its own batch
(replicas, weak scaling, no data-path collective).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
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
WEIGHT_SEED, CALIB_SEED, EVAL_SEED = 2, 1, 2
RECIPE = ("counter-based draws (synth.bench_*): linear weights and biases N(0, 0.02), norm gains 1, "
          "norm biases 0, weight seed 2; token ids uniform over the vocabulary, calibration seed 1, "
          "evaluation seed 2")
L2_NOTE = ("GPU arm: L2 flushed between timed steps (256 MiB write outside the step events); "
           "CPU oracle arm: each step's fp64 layer weights exceed every host cache")


def rank_seed(seed, rank):
    return seed + 7919 * rank


def device_model(A, shape, seed, device, fold=False, gathered=False):
    """Random-init weights of the backbone shape in the benchmark recipe,
    drawn on the device (the reference arm draws the same tensors). With
    fold, the norm parameters are folded into the projections
    (adadsf_fold_norms; exact here, as the recipe's gains are 1 and biases 0)
    and the layers run with ADADSF_FLAG_FOLDED_NORMS (and, with gathered,
    ADADSF_FLAG_GATHERED_QKV)."""
    td = torch.bfloat16 if shape.dtype == "bf16" else torch.float32
    flags = (A.FLAG_FOLDED_NORMS | (A.FLAG_GATHERED_QKV if gathered else 0)) if fold else 0
    cfg = A.make_cfg(shape, flags)
    layers = []
    for l in range(shape.n_layers):
        w = {k: v.to(td) for k, v in S.bench_layer_weights(shape, seed, l, device).items()}
        if fold:
            A.adadsf_fold_norms(cfg, w)
        layers.append(w)
    extra = {"embed": S.bench_embed(shape, seed, device).to(td),
             "final_w": torch.ones(shape.d, device=device, dtype=td)}
    if shape.arch == S.NEOX:
        extra["final_b"] = torch.zeros(shape.d, device=device, dtype=td)
    return A.DeviceModel(cfg, layers, extra)


def shared_config(wl, t_target, world):
    """The workload's definition: identical in both arms' JSON lines."""
    shape = wl.shape
    return {"workload": wl.name, "model": shape.name, "B": wl.B, "T": wl.T, "layers": shape.n_layers,
            "global_batch": wl.B * world, "seq_len": wl.T, "retention_target": t_target,
            "tau": TAU, "beta": BETA, "calibration_batch": list(wl.calib), "inputs": RECIPE,
            "parallelism": f"replicas x{world} (batch-sharded, no collective)", "l2": L2_NOTE}


def dense_flops_per_layer(shape, B, T):
    """GEMM + causal-attention flops of one dense layer over B sequences of T."""
    per_tok = 2.0 * (shape.qkv_dim * shape.d + shape.d * shape.q_dim
                     + (3 if shape.arch == S.QWEN else 2) * shape.d * shape.ffn)
    return B * T * per_tok + 2.0 * B * shape.n_heads * shape.head_dim * T * (T + 1)


# ----------------------------------------------------------------------------- our arm
def run_ours(args, rank, world, local_rank):
    from paper_2607_21291_gb300 import adadsf as A
    from paper_2607_21291_gb300 import calibrate as C
    A.lib()
    device = torch.device("cuda", local_rank)
    torch.cuda.set_device(device)
    wl = S.WORKLOADS[args.workload]
    shape, B, T = wl.shape, wl.B, wl.T
    L = shape.n_layers
    t_target = retention_of(args, wl)
    stream = torch.cuda.Stream(device)
    model = device_model(A, shape, WEIGHT_SEED, device, fold=args.folded_norms or args.gathered_qkv,
                         gathered=args.gathered_qkv)
    sampler = ClockSampler(gpu_id_for_smi(local_rank))
    n_rec = 4 + 12 * L

    with torch.cuda.stream(stream):
        # ---- calibration (Eq. 4, dense forward) + allocation (Eqs. 5-8), once
        ids_cal = S.counter_ids(rank_seed(CALIB_SEED, rank), *wl.calib, shape.vocab, device)
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
        A.adadsf_profile_begin(n_rec)
        A.adadsf_sparse_model_forward(model, ids_cal, Kd, hid_cal, stats_acc=acc, ws=ws, stream=stream)
        cal_recs = A.adadsf_profile_end(n_rec)
        acc = C.allreduce_stats(acc)          # the one exchange: 2L doubles over replicas
        plans = {}
        for t in sorted(set((t_target,) + tuple(wl.retention))):
            s_, r_, K_ = C.retention_plan(acc, T, t, TAU, BETA)
            plans[t] = (s_, r_, [int(k) for k in K_])
        s, r, K = plans[t_target]
        del hid_cal

        # spin-up: keep the GPU busy before anything is measured, so its
        # clocks leave the idle state (the calibration forward, repeated)
        spin_t0 = time.time()
        spin_n = 0
        spin_out = torch.empty((wl.calib[0], T, shape.d), dtype=torch.bfloat16, device=device)
        while time.time() - spin_t0 < args.spin_up:
            A.adadsf_sparse_model_forward(model, ids_cal, Kd, spin_out, ws=ws, stream=stream)
            spin_n += 1
            torch.cuda.synchronize()
        del spin_out

        ids = S.counter_ids(rank_seed(EVAL_SEED, rank), B, T, shape.vocab, device)
        hidden = torch.empty((B, T, shape.d), dtype=torch.bfloat16, device=device)
        flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=device)

        def fwd(Ks):
            A.adadsf_sparse_model_forward(model, ids, Ks, hidden, ws=ws, stream=stream)

        # ---- per-launch profile (eager), a handful of steps
        for _ in range(2):
            fwd(K)
        torch.cuda.synchronize()
        n_prof = max(3, min(10, args.steps))
        A.adadsf_profile_begin(n_rec * n_prof)
        for _ in range(n_prof):
            flush.zero_()
            torch.cuda.nvtx.range_push("adadsf_sparse_step")
            fwd(K)
            torch.cuda.nvtx.range_pop()
        recs = A.adadsf_profile_end(n_rec * n_prof)
        bad = [x for x in recs if x[2] < 0]
        assert not bad, f"launch timing failed: {bad[:3]}"
        assert A.adadsf_sync_check(ws, stream) == A.OK, A.adadsf_last_error()
        launches_per_step = len(recs) // n_prof

        def capture(Ks):
            for _ in range(max(3, args.warmup)):
                fwd(Ks)
            torch.cuda.synchronize()
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                fwd(Ks)
            torch.cuda.synchronize()
            return g

        def time_graph(g, steps, warmup, barrier=False, nvtx_name="adadsf_replay"):
            for _ in range(warmup):
                flush.zero_()
                g.replay()
            ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
            if barrier and world > 1:
                torch.distributed.barrier()
            torch.cuda.synchronize()
            t0 = time.time()
            for e0, e1 in ev:
                flush.zero_()
                e0.record(stream)
                torch.cuda.nvtx.range_push(nvtx_name)   # lets an ncu launch list select the replays
                g.replay()
                torch.cuda.nvtx.range_pop()
                e1.record(stream)
            torch.cuda.synchronize()
            t1 = time.time()
            if barrier and world > 1:
                torch.distributed.barrier()
            return [e0.elapsed_time(e1) for e0, e1 in ev], t0, t1

        # ---- the timed region: the sparse forward at the target retention
        g_sparse = capture(K)
        step_ms, t0, t1 = time_graph(g_sparse, args.steps, args.warmup, barrier=True,
                                     nvtx_name="adadsf_sparse_replay")
        clocks = sampler.stop(t0, t1)
        assert A.adadsf_sync_check(ws, stream) == A.OK, A.adadsf_last_error()
        del g_sparse

        # ---- the dense forward on the same kernels, and the retention sweep
        n_side = max(3, args.steps // 4)
        g_dense = capture(Kd)
        dense_ms, _, _ = time_graph(g_dense, n_side, 2)
        del g_dense
        sweep = {}
        for t, (_, _, Kt) in sorted(plans.items()):
            if t == t_target:
                continue
            if all(k == T for k in Kt):
                ms_t = dense_ms
            else:
                g_t = capture(Kt)
                ms_t, _, _ = time_graph(g_t, n_side, 2)
                del g_t
            mt = float(np.mean(ms_t))
            sweep[f"{t:g}"] = {"ms_per_step": mt, "value": B * T * world / (mt * 1e-3), "unit": "tokens/s",
                               "K_per_layer": Kt, "retention_mean": float(np.mean(Kt)) / T, "steps": len(ms_t),
                               "normalized_flops": A.adadsf_normalized_flops(model.cfg, T, Kt),
                               "dense": all(k == T for k in Kt)}
        assert A.adadsf_sync_check(ws, stream) == A.OK, A.adadsf_last_error()

        # ---- generation: prefill the batch into a kept-token cache, then
        # decode steps (one token per sequence) replayed from a CUDA graph
        decode = None
        if args.decode_steps > 0:
            decode = run_decode(A, model, shape, ids, K, B, T, args, stream, device, world)

        # ---- end to end through the public call, host buffers in and out:
        # every step copies its token ids in from pinned host memory and its
        # hidden states back out, inside the timed region; the copy back of
        # step i runs on a second stream under step i + 1's forward (two
        # device output buffers), and the region ends when the last copy has
        # landed. The L2 flush between steps stays inside the region too.
        ids_host = ids.cpu().pin_memory()
        outs = [hidden, torch.empty_like(hidden)]
        out_host = [torch.empty(hidden.shape, dtype=hidden.dtype, pin_memory=True) for _ in range(2)]
        copy_stream = torch.cuda.Stream(device)
        done = [torch.cuda.Event() for _ in range(2)]     # forward i has written outs[i % 2]
        copied = [torch.cuda.Event() for _ in range(2)]   # outs[i % 2] has been read back

        def e2e_step(i):
            b = i % 2
            if i >= 2:
                stream.wait_event(copied[b])
            flush.zero_()
            ids.copy_(ids_host, non_blocking=True)
            A.adadsf_sparse_model_forward(model, ids, K, outs[b], ws=ws, stream=stream)
            done[b].record(stream)
            copy_stream.wait_event(done[b])
            with torch.cuda.stream(copy_stream):
                out_host[b].copy_(outs[b], non_blocking=True)
            copied[b].record(copy_stream)

        for i in range(args.warmup):
            e2e_step(i)
        torch.cuda.synchronize()
        e_start, e_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e_start.record(stream)
        for i in range(args.steps):
            e2e_step(i)
        for b in range(min(2, args.steps)):
            stream.wait_event(copied[b])
        e_end.record(stream)
        torch.cuda.synchronize()
        e2e_ms = [e_start.elapsed_time(e_end) / args.steps]

    ms = float(np.mean(step_ms))
    e2e = float(np.mean(e2e_ms))
    dense = float(np.mean(dense_ms))
    if world > 1:
        tt = torch.tensor([ms, e2e, dense], device=device, dtype=torch.float64)
        torch.distributed.all_reduce(tt, op=torch.distributed.ReduceOp.MAX)
        ms, e2e, dense = tt.tolist()
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
    st = [x for x in cal_recs if x[0] == "stats" and x[2] > 0]
    stats_kernel = None
    if st:
        st_ms, st_bytes = sum(x[2] for x in st), sum(x[4] for x in st)
        stats_kernel = {"launches": len(st), "ms_per_launch": st_ms / len(st),
                        "gbs": st_bytes / (st_ms * 1e6), "frac_of_hbm_peak": st_bytes / (st_ms * 1e6) / peaks["hbm_gbs"]}
    long_step = ms * args.steps > 1000.0
    tc_key = "bf16_tflops_sustained" if long_step else "bf16_tflops"
    tc_peak = peaks[tc_key]
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
    # the dominant kernel binary is the tcgen05 GEMM (QKV / output / MLP projections)
    gemm_names = [n for n in agg if n.startswith("gemm_")]
    gemm_ms = sum(agg[n]["ms"] for n in gemm_names)
    top = max(agg, key=lambda n: agg[n]["ms"])
    if gemm_names and gemm_ms >= agg[top]["ms"]:
        launches = sum(agg[n]["launches"] for n in gemm_names)
        flops = sum(agg[n]["flops"] for n in gemm_names)
        achieved = flops / (gemm_ms * 1e9)
        roof = {"kernel": "tcgen05 projection GEMMs (" + ",".join(sorted(gemm_names)) + ")",
                "bound": "tensor", "achieved": achieved, "peak": tc_peak, "unit": "TFLOP/s",
                "frac": achieved / tc_peak, "peak_source": f"{peak_src} {tc_key}",
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
        "config": shared_config(wl, t_target, world),
        "timing": {"how": "CUDA graph replay of adadsf_sparse_model_forward, CUDA events per step on the "
                          "launching stream",
                   "spin_up": f"{spin_n} dense forwards over {args.spin_up:.1f} s before any measurement"},
        "retention_plan": {"K_per_layer": K, "retention_mean": float(np.mean(K)) / T,
                           "similarity": [float(x) for x in s], "ratios": [float(x) for x in r],
                           "calibration": f"dense forward with Eq. 4 statistics over {wl.calib[0]} x {wl.calib[1]} "
                                          f"tokens per replica on this GPU, summed over {world} replica(s)"},
        "roofline": roof,
        "e2e": {"value": tokens / (e2e * 1e-3), "unit": "tokens/s",
                "h2d_bytes_per_step": int(ids.numel() * ids.element_size()),
                "d2h_bytes_per_step": int(hidden.numel() * hidden.element_size()),
                "how": "eager adadsf_sparse_model_forward per step, pinned-host ids copied in and hidden states "
                       "copied out every step (the copy out of step i on a second stream under step i+1); "
                       "one event pair around all steps, L2 flush between steps inside it"},
        "gpu_launches": launches_per_step * args.steps,
        "folded_norms": bool(args.folded_norms or args.gathered_qkv),
        "gathered_qkv": bool(args.gathered_qkv),
        "clocks": clocks,
        "dense_same_kernels": {"ms_per_step": dense, "value": tokens / (dense * 1e-3), "unit": "tokens/s",
                               "steps": n_side},
        "retention_sweep": sweep,
        "hbm_path": hbm_path,
        "decode": decode,
        "calibration": {"ms": calib_ms, "stats_kernel": stats_kernel, "batch": list(wl.calib)},
        "normalized_flops": A.adadsf_normalized_flops(model.cfg, T, K),
        "kernels": kernels,
        "kernels_vs_step": {"sum_ms_per_step": tot_ms / n_prof, "graph_ms_per_step": ms,
                            "ratio": tot_ms / n_prof / ms,
                            "how": "kernels: an eager pass with CUDA events around every launch (no overlap "
                                   "between launches); graph: the timed replay, where each launch's prologue "
                                   "overlaps the previous one (programmatic dependent launch)"},
    }
    if world == 1 and not args.no_cpu_baseline:
        out["cpu_baseline"] = cpu_baseline(model, shape, K, ids, budget_s=args.cpu_budget)
    print(json.dumps(out), flush=True)


def run_decode(A, model, shape, ids, K, B, T, args, stream, device, world):
    """Prefill of the evaluation batch into a kept-token cache at the plan's
    K_l, then args.decode_steps decode steps (one new token per sequence),
    captured once in a CUDA graph and replayed; per step the algorithmic HBM
    bytes are every layer's weights (routers included) plus the cached keys
    and values the step's attention reads."""
    L, n = shape.n_layers, args.decode_steps
    C_max = T + n + 8
    cache = A.kv_cache(model.cfg, B, C_max, device)
    hid = torch.empty((B, T, shape.d), dtype=torch.bfloat16, device=device)
    pws = A.workspace(A.adadsf_model_workspace_size(model.cfg, B, T, K, False), device)
    A.adadsf_prefill(model, ids, K, hid, cache, C_max, ws=pws, stream=stream)
    del hid, pws
    dws = A.workspace(A.adadsf_decode_workspace_size(model.cfg, B, C_max), device)
    new_ids = S.counter_ids(rank_seed(3, 0), n + 1, B, shape.vocab, device)
    tok = torch.empty(B, dtype=torch.int32, device=device)
    h = torch.empty((B, shape.d), dtype=torch.bfloat16, device=device)
    kept = torch.zeros((L, B), dtype=torch.int32, device=device)
    kept_sum = torch.zeros((L, B), dtype=torch.int64, device=device)
    tok.copy_(new_ids[0])
    A.adadsf_decode_step(model, tok, h, cache, C_max, kept_out=kept, ws=dws, stream=stream)   # outside the graph
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        A.adadsf_decode_step(model, tok, h, cache, C_max, kept_out=kept, ws=dws, stream=stream)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n)]
    torch.cuda.synchronize()
    for i, (e0, e1) in enumerate(ev):
        tok.copy_(new_ids[i + 1])
        e0.record(stream)
        g.replay()
        e1.record(stream)
        kept_sum += kept
    torch.cuda.synchronize()
    assert A.adadsf_sync_check(dws, stream) == A.OK, A.adadsf_last_error()
    ms = float(np.mean([e0.elapsed_time(e1) for e0, e1 in ev]))
    # one more step, eager under the library's per-launch events: where a
    # decode step's time goes
    tok.copy_(new_ids[0])
    torch.cuda.synchronize()
    A.adadsf_profile_begin(64 * L + 16)
    A.adadsf_decode_step(model, tok, h, cache, C_max, kept_out=kept, ws=dws, stream=stream)
    recs = A.adadsf_profile_end(64 * L + 16)
    prof = {}
    for name, _, kms, _, by in recs:
        a_ = prof.setdefault(name, {"launches": 0, "ms": 0.0, "bytes": 0.0})
        a_["launches"] += 1
        a_["ms"] += kms
        a_["bytes"] += by
    es = 2 if shape.dtype == "bf16" else 4
    w_bytes = sum(v.numel() for lw in model.layers for v in lw.values()) * es
    # cached keys / values read by the timed steps: the prompt's kept tokens
    # plus those kept during the steps (mean over the steps)
    kv_tok = sum(K) * B + float(kept_sum.sum()) / 2
    kv_bytes = kv_tok * 2 * shape.kv_dim * es
    peaks, _ = load_peaks()
    bytes_step = w_bytes + kv_bytes
    gbs = bytes_step / (ms * 1e6)
    return {"steps": n, "ms_per_step": ms, "value": B * world / (ms * 1e-3), "unit": "tokens/s",
            "prompt": T, "kept_fraction": float(kept_sum.sum()) / (n * L * B),
            "roofline": {"bound": "hbm", "achieved": gbs, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                         "frac": gbs / peaks["hbm_gbs"], "bytes_per_step": bytes_step},
            "kernels_eager": {k: {"launches": v["launches"], "ms": v["ms"],
                                  "gbs": v["bytes"] / (v["ms"] * 1e6) if v["ms"] > 0 else None}
                              for k, v in sorted(prof.items(), key=lambda kv: -kv[1]["ms"])},
            "how": f"prefill of the batch at this line's K_l into a kept-token cache, then {n} decode steps "
                   "(one token per sequence) replayed from one CUDA graph, CUDA events per step; "
                   "kernels_eager: one more step run eagerly with events around every launch"}


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


# ----------------------------------------------------------------------------- the oracle on the host
def _f64(t):
    return t.float().cpu().numpy().astype(np.float64)


def layer_order(L: int):
    """Layers in an order that spreads any prefix over the depth (a stride
    coprime with L)."""
    stride = max(1, round(L * 0.618))
    while math.gcd(stride, L) != 1:
        stride += 1
    return [(j * stride) % L for j in range(L)]


def oracle_sample(shape, K, ids_host, layer_weights, budget_s, max_evals=None):
    """Times the oracle's sparse layer (Sec. 3.4) on (sequence, layer) pairs of
    the workload: sequences in turn, layers spread over the depth, until
    budget_s seconds of oracle time (or max_evals pairs). layer_weights(l)
    returns layer l's weights as fp64 NumPy arrays (drawn outside the timing);
    the layer input is the sequence's embedding. Returns (seconds per pair,
    pairs, sequences touched)."""
    from oracle import adadsf_oracle as O
    p = O.params_of(shape)
    B = ids_host.shape[0]
    order = layer_order(shape.n_layers)
    spent, times, seqs = 0.0, [], set()
    j = 0
    while spent < budget_s and (max_evals is None or j < max_evals):
        b = j % B
        l = order[j % len(order)]
        W = layer_weights(l)
        x = _f64(S.round_to_torch(S.bench_embed_rows(shape, WEIGHT_SEED, ids_host[b:b + 1]), shape.dtype))
        t0 = time.time()
        O.sparse_layer_forward(x, W, p, K[l])
        dt = time.time() - t0
        times.append(dt)
        spent += dt
        seqs.add(b)
        j += 1
    return float(np.mean(times)), len(times), len(seqs)


def cpu_baseline(model, shape, K, ids, budget_s=20.0):
    """The fp64 oracle as it stands on the host cores, on a bounded sample of the
    same workload (the GPU arm's weights and kept counts), extrapolated to all
    layers."""
    T = ids.shape[1]
    L = shape.n_layers
    cache = {}

    def weights(l):
        if l not in cache:
            cache.clear()
            cache[l] = {k: _f64(v) for k, v in model.layers[l].items()}
        return cache[l]

    per, n, seqs = oracle_sample(shape, K, ids.cpu(), weights, budget_s)
    return {"value": T / (per * L), "unit": "tokens/s", "cores": host_threads(), "kind": "oracle",
            "sample": f"{n} (sequence, layer) evaluations of the oracle's sparse layer over {seqs} of "
                      f"{ids.shape[0]} sequences x {T} tokens at this line's K_l, layers spread over the depth, "
                      f"{per:.2f} s each on average; rate extrapolated to all {L} layers (fp64 NumPy, BLAS threads = "
                      f"host cores)"}


# ----------------------------------------------------------------------------- reference arm
def reference_calibration(shape, wl, layer_weights, flop_budget=2e12):
    """Eq. 4 statistics of the dense model with the oracle on a bounded prefix
    of the calibration batch (the first n tokens of its first sequences, n
    sized to about flop_budget fp64 flops), then Eqs. 5-8 at the workload's
    full T. Returns (s, n_sequences, n_tokens)."""
    from oracle import adadsf_oracle as O
    p = O.params_of(shape)
    L = shape.n_layers
    per_tok = dense_flops_per_layer(shape, 1, 1) - 4.0 * shape.n_heads * shape.head_dim
    n_tok = int(max(128, min(wl.calib[0] * wl.calib[1], flop_budget / (L * per_tok))))
    n_seq = max(1, min(wl.calib[0], n_tok // wl.calib[1]))
    n_len = min(wl.calib[1], n_tok)
    ids = S.counter_ids(CALIB_SEED, *wl.calib, shape.vocab)[:n_seq, :n_len]
    x = _f64(S.round_to_torch(S.bench_embed_rows(shape, WEIGHT_SEED, ids), shape.dtype))
    s = []
    for l in range(L):
        W = layer_weights(l)
        x_new, _, _ = O.sparse_layer_forward(x, W, p, n_len)
        s.append(O.similarity(O.cos_sim_stat(x, x_new)))
        x = x_new
    return np.array(s), n_seq, n_len


def run_reference(args, rank, world):
    """The fp64 CPU oracle timed on the host cores: each step is one bounded
    sample of the workload -- the oracle's sparse layer on one sequence of the
    batch, layers spread over the depth -- and the rate is extrapolated to the
    whole model. The kept counts come from the oracle's own Eq. 4 statistics
    on a bounded prefix of the calibration batch."""
    if rank != 0:
        return
    from oracle import adadsf_oracle as O
    wl = S.WORKLOADS[args.workload]
    shape, B, T = wl.shape, wl.B, wl.T
    L = shape.n_layers
    t_target = retention_of(args, wl)
    # inputs: the same counter-based draws as the GPU arm; drawn with PyTorch
    # on the GPU when one is present (seconds instead of minutes), the
    # oracle's arithmetic always on the host
    gen = "cuda" if torch.cuda.is_available() else "cpu"
    td = torch.bfloat16 if shape.dtype == "bf16" else torch.float32

    def layer_weights(l):
        return {k: _f64(v.to(td)) for k, v in S.bench_layer_weights(shape, WEIGHT_SEED, l, gen).items()}

    c0 = time.time()
    s, n_seq, n_len = reference_calibration(shape, wl, layer_weights)
    r, _ = O.allocate_ratios(s, t_target, TAU, BETA)
    K = O.kept_counts(r, T).tolist()
    calib_s = time.time() - c0
    ids = S.counter_ids(rank_seed(EVAL_SEED, 0), B, T, shape.vocab)
    p = O.params_of(shape)
    order = layer_order(L)
    t = []
    for i in range(args.warmup + args.steps):
        j = i - args.warmup if i >= args.warmup else args.steps + i     # warm-up pairs after the timed ones
        b, l = j % B, order[j % L]
        W = layer_weights(l)
        x = _f64(S.round_to_torch(S.bench_embed_rows(shape, WEIGHT_SEED, ids[b:b + 1]), shape.dtype))
        t0 = time.time()
        O.sparse_layer_forward(x, W, p, K[l])
        if i >= args.warmup:
            t.append(time.time() - t0)
    sec = float(np.mean(t))
    v = T / (sec * L)
    sample = (f"each step: the oracle's sparse layer on one sequence x {T} tokens (layer input = the sequence's "
              f"embedding), layers spread over the depth ({len(set(order[j % L] for j in range(args.steps)))} "
              f"distinct layers over {args.steps} steps); rate extrapolated to all {L} layers "
              f"(tokens/s = T / (L x mean step time)); K_l from the oracle's Eq. 4 statistics on "
              f"{n_seq} x {n_len} calibration tokens ({calib_s:.0f} s)")
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": v, "unit": "tokens/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": sec * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "extrapolated": True,
        "config": shared_config(wl, t_target, world),
        "retention_plan": {"K_per_layer": K, "retention_mean": float(np.mean(K)) / T,
                           "similarity": [float(x) for x in s],
                           "calibration": f"oracle dense forward with Eq. 4 statistics over {n_seq} x {n_len} "
                                          f"tokens of the calibration batch"},
        "cpu_baseline": {"value": v, "unit": "tokens/s", "cores": host_threads(), "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": v, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }), flush=True)


# ----------------------------------------------------------------------------- main
def main():
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--workload", choices=("c2", "c3", "c4", "c5"), default="c5")
    ap.add_argument("--retention", type=float, default=None)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-budget", type=float, default=20.0)
    ap.add_argument("--spin-up", type=float, default=1.5, help="seconds of untimed GPU work before measuring")
    ap.add_argument("--decode-steps", type=int, default=32, help="decode steps timed after a prefill (0: none)")
    ap.add_argument("--folded-norms", action="store_true",
                    help="fold the norm gains into the projections (ADADSF_FLAG_FOLDED_NORMS; exact for the "
                         "benchmark models, whose gains are 1): a decode step's post-attention RMSNorm then "
                         "runs inside its projections")
    ap.add_argument("--gathered-qkv", action="store_true",
                    help="with folded norms, the first RMSNorm inside the QKV projection, whose loads gather the "
                         "kept rows of x (ADADSF_FLAG_GATHERED_QKV)")
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
