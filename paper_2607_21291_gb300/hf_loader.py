"""Weights of pre-trained GPT-NeoX and Qwen2 checkpoints in the Hugging Face
layout (config.json + safetensors), mapped onto the library's layer layout.

AdaDSF adapts a pre-trained decoder (Sec. 3.2: the backbone keeps its
weights; only the routers are new), so a user starts from a released
checkpoint. This module reads such a checkpoint without any third-party
package: the safetensors container is an 8-byte little-endian header length,
a JSON header of {name: {dtype, shape, data_offsets}} and the raw tensor bytes
(read through a memory map, one tensor at a time).

Name and layout mapping (library layout: weights [out, in], the fused QKV
weight stacking all query rows, then all key rows, then all value rows):

GPT-NeoX (``model_type == "gpt_neox"``, parallel residual):
  gpt_neox.embed_in.weight                      -> embed
  layers.{l}.input_layernorm.{weight,bias}      -> ln1_w, ln1_b
  layers.{l}.post_attention_layernorm.{w,b}     -> ln2_w, ln2_b
  layers.{l}.attention.query_key_value.{w,b}    -> w_qkv, b_qkv, rows regrouped:
      the checkpoint interleaves them per head as [head][q | k | v][head_dim]
  layers.{l}.attention.dense.{weight,bias}      -> w_o, b_o
  layers.{l}.mlp.dense_h_to_4h.{weight,bias}    -> w_up, b_up
  layers.{l}.mlp.dense_4h_to_h.{weight,bias}    -> w_down, b_down
  gpt_neox.final_layer_norm.{weight,bias}       -> final_w, final_b
Qwen2 (``model_type == "qwen2"``):
  model.embed_tokens.weight                     -> embed
  layers.{l}.input_layernorm.weight             -> ln1_w
  layers.{l}.post_attention_layernorm.weight    -> ln2_w
  layers.{l}.self_attn.{q,k,v}_proj.{w,b}       -> w_qkv, b_qkv (stacked q, k, v)
  layers.{l}.self_attn.o_proj.weight            -> w_o
  layers.{l}.mlp.{gate,up,down}_proj.weight     -> w_gate, w_up, w_down
  model.norm.weight                             -> final_w

Routers are not part of these checkpoints. ``router`` may name a safetensors
file holding ``router.{l}.w1 [h, d]``, ``router.{l}.b1 [h]``,
``router.{l}.w2 [h]``, ``router.{l}.b2 [1]`` per layer; without it they are
drawn N(0, 0.02) from ``router_seed`` (untrained: the kept sets are then
score-driven but arbitrary).
"""
from __future__ import annotations

import json
import mmap
import os
import struct
from typing import Dict, Optional

import numpy as np

from . import synth as S

_DTYPES = {"F32": (np.float32, 4), "F16": (np.float16, 2), "BF16": (np.uint16, 2), "F64": (np.float64, 8)}


class SafeTensors:
    """Read-only view of one .safetensors file; get(name) returns float32."""

    def __init__(self, path: str):
        self.path = path
        self._f = open(path, "rb")
        n = struct.unpack("<Q", self._f.read(8))[0]
        if n <= 0 or n > (1 << 27):
            raise ValueError(f"{path}: header length {n} is not plausible")
        hdr = json.loads(self._f.read(n).decode("utf-8"))
        hdr.pop("__metadata__", None)
        self.header = hdr
        self._base = 8 + n
        self._mm = mmap.mmap(self._f.fileno(), 0, access=mmap.ACCESS_READ)

    def names(self):
        return list(self.header)

    def get(self, name: str) -> np.ndarray:
        info = self.header[name]
        if info["dtype"] not in _DTYPES:
            raise ValueError(f"{self.path}: {name} has unsupported dtype {info['dtype']}")
        npt, size = _DTYPES[info["dtype"]]
        lo, hi = info["data_offsets"]
        shape = tuple(info["shape"])
        count = int(np.prod(shape)) if shape else 1
        if hi - lo != count * size:
            raise ValueError(f"{self.path}: {name} has {hi - lo} bytes for shape {shape}")
        raw = np.frombuffer(self._mm, dtype=npt, count=count, offset=self._base + lo)
        if info["dtype"] == "BF16":
            # bf16 is the top half of an fp32 bit pattern
            out = (raw.astype(np.uint32) << 16).view(np.float32)
        else:
            out = raw.astype(np.float32)
        return out.reshape(shape)

    def close(self):
        self._mm.close()
        self._f.close()


class Checkpoint:
    """All tensors of a checkpoint directory (single file or sharded with
    model.safetensors.index.json), or of one .safetensors file."""

    def __init__(self, path: str):
        self.dir = path if os.path.isdir(path) else os.path.dirname(path)
        files = []
        if os.path.isdir(path):
            idx = os.path.join(path, "model.safetensors.index.json")
            if os.path.exists(idx):
                with open(idx) as f:
                    files = sorted(set(json.load(f)["weight_map"].values()))
            else:
                files = sorted(f for f in os.listdir(path) if f.endswith(".safetensors"))
            files = [os.path.join(path, f) for f in files]
        else:
            files = [path]
        if not files:
            raise FileNotFoundError(f"no .safetensors file under {path}")
        self._readers = [SafeTensors(f) for f in files]
        self._where = {}
        for r in self._readers:
            for n in r.names():
                self._where[n] = r

    def has(self, name: str) -> bool:
        return name in self._where

    def get(self, name: str) -> np.ndarray:
        if name not in self._where:
            raise KeyError(f"checkpoint has no tensor {name}")
        return self._where[name].get(name)

    def close(self):
        for r in self._readers:
            r.close()


def shape_from_config(cfg: dict, dtype: str = "bf16", router_hidden: int = 64) -> S.Shape:
    """Backbone shape of a Hugging Face config dict."""
    mt = cfg.get("model_type")
    d, H = int(cfg["hidden_size"]), int(cfg["num_attention_heads"])
    hd = d // H
    if mt == "gpt_neox":
        if not cfg.get("use_parallel_residual", True):
            raise ValueError("GPT-NeoX with use_parallel_residual = false is not supported")
        if cfg.get("hidden_act", "gelu") != "gelu":
            raise ValueError(f"GPT-NeoX hidden_act {cfg.get('hidden_act')} is not supported (exact GELU only)")
        return S.Shape(cfg.get("_name_or_path", "gpt-neox") or "gpt-neox", S.NEOX, d, H, H, hd,
                       int(cfg["intermediate_size"]), int(cfg["num_hidden_layers"]), int(cfg["vocab_size"]),
                       int(hd * float(cfg.get("rotary_pct", 0.25))), float(cfg.get("rotary_emb_base", 10000)),
                       float(cfg.get("layer_norm_eps", 1e-5)), dtype, router_hidden)
    if mt == "qwen2":
        if cfg.get("rope_scaling"):
            raise ValueError("Qwen2 rope_scaling is not supported")
        if cfg.get("use_sliding_window", False):
            raise ValueError("Qwen2 sliding-window attention is not supported")
        if cfg.get("hidden_act", "silu") != "silu":
            raise ValueError(f"Qwen2 hidden_act {cfg.get('hidden_act')} is not supported")
        return S.Shape(cfg.get("_name_or_path", "qwen2") or "qwen2", S.QWEN, d, H,
                       int(cfg.get("num_key_value_heads", H)), hd, int(cfg["intermediate_size"]),
                       int(cfg["num_hidden_layers"]), int(cfg["vocab_size"]), hd,
                       float(cfg.get("rope_theta", 10000.0)), float(cfg.get("rms_norm_eps", 1e-6)), dtype,
                       router_hidden)
    raise ValueError(f"model_type {mt!r} is not supported (gpt_neox, qwen2)")


def _neox_qkv_rows(a: np.ndarray, H: int, hd: int) -> np.ndarray:
    """[head][q|k|v][hd](...) -> [q|k|v][head][hd](...) along the first axis."""
    rest = a.shape[1:]
    return a.reshape((H, 3, hd) + rest).swapaxes(0, 1).reshape((3 * H * hd,) + rest)


def layer_weights(ck: Checkpoint, shape: S.Shape, l: int) -> Dict[str, np.ndarray]:
    """Backbone weights of layer l in the library layout (float32 arrays)."""
    if shape.arch == S.NEOX:
        p = f"gpt_neox.layers.{l}."
        H, hd = shape.n_heads, shape.head_dim
        return {"ln1_w": ck.get(p + "input_layernorm.weight"), "ln1_b": ck.get(p + "input_layernorm.bias"),
                "ln2_w": ck.get(p + "post_attention_layernorm.weight"),
                "ln2_b": ck.get(p + "post_attention_layernorm.bias"),
                "w_qkv": _neox_qkv_rows(ck.get(p + "attention.query_key_value.weight"), H, hd),
                "b_qkv": _neox_qkv_rows(ck.get(p + "attention.query_key_value.bias"), H, hd),
                "w_o": ck.get(p + "attention.dense.weight"), "b_o": ck.get(p + "attention.dense.bias"),
                "w_up": ck.get(p + "mlp.dense_h_to_4h.weight"), "b_up": ck.get(p + "mlp.dense_h_to_4h.bias"),
                "w_down": ck.get(p + "mlp.dense_4h_to_h.weight"), "b_down": ck.get(p + "mlp.dense_4h_to_h.bias")}
    p = f"model.layers.{l}."
    qkv_w = [ck.get(p + f"self_attn.{n}_proj.weight") for n in "qkv"]
    qkv_b = [ck.get(p + f"self_attn.{n}_proj.bias") if ck.has(p + f"self_attn.{n}_proj.bias")
             else np.zeros(w.shape[0], np.float32) for n, w in zip("qkv", qkv_w)]
    return {"ln1_w": ck.get(p + "input_layernorm.weight"), "ln2_w": ck.get(p + "post_attention_layernorm.weight"),
            "w_qkv": np.concatenate(qkv_w, 0), "b_qkv": np.concatenate(qkv_b, 0),
            "w_o": ck.get(p + "self_attn.o_proj.weight"),
            "w_gate": ck.get(p + "mlp.gate_proj.weight"), "w_up": ck.get(p + "mlp.up_proj.weight"),
            "w_down": ck.get(p + "mlp.down_proj.weight")}


def extra_weights(ck: Checkpoint, shape: S.Shape) -> Dict[str, np.ndarray]:
    if shape.arch == S.NEOX:
        return {"embed": ck.get("gpt_neox.embed_in.weight"), "final_w": ck.get("gpt_neox.final_layer_norm.weight"),
                "final_b": ck.get("gpt_neox.final_layer_norm.bias")}
    return {"embed": ck.get("model.embed_tokens.weight"), "final_w": ck.get("model.norm.weight")}


def router_weights(shape: S.Shape, l: int, router: Optional[Checkpoint], seed: int) -> Dict[str, np.ndarray]:
    h = shape.router_hidden
    if router is not None:
        w = {"router_w1": router.get(f"router.{l}.w1"), "router_b1": router.get(f"router.{l}.b1"),
             "router_w2": router.get(f"router.{l}.w2"), "router_b2": router.get(f"router.{l}.b2")}
        want = {"router_w1": (h, shape.d), "router_b1": (h,), "router_w2": (h,), "router_b2": (1,)}
        for k, shp in want.items():
            if tuple(w[k].shape) != shp:
                raise ValueError(f"router.{l}: {k} has shape {w[k].shape}, expected {shp}")
        return w
    return {k: S.normal(seed, ("router", l, k), shp, 0.02)
            for k, shp in (("router_w1", (h, shape.d)), ("router_b1", (h,)), ("router_w2", (h,)),
                           ("router_b2", (1,)))}


def check_shapes(shape: S.Shape, w: Dict[str, np.ndarray], l: int):
    want = S.layer_weight_shapes(shape)
    for k, shp in want.items():
        if k in w and tuple(w[k].shape) != tuple(shp):
            raise ValueError(f"layer {l}: {k} has shape {tuple(w[k].shape)}, expected {tuple(shp)}")


def load(path: str, dtype: str = "bf16", router: Optional[str] = None, router_seed: int = 0,
         device=None):
    """(shape, layers, extra) of the checkpoint at `path`: per-layer dicts and
    the embedding / final norm in the library layout, as float32 NumPy arrays
    (device=None) or as torch tensors of the storage dtype on `device`."""
    cfg_dir = path if os.path.isdir(path) else os.path.dirname(path)
    with open(os.path.join(cfg_dir, "config.json")) as f:
        shape = shape_from_config(json.load(f), dtype)
    ck = Checkpoint(path)
    rk = Checkpoint(router) if router else None
    try:
        layers = []
        for l in range(shape.n_layers):
            w = layer_weights(ck, shape, l)
            w.update(router_weights(shape, l, rk, router_seed))
            check_shapes(shape, w, l)
            layers.append(_place(w, dtype, device))
        extra = extra_weights(ck, shape)
        if tuple(extra["embed"].shape) != (shape.vocab, shape.d):
            raise ValueError(f"embedding has shape {extra['embed'].shape}, expected {(shape.vocab, shape.d)}")
        extra = _place(extra, dtype, device)
    finally:
        ck.close()
        if rk is not None:
            rk.close()
    return shape, layers, extra


def _place(w: Dict[str, np.ndarray], dtype: str, device):
    if device is None:
        return {k: np.ascontiguousarray(v, dtype=np.float32) for k, v in w.items()}
    import torch
    td = torch.bfloat16 if dtype == "bf16" else torch.float32
    return {k: torch.from_numpy(np.ascontiguousarray(v, dtype=np.float32)).to(device=device, dtype=td)
            for k, v in w.items()}


def device_model(path: str, dtype: str = "bf16", router: Optional[str] = None, router_seed: int = 0,
                 device="cuda"):
    """The checkpoint as an adadsf.DeviceModel ready for adadsf_sparse_model_forward."""
    from . import adadsf as A
    shape, layers, extra = load(path, dtype, router, router_seed, device)
    return shape, A.DeviceModel(A.make_cfg(shape), layers, extra)
