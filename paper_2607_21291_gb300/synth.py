"""Seeded synthetic inputs and workload shapes for the AdaDSF depth-sparse forward.

This module is shared by the CUDA path's tests, the benchmark and the oracle's
tests. It holds no arithmetic of the method: only shapes (the GPT-NeoX / Qwen2.5
backbones of the paper's Sec. 4.1, "Models") and seeded random draws.

Recipe (the same for every workload):
  * hidden states          x ~ N(0, 1)
  * linear weights/biases  ~ N(0, 0.02)             (router included)
  * norm gains             1 + N(0, gain_std)       (gain_std = 0 for benchmarks)
  * norm biases            N(0, gain_std)
  * token ids              uniform over [0, vocab)
All draws use NumPy's PCG64 stream keyed by (seed, layer, tensor name), so every
tensor is reproducible on its own and independent of draw order.
"""
from __future__ import annotations

import dataclasses
import zlib

import numpy as np

NEOX = 0   # parallel residual, LayerNorm, GELU MLP, biases on every linear
QWEN = 1   # sequential residual, RMSNorm, SwiGLU MLP, bias on QKV only


@dataclasses.dataclass(frozen=True)
class Shape:
    """Backbone shape of one decoder stack plus the router width."""
    name: str
    arch: int
    d: int
    n_heads: int
    n_kv_heads: int
    head_dim: int
    ffn: int
    n_layers: int
    vocab: int
    rotary_dim: int
    rope_theta: float
    norm_eps: float
    dtype: str            # "f32" or "bf16": storage type of weights and activations
    router_hidden: int = 64

    @property
    def q_dim(self) -> int:
        return self.n_heads * self.head_dim

    @property
    def kv_dim(self) -> int:
        return self.n_kv_heads * self.head_dim

    @property
    def qkv_dim(self) -> int:
        return self.q_dim + 2 * self.kv_dim

    def replace(self, **kw) -> "Shape":
        return dataclasses.replace(self, **kw)


@dataclasses.dataclass(frozen=True)
class Workload:
    """A batch shape and retention targets on a backbone."""
    name: str
    shape: Shape
    B: int
    T: int
    retention: tuple        # mean retention t values (Eq. 8) for the sweep
    calib: tuple            # (B, T) of the calibration batch for Eq. 4


PYTHIA_70M = Shape("pythia-70m", NEOX, 512, 8, 8, 64, 2048, 6, 50304, 16, 1e4, 1e-5, "f32")
PYTHIA_160M = Shape("pythia-160m", NEOX, 768, 12, 12, 64, 3072, 12, 50304, 16, 1e4, 1e-5, "bf16")
PYTHIA_1_4B = Shape("pythia-1.4b", NEOX, 2048, 16, 16, 128, 8192, 24, 50304, 32, 1e4, 1e-5, "bf16")
QWEN25_1_5B = Shape("qwen2.5-1.5b", QWEN, 1536, 12, 2, 128, 8960, 28, 151936, 128, 1e6, 1e-6, "bf16")
QWEN25_7B = Shape("qwen2.5-7b", QWEN, 3584, 28, 4, 128, 18944, 28, 152064, 128, 1e6, 1e-6, "bf16")

WORKLOADS = {
    # one GPT-NeoX layer, fp32, B=1 T=128, r=0.5
    "c1": Workload("pythia-70m-layer-f32-B1-T128", PYTHIA_70M.replace(n_layers=1), 1, 128, (0.5,), (1, 128)),
    # full 12-layer Pythia-160M shape, bf16, B=4 T=512, mean retention 0.5
    "c2": Workload("pythia-160m-bf16-B4-T512", PYTHIA_160M, 4, 512, (0.5,), (4, 512)),
    "c3": Workload("pythia-1.4b-bf16-B8-T2048", PYTHIA_1_4B, 8, 2048, (0.75, 0.5, 0.25), (8, 2048)),
    "c4": Workload("qwen2.5-1.5b-bf16-B8-T2048", QWEN25_1_5B, 8, 2048, (0.5,), (8, 2048)),
    "c5": Workload("qwen2.5-7b-bf16-B16-T4096", QWEN25_7B, 16, 4096, (1.0, 0.75, 0.5, 0.25), (16, 4096)),
}


def _rng(seed: int, *key) -> np.random.Generator:
    tag = zlib.crc32(repr(key).encode())
    return np.random.Generator(np.random.PCG64([seed, tag]))


def normal(seed: int, key: tuple, shape, std: float = 1.0, mean: float = 0.0) -> np.ndarray:
    """float32 array of N(mean, std^2) draws from the stream named by (seed, key)."""
    a = _rng(seed, *key).standard_normal(size=shape, dtype=np.float32)
    if std != 1.0:
        a *= np.float32(std)
    if mean != 0.0:
        a += np.float32(mean)
    return a


def layer_weight_shapes(s: Shape) -> dict:
    """Tensor name -> shape for one decoder layer (weights are [out, in])."""
    shapes = {
        "router_w1": (s.router_hidden, s.d), "router_b1": (s.router_hidden,),
        "router_w2": (s.router_hidden,), "router_b2": (1,),
        "ln1_w": (s.d,), "ln2_w": (s.d,),
        "w_qkv": (s.qkv_dim, s.d), "b_qkv": (s.qkv_dim,),
        "w_o": (s.d, s.q_dim),
        "w_up": (s.ffn, s.d), "w_down": (s.d, s.ffn),
    }
    if s.arch == NEOX:
        shapes.update({"ln1_b": (s.d,), "ln2_b": (s.d,), "b_o": (s.d,),
                       "b_up": (s.ffn,), "b_down": (s.d,)})
    else:
        shapes.update({"w_gate": (s.ffn, s.d)})
    return shapes


def layer_weights(s: Shape, seed: int, layer: int, gain_std: float = 0.1,
                  std: float = 0.02) -> dict:
    """Host float32 weights of one layer (not yet rounded to the storage dtype)."""
    out = {}
    for name, shp in layer_weight_shapes(s).items():
        if name in ("ln1_w", "ln2_w"):
            out[name] = normal(seed, (layer, name), shp, gain_std, 1.0)
        elif name in ("ln1_b", "ln2_b"):
            out[name] = normal(seed, (layer, name), shp, gain_std)
        else:
            out[name] = normal(seed, (layer, name), shp, std)
    return out


def model_extra_weights(s: Shape, seed: int, gain_std: float = 0.1, std: float = 0.02) -> dict:
    """Embedding table and final norm."""
    out = {"embed": normal(seed, ("embed",), (s.vocab, s.d), std),
           "final_w": normal(seed, ("final_w",), (s.d,), gain_std, 1.0)}
    if s.arch == NEOX:
        out["final_b"] = normal(seed, ("final_b",), (s.d,), gain_std)
    return out


def hidden(seed: int, B: int, T: int, d: int, key: str = "x") -> np.ndarray:
    return normal(seed, ("hidden", key), (B, T, d))


def token_ids(seed: int, B: int, T: int, vocab: int) -> np.ndarray:
    return _rng(seed, "ids").integers(0, vocab, size=(B, T), dtype=np.int64).astype(np.int32)


def round_to(a: np.ndarray, dtype: str) -> np.ndarray:
    """Round a float32 array to the storage dtype and return it as float32
    (bf16: round to nearest even on the top 16 bits)."""
    a = np.ascontiguousarray(a, dtype=np.float32)
    if dtype == "f32":
        return a.copy()
    u = a.view(np.uint32)
    # In place on one uint32 array: u + 0x7FFF + (bit 16 of u), low half
    # cleared. Finite inputs cannot wrap (largest 0xFF7FFFFF + 0x8000); NaNs
    # may, and are replaced below.
    r = np.asarray((u >> 16) & np.uint32(1))   # an array also for 0-d input
    r += np.uint32(0x7FFF)
    r += u
    r &= np.uint32(0xFFFF0000)
    out = r.view(np.float32)
    nan = np.isnan(a)
    if nan.any():
        out[nan] = np.float32(np.nan)
    return out
