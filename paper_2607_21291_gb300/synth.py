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
tensor is reproducible on its own and independent of draw order. The
benchmark-size models use the counter-based draws at the end of this module
(same recipe, norm gains 1 and biases 0).
"""
from __future__ import annotations

import dataclasses
import math
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


# ----------------------------------------------------------------------------
# Counter-based draws (benchmark-size models)
#
# The full-size benchmark models hold billions of parameters: drawing them with
# the NumPy streams above on the host would take minutes. These draws use a
# counter-based generator instead -- element i of the tensor named by
# (seed, key) is a pure function of (seed, key, i) -- written with PyTorch
# integer and float64 operations, so the same tensor comes out on the GPU (in
# milliseconds) and on the host (for any subset of its elements, such as the
# embedding rows of a few token ids), apart from float64 ulps of log / cos that
# vanish in the final float32 / bf16 rounding.
#
# Generator: SplitMix64 (G. Steele, D. Lea, C. Flood, "Fast splittable
# pseudorandom number generators", OOPSLA 2014), the 64-bit finaliser applied
# to stream_base + (i + 1) * 0x9E3779B97F4A7C15. Normal draws take two 24-bit
# uniforms from one 64-bit output and apply the Box-Muller transform in
# float64; token ids take the output modulo the vocabulary size.
# ----------------------------------------------------------------------------
_SM_GAMMA = 0x9E3779B97F4A7C15
_SM_MUL1 = 0xBF58476D1CE4E5B9
_SM_MUL2 = 0x94D049BB133111EB
_CHUNK = 1 << 24


def _i64(u: int) -> int:
    """Two's-complement int64 value of a 64-bit unsigned constant."""
    return u - (1 << 64) if u >= (1 << 63) else u


def _lsr(z, s: int):
    """Logical right shift of int64 tensor z by s bits."""
    import torch
    return torch.bitwise_and(torch.bitwise_right_shift(z, s), (1 << (64 - s)) - 1)


def _splitmix64(ctr, base: int):
    """SplitMix64 outputs for int64 counters ctr (wrapping int64 arithmetic)."""
    z = ctr * _i64(_SM_GAMMA) + _i64(base)
    z = _xor(z, _lsr(z, 30)) * _i64(_SM_MUL1)
    z = _xor(z, _lsr(z, 27)) * _i64(_SM_MUL2)
    return _xor(z, _lsr(z, 31))


def _xor(a, b):
    import torch
    return torch.bitwise_xor(a, b)


def _stream_base(seed: int, key: tuple) -> int:
    h = zlib.crc32(repr((int(seed),) + tuple(key)).encode())
    return ((int(seed) & 0xFFFFFFFF) << 32 | h) & 0xFFFFFFFFFFFFFFFF


def counter_normal_at(seed: int, key: tuple, index, std: float = 1.0, mean: float = 0.0):
    """float32 tensor of N(mean, std^2) draws at the flat element positions
    `index` (int64 tensor, on the device the result should live on) of the
    tensor named by (seed, key)."""
    import torch
    base = _stream_base(seed, key)
    out = torch.empty(index.shape, dtype=torch.float32, device=index.device)
    flat_i, flat_o = index.reshape(-1), out.view(-1)
    for s in range(0, flat_i.numel(), _CHUNK):
        z = _splitmix64(flat_i[s:s + _CHUNK] + 1, base)
        u1 = (_lsr(z, 40).double() + 0.5) * (1.0 / (1 << 24))
        u2 = (torch.bitwise_and(_lsr(z, 16), 0xFFFFFF).double() + 0.5) * (1.0 / (1 << 24))
        n = torch.sqrt(-2.0 * torch.log(u1)) * torch.cos((2.0 * math.pi) * u2)
        flat_o[s:s + _CHUNK] = (n * std + mean).float()
    return out


def counter_normal(seed: int, key: tuple, shape, std: float = 1.0, mean: float = 0.0, device="cpu"):
    """The whole tensor of counter_normal_at, shaped `shape`."""
    import torch
    n = int(np.prod(shape)) if len(shape) else 1
    out = torch.empty(n, dtype=torch.float32, device=device)
    for s in range(0, n, _CHUNK):
        e = min(n, s + _CHUNK)
        out[s:e] = counter_normal_at(seed, key, torch.arange(s, e, dtype=torch.int64, device=device), std, mean)
    return out.view(*shape)


def counter_ids(seed: int, B: int, T: int, vocab: int, device="cpu"):
    """int32 token ids (B, T), uniform over [0, vocab) (modulo bias < vocab / 2^63)."""
    import torch
    z = _splitmix64(torch.arange(B * T, dtype=torch.int64, device=device) + 1, _stream_base(seed, ("ids",)))
    return torch.remainder(_lsr(z, 1), vocab).to(torch.int32).view(B, T)


def bench_layer_weights(s: Shape, seed: int, layer: int, device="cpu") -> dict:
    """float32 torch tensors of one layer in the benchmark recipe (counter-based
    N(0, std 0.02) weights and biases, norm gains 1, norm biases 0)."""
    import torch
    out = {}
    for name, shp in layer_weight_shapes(s).items():
        if name in ("ln1_w", "ln2_w"):
            out[name] = torch.ones(shp, dtype=torch.float32, device=device)
        elif name in ("ln1_b", "ln2_b"):
            out[name] = torch.zeros(shp, dtype=torch.float32, device=device)
        else:
            out[name] = counter_normal(seed, ("layer", layer, name), shp, 0.02, device=device)
    return out


def bench_embed(s: Shape, seed: int, device="cpu"):
    """The whole embedding table [vocab, d] of the benchmark recipe (float32)."""
    return counter_normal(seed, ("embed",), (s.vocab, s.d), 0.02, device=device)


def bench_embed_rows(s: Shape, seed: int, ids):
    """Rows ids (int tensor, any shape) of bench_embed, shape ids.shape + (d,),
    drawn without building the table."""
    import torch
    flat = ids.reshape(-1).to(torch.int64)
    cols = torch.arange(s.d, dtype=torch.int64, device=flat.device)
    return counter_normal_at(seed, ("embed",), flat[:, None] * s.d + cols[None, :], 0.02).view(
        *ids.shape, s.d)


def round_to_torch(t, dtype: str):
    """float32 copy of tensor t rounded to the storage dtype (bf16: round to
    nearest even, as round_to)."""
    import torch
    return t.to(torch.bfloat16).float() if dtype == "bf16" else t.float().clone()
