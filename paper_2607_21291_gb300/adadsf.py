"""Python binding of the C ABI in include/adadsf.h (libadadsf.so).

Argument marshalling only: every step of the depth-sparse forward runs in the
library's CUDA kernels. PyTorch provides device memory and streams. The
functions carry the C names; tensors replace (pointer, size) pairs.

The library is loaded from this package directory; if it is missing every call
raises (there is no fallback path)."""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Sequence

import numpy as np
import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libadadsf.so")

OK, ERR_INVALID_ARG, ERR_UNSUPPORTED, ERR_CUDA, ERR_WORKSPACE_TOO_SMALL, ERR_DEVICE_TIMEOUT = range(6)
F32, BF16 = 0, 1
ARCH_NEOX, ARCH_QWEN = 0, 1
STATS_TOKEN, STATS_FLAT = 0, 1
LINEAR_SPLIT_WS_BYTES = 256 + 160 * 128 * 256 * 4   # ADADSF_LINEAR_SPLIT_WS_BYTES
ALLOC_RAW, ALLOC_ROUND = 1, 2
FLAG_GATE_SIGMOID = 1
FLAG_FOLDED_NORMS = 2
FLAG_GATHERED_QKV = 4

TORCH_DTYPE = {F32: torch.float32, BF16: torch.bfloat16}
DTYPE_CODE = {torch.float32: F32, torch.bfloat16: BF16}

LAYER_FIELDS = ("router_w1", "router_b1", "router_w2", "router_b2", "ln1_w", "ln1_b", "ln2_w",
                "ln2_b", "w_qkv", "b_qkv", "w_o", "b_o", "w_up", "b_up", "w_gate", "w_down", "b_down")


class ModelCfg(ctypes.Structure):
    _fields_ = [("d", ctypes.c_int32), ("n_heads", ctypes.c_int32), ("n_kv_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("ffn", ctypes.c_int32), ("n_layers", ctypes.c_int32),
                ("vocab", ctypes.c_int32), ("router_hidden", ctypes.c_int32), ("arch", ctypes.c_int32),
                ("rotary_dim", ctypes.c_int32), ("rope_theta", ctypes.c_float),
                ("norm_eps", ctypes.c_float), ("dtype", ctypes.c_int32), ("flags", ctypes.c_int32)]


class LayerWeights(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in LAYER_FIELDS]


class ModelWeights(ctypes.Structure):
    _fields_ = [("embed", ctypes.c_void_p), ("final_w", ctypes.c_void_p),
                ("final_b", ctypes.c_void_p), ("layers", ctypes.POINTER(LayerWeights))]


class LaunchRecord(ctypes.Structure):
    _fields_ = [("kind", ctypes.c_int32), ("dense", ctypes.c_int32), ("ms", ctypes.c_double),
                ("flops", ctypes.c_double), ("bytes", ctypes.c_double)]


class AdadsfError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"adadsf status {status}: {msg}")
        self.status = status


_lib = None


def lib() -> ctypes.CDLL:
    """The loaded libadadsf.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with "
                               "`python -c 'import __graft_entry__ as g; g.build()'`")
        L = ctypes.CDLL(LIB_PATH)
        vp, i32, i64, sz, f64, u32 = (ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_size_t,
                                      ctypes.c_double, ctypes.c_uint)
        pcfg, plw, pmw = ctypes.POINTER(ModelCfg), ctypes.POINTER(LayerWeights), ctypes.POINTER(ModelWeights)
        sig = {
            "adadsf_last_error": (ctypes.c_char_p, []),
            "adadsf_layer_workspace_size": (sz, [pcfg, i32, i32, i32]),
            "adadsf_model_workspace_size": (sz, [pcfg, i32, i32, vp, i32]),
            "adadsf_stats_workspace_size": (sz, [i64]),
            "adadsf_layer_stats": (i32, [vp, vp, i64, i32, i32, i32, vp, vp, sz, vp]),
            "adadsf_layer_stats_noalloc": (i32, [vp, vp, i64, i32, i32, i32, vp, vp]),
            "adadsf_similarity": (i32, [vp, i32, i32, vp]),
            "adadsf_normalized_flops": (i32, [pcfg, i32, vp, vp]),
            "adadsf_fold_norms": (i32, [pcfg, plw, vp]),
            "adadsf_align_workspace_size": (sz, [i64, i32]),
            "adadsf_align_hidden": (i32, [vp, vp, i64, i32, i32, vp, vp, vp, sz, vp]),
            "adadsf_align_output": (i32, [vp, vp, vp, i64, i32, i32, i32, vp, vp, sz, vp]),
            "adadsf_router_backward_workspace_size": (sz, [pcfg, i64]),
            "adadsf_router_backward": (i32, [pcfg, plw, vp, vp, vp, i64, vp, vp, vp, sz, vp]),
            "adadsf_alloc_ratios": (i32, [vp, i32, f64, f64, f64, i32, u32, vp, vp]),
            "adadsf_router_scores": (i32, [pcfg, plw, vp, i64, vp, vp, sz, vp]),
            "adadsf_topk_select": (i32, [vp, i32, i32, i32, vp, vp, vp]),
            "adadsf_router_select_workspace_size": (sz, [pcfg, i32, i32]),
            "adadsf_router_select": (i32, [pcfg, plw, vp, i32, i32, i32, vp, vp, vp, vp, sz, vp]),
            "adadsf_linear": (i32, [vp, vp, vp, i64, i32, i32, i32, i32, vp, vp, sz, vp]),
            "adadsf_attention_workspace_size": (sz, [pcfg, i32, i32]),
            "adadsf_causal_attention": (i32, [pcfg, vp, i32, i32, vp, vp, sz, vp]),
            "adadsf_sparse_layer_forward": (i32, [pcfg, plw, vp, i32, i32, i32, vp, vp, vp, sz, vp]),
            "adadsf_sparse_model_forward": (i32, [pcfg, pmw, vp, i32, i32, vp, vp, vp, vp, vp, sz, vp]),
            "adadsf_kv_cache_size": (sz, [pcfg, i32, i32]),
            "adadsf_prefill": (i32, [pcfg, pmw, vp, i32, i32, vp, vp, vp, vp, sz, i32, vp, sz, vp]),
            "adadsf_decode_workspace_size": (sz, [pcfg, i32, i32]),
            "adadsf_decode_step": (i32, [pcfg, pmw, vp, i32, vp, vp, vp, sz, i32, vp, sz, vp]),
            "adadsf_sync_check": (i32, [vp, sz, vp]),
            "adadsf_selftest_bounded_wait": (i32, [vp, sz, i32, vp]),
            "adadsf_profile_begin": (i32, [i32]),
            "adadsf_profile_end": (i32, [ctypes.POINTER(LaunchRecord), i32]),
            "adadsf_kernel_name": (ctypes.c_char_p, [i32]),
        }
        for name, (res, args) in sig.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _lib = L
    return _lib


def _check(status: int):
    if status != OK:
        raise AdadsfError(status, lib().adadsf_last_error().decode())


def _p(t: Optional[torch.Tensor]):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _s(stream) -> ctypes.c_void_p:
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _dev(t: torch.Tensor, name: str):
    if not t.is_cuda or not t.is_contiguous():
        raise ValueError(f"{name} must be a contiguous CUDA tensor")


def workspace(nbytes: int, device=None) -> torch.Tensor:
    """Zero-initialised device workspace (its first 256 bytes are the error word)."""
    return torch.zeros(max(int(nbytes), 256), dtype=torch.uint8, device=device or "cuda")


# --------------------------------------------------------------------- config
def make_cfg(shape, flags: int = 0) -> ModelCfg:
    """ModelCfg from any object with the backbone fields (see synth.Shape);
    flags: FLAG_* bits (FLAG_GATE_SIGMOID: the score-gated variant)."""
    return ModelCfg(shape.d, shape.n_heads, shape.n_kv_heads, shape.head_dim, shape.ffn,
                    shape.n_layers, shape.vocab, shape.router_hidden, shape.arch, shape.rotary_dim,
                    shape.rope_theta, shape.norm_eps, BF16 if shape.dtype == "bf16" else F32, int(flags))


def layer_struct(w: dict) -> LayerWeights:
    """LayerWeights pointing at the device tensors of dict w (missing -> NULL)."""
    s = LayerWeights()
    for n in LAYER_FIELDS:
        t = w.get(n)
        if t is not None:
            _dev(t, n)
        setattr(s, n, None if t is None else t.data_ptr())
    return s


def to_device(host: dict, dtype: torch.dtype, device="cuda") -> dict:
    """Copies a dict of host arrays to device tensors of the storage dtype."""
    return {k: torch.from_numpy(np.ascontiguousarray(v)).to(device=device, dtype=dtype)
            for k, v in host.items()}


# --------------------------------------------------------------------- C entry points
def adadsf_last_error() -> str:
    return lib().adadsf_last_error().decode()


def adadsf_layer_workspace_size(cfg: ModelCfg, B: int, T: int, K: int) -> int:
    n = lib().adadsf_layer_workspace_size(ctypes.byref(cfg), B, T, K)
    if n == 0:
        raise AdadsfError(ERR_INVALID_ARG, adadsf_last_error())
    return n


def adadsf_model_workspace_size(cfg: ModelCfg, B: int, T: int, K: Sequence[int], with_stats=False) -> int:
    arr = (ctypes.c_int32 * len(K))(*[int(k) for k in K])
    n = lib().adadsf_model_workspace_size(ctypes.byref(cfg), B, T, ctypes.cast(arr, ctypes.c_void_p),
                                          1 if with_stats else 0)
    if n == 0:
        raise AdadsfError(ERR_INVALID_ARG, adadsf_last_error())
    return n


def adadsf_stats_workspace_size(n_rows: int) -> int:
    return lib().adadsf_stats_workspace_size(int(n_rows))


def adadsf_layer_stats(x_in: torch.Tensor, x_out: torch.Tensor, acc: torch.Tensor,
                       mode: int = STATS_TOKEN, ws: Optional[torch.Tensor] = None, stream=None):
    """Adds the Eq. 4 partial sums of (x_in, x_out) rows to the fp64 tensor acc."""
    _dev(x_in, "x_in"); _dev(x_out, "x_out"); _dev(acc, "acc")
    if acc.dtype != torch.float64:
        raise ValueError("acc must be float64")
    d = x_in.shape[-1]
    n = x_in.numel() // d
    if ws is None:
        ws = workspace(adadsf_stats_workspace_size(n), x_in.device)
    _check(lib().adadsf_layer_stats(_p(x_in), _p(x_out), n, d, DTYPE_CODE[x_in.dtype], mode,
                                    _p(acc), _p(ws), ws.numel(), _s(stream)))


def adadsf_layer_stats_noalloc(x_in: torch.Tensor, x_out: torch.Tensor, acc: torch.Tensor,
                               mode: int = STATS_TOKEN, stream=None):
    """adadsf_layer_stats without a workspace: the library keeps the partial
    sums in a fixed device array of its own (see include/adadsf.h for the
    set-up, sharing and size limits)."""
    _dev(x_in, "x_in"); _dev(x_out, "x_out"); _dev(acc, "acc")
    if acc.dtype != torch.float64:
        raise ValueError("acc must be float64")
    d = x_in.shape[-1]
    n = x_in.numel() // d
    _check(lib().adadsf_layer_stats_noalloc(_p(x_in), _p(x_out), n, d, DTYPE_CODE[x_in.dtype], mode,
                                            _p(acc), _s(stream)))


def adadsf_similarity(acc, mode: int = STATS_TOKEN) -> np.ndarray:
    """Host-only Eq. 4: s_l from the accumulated partial sums (any array-like,
    [L, 2] for TOKEN mode or [L, 3] for FLAT)."""
    if isinstance(acc, torch.Tensor):
        acc = acc.detach().cpu()
    a = np.ascontiguousarray(np.asarray(acc, dtype=np.float64).reshape(-1))
    width = 2 if mode == STATS_TOKEN else 3
    if a.size == 0 or a.size % width:
        raise ValueError(f"accumulator of {a.size} values is not a multiple of {width}")
    L = a.size // width
    s = np.zeros(L, dtype=np.float64)
    _check(lib().adadsf_similarity(a.ctypes.data_as(ctypes.c_void_p), L, int(mode),
                                   s.ctypes.data_as(ctypes.c_void_p)))
    return s


def adadsf_fold_norms(cfg: ModelCfg, w: dict, stream=None):
    """Folds the layer's norm parameters into its projections, modifying the
    device tensors of w in place (then run with FLAG_FOLDED_NORMS)."""
    lw = layer_struct(w)
    _check(lib().adadsf_fold_norms(ctypes.byref(cfg), ctypes.byref(lw), _s(stream)))


def adadsf_align_hidden(hs: torch.Tensor, hd: torch.Tensor, acc: torch.Tensor,
                        grad: Optional[torch.Tensor] = None, ws: Optional[torch.Tensor] = None, stream=None):
    """Eq. 9: adds {sum of per-row softmax distances, rows} to acc (fp64);
    grad (fp32, hs's shape) receives each row's gradient."""
    _dev(hs, "hs"); _dev(hd, "hd"); _dev(acc, "acc")
    d = hs.shape[-1]
    n = hs.numel() // d
    if ws is None:
        ws = workspace(lib().adadsf_align_workspace_size(n, 0), hs.device)
    _check(lib().adadsf_align_hidden(_p(hs), _p(hd), n, d, DTYPE_CODE[hs.dtype], _p(acc), _p(grad), _p(ws),
                                     ws.numel(), _s(stream)))


def adadsf_align_output(hs: torch.Tensor, hd: torch.Tensor, w_head: torch.Tensor, acc: torch.Tensor,
                        ws: Optional[torch.Tensor] = None, stream=None):
    """Eq. 10: adds {sum of per-row KL(P_dense || P_sparse), rows} to acc (fp64)."""
    _dev(hs, "hs"); _dev(hd, "hd"); _dev(w_head, "w_head"); _dev(acc, "acc")
    n_cls, d = w_head.shape
    n = hs.numel() // d
    if ws is None:
        ws = workspace(lib().adadsf_align_workspace_size(n, n_cls), hs.device)
    _check(lib().adadsf_align_output(_p(hs), _p(hd), _p(w_head), n, d, n_cls, DTYPE_CODE[hs.dtype], _p(acc),
                                     _p(ws), ws.numel(), _s(stream)))


def adadsf_router_backward(cfg: ModelCfg, w: dict, x: torch.Tensor, y_plain: torch.Tensor, rows: torch.Tensor,
                           grad_y: torch.Tensor, ws: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    """Router gradient through the score gate; returns fp32 [h*d + 2h + 1]
    (dW1, db1, dw2, db2)."""
    _dev(x, "x"); _dev(y_plain, "y_plain"); _dev(rows, "rows"); _dev(grad_y, "grad_y")
    n = rows.numel()
    h = cfg.router_hidden
    out = torch.empty(h * cfg.d + 2 * h + 1, dtype=torch.float32, device=x.device)
    if ws is None:
        ws = workspace(lib().adadsf_router_backward_workspace_size(ctypes.byref(cfg), n), x.device)
    lw = layer_struct(w)
    _check(lib().adadsf_router_backward(ctypes.byref(cfg), ctypes.byref(lw), _p(x), _p(y_plain), _p(rows), n,
                                        _p(grad_y), _p(out), _p(ws), ws.numel(), _s(stream)))
    return out


def adadsf_normalized_flops(cfg: ModelCfg, T: int, K: Sequence[int]) -> float:
    """Host-only: sparse-forward FLOPs over the dense model's (Sec. 4.1)."""
    arr = (ctypes.c_int32 * len(K))(*[int(k) for k in K])
    out = ctypes.c_double(0.0)
    _check(lib().adadsf_normalized_flops(ctypes.byref(cfg), int(T), ctypes.cast(arr, ctypes.c_void_p),
                                         ctypes.byref(out)))
    return out.value


def adadsf_alloc_ratios(s: Sequence[float], t: float, tau: float = 0.05, beta: float = 10.0,
                        T: int = 0, flags: int = 0):
    """Host-only Eqs. 5-8 (+ clamp) -> (r, K) as NumPy arrays."""
    s = np.ascontiguousarray(s, dtype=np.float64)
    L = s.shape[0]
    r = np.zeros(L, dtype=np.float64)
    K = np.zeros(L, dtype=np.int32)
    _check(lib().adadsf_alloc_ratios(s.ctypes.data_as(ctypes.c_void_p), L, float(t), float(tau),
                                     float(beta), int(T), int(flags), r.ctypes.data_as(ctypes.c_void_p),
                                     K.ctypes.data_as(ctypes.c_void_p)))
    return r, K


def adadsf_router_scores(cfg: ModelCfg, w: dict, x: torch.Tensor, scores: torch.Tensor,
                         ws: Optional[torch.Tensor] = None, stream=None):
    _dev(x, "x"); _dev(scores, "scores")
    n = x.numel() // cfg.d
    if ws is None:
        ws = workspace(256, x.device)
    lw = layer_struct(w)
    _check(lib().adadsf_router_scores(ctypes.byref(cfg), ctypes.byref(lw), _p(x), n, _p(scores),
                                      _p(ws), ws.numel(), _s(stream)))


def adadsf_topk_select(scores: torch.Tensor, K: int, idx: torch.Tensor,
                       rows: Optional[torch.Tensor] = None, stream=None):
    _dev(scores, "scores"); _dev(idx, "idx")
    B, T = scores.shape
    _check(lib().adadsf_topk_select(_p(scores), B, T, int(K), _p(idx), _p(rows), _s(stream)))


def adadsf_router_select_workspace_size(cfg: ModelCfg, B: int, T: int) -> int:
    return int(lib().adadsf_router_select_workspace_size(ctypes.byref(cfg), int(B), int(T)))


def adadsf_router_select(cfg: ModelCfg, w: dict, x: torch.Tensor, B: int, T: int, K: int,
                         scores: torch.Tensor, idx: torch.Tensor, rows: Optional[torch.Tensor] = None,
                         ws: Optional[torch.Tensor] = None, stream=None):
    _dev(x, "x"); _dev(scores, "scores"); _dev(idx, "idx")
    if ws is None:
        ws = workspace(adadsf_router_select_workspace_size(cfg, B, T), x.device)
    lw = layer_struct(w)
    _check(lib().adadsf_router_select(ctypes.byref(cfg), ctypes.byref(lw), _p(x), int(B), int(T), int(K),
                                      _p(scores), _p(idx), _p(rows), _p(ws), ws.numel(), _s(stream)))


def adadsf_linear(x: torch.Tensor, w: torch.Tensor, bias: Optional[torch.Tensor], out: torch.Tensor,
                  act: int = 0, ws: Optional[torch.Tensor] = None, stream=None):
    _dev(x, "x"); _dev(w, "w"); _dev(out, "out")
    n_out, k_in = w.shape
    M = x.numel() // k_in
    if ws is None:
        ws = workspace(256, x.device)
    _check(lib().adadsf_linear(_p(x), _p(w), _p(bias), M, n_out, k_in, DTYPE_CODE[x.dtype], act,
                               _p(out), _p(ws), ws.numel(), _s(stream)))


def adadsf_attention_workspace_size(cfg: ModelCfg, B: int, K: int) -> int:
    n = lib().adadsf_attention_workspace_size(ctypes.byref(cfg), B, K)
    if n == 0:
        raise AdadsfError(ERR_INVALID_ARG, adadsf_last_error())
    return n


def adadsf_causal_attention(cfg: ModelCfg, qkv: torch.Tensor, B: int, K: int, out: torch.Tensor,
                            ws: Optional[torch.Tensor] = None, stream=None):
    _dev(qkv, "qkv"); _dev(out, "out")
    if ws is None:
        ws = workspace(adadsf_attention_workspace_size(cfg, B, K), qkv.device)
    _check(lib().adadsf_causal_attention(ctypes.byref(cfg), _p(qkv), B, K, _p(out), _p(ws), ws.numel(),
                                         _s(stream)))


def adadsf_sparse_layer_forward(cfg: ModelCfg, w: dict, x: torch.Tensor, K: int,
                                idx_out: Optional[torch.Tensor] = None,
                                scores_out: Optional[torch.Tensor] = None,
                                ws: Optional[torch.Tensor] = None, stream=None):
    """In place on x (B, T, d)."""
    _dev(x, "x")
    B, T, _ = x.shape
    if ws is None:
        ws = workspace(adadsf_layer_workspace_size(cfg, B, T, K), x.device)
    lw = layer_struct(w)
    _check(lib().adadsf_sparse_layer_forward(ctypes.byref(cfg), ctypes.byref(lw), _p(x), B, T, int(K),
                                             _p(idx_out), _p(scores_out), _p(ws), ws.numel(),
                                             _s(stream)))


class DeviceModel:
    """Device tensors of a whole model plus the ctypes structs that point at them."""

    def __init__(self, cfg: ModelCfg, layers: Sequence[dict], extra: dict):
        self.cfg = cfg
        self.layers = list(layers)
        self.extra = extra
        self._lw = (LayerWeights * len(self.layers))(*[layer_struct(w) for w in self.layers])
        self.struct = ModelWeights(extra["embed"].data_ptr(), extra["final_w"].data_ptr(),
                                   extra["final_b"].data_ptr() if extra.get("final_b") is not None else None,
                                   ctypes.cast(self._lw, ctypes.POINTER(LayerWeights)))


def adadsf_sparse_model_forward(model: DeviceModel, ids: torch.Tensor, K: Sequence[int],
                                hidden_out: torch.Tensor, stats_acc: Optional[torch.Tensor] = None,
                                idx_out: Optional[torch.Tensor] = None,
                                ws: Optional[torch.Tensor] = None, stream=None):
    _dev(ids, "ids"); _dev(hidden_out, "hidden_out")
    B, T = ids.shape
    Karr = (ctypes.c_int32 * len(K))(*[int(k) for k in K])
    if ws is None:
        ws = workspace(adadsf_model_workspace_size(model.cfg, B, T, K, stats_acc is not None), ids.device)
    _check(lib().adadsf_sparse_model_forward(ctypes.byref(model.cfg), ctypes.byref(model.struct),
                                             _p(ids), B, T, ctypes.cast(Karr, ctypes.c_void_p),
                                             _p(hidden_out), _p(stats_acc), _p(idx_out), _p(ws),
                                             ws.numel(), _s(stream)))


def adadsf_kv_cache_size(cfg: ModelCfg, B: int, C_max: int) -> int:
    n = lib().adadsf_kv_cache_size(ctypes.byref(cfg), int(B), int(C_max))
    if n == 0:
        raise AdadsfError(ERR_INVALID_ARG, adadsf_last_error())
    return n


def adadsf_decode_workspace_size(cfg: ModelCfg, B: int, C_max: int) -> int:
    n = lib().adadsf_decode_workspace_size(ctypes.byref(cfg), int(B), int(C_max))
    if n == 0:
        raise AdadsfError(ERR_INVALID_ARG, adadsf_last_error())
    return n


def kv_cache(cfg: ModelCfg, B: int, C_max: int, device=None) -> torch.Tensor:
    """A zeroed decode cache for B sequences of up to C_max positions."""
    return torch.zeros(adadsf_kv_cache_size(cfg, B, C_max), dtype=torch.uint8, device=device or "cuda")


def adadsf_prefill(model: DeviceModel, ids: torch.Tensor, K: Sequence[int], hidden_out: torch.Tensor,
                   cache: torch.Tensor, C_max: int, idx_out: Optional[torch.Tensor] = None,
                   ws: Optional[torch.Tensor] = None, stream=None):
    """The sparse forward on the prompt ids (B, T), filling the decode cache."""
    _dev(ids, "ids"); _dev(hidden_out, "hidden_out"); _dev(cache, "cache")
    B, T = ids.shape
    Karr = (ctypes.c_int32 * len(K))(*[int(k) for k in K])
    if ws is None:
        ws = workspace(adadsf_model_workspace_size(model.cfg, B, T, K, False), ids.device)
    _check(lib().adadsf_prefill(ctypes.byref(model.cfg), ctypes.byref(model.struct), _p(ids), B, T,
                                ctypes.cast(Karr, ctypes.c_void_p), _p(hidden_out), _p(idx_out), _p(cache),
                                cache.numel(),
                                int(C_max), _p(ws), ws.numel(), _s(stream)))


def adadsf_decode_step(model: DeviceModel, ids: torch.Tensor, hidden_out: torch.Tensor, cache: torch.Tensor,
                       C_max: int, kept_out: Optional[torch.Tensor] = None, ws: Optional[torch.Tensor] = None,
                       stream=None):
    """One generated token per sequence (ids (B,)) through every layer."""
    _dev(ids, "ids"); _dev(hidden_out, "hidden_out"); _dev(cache, "cache")
    B = ids.numel()
    if ws is None:
        ws = workspace(adadsf_decode_workspace_size(model.cfg, B, C_max), ids.device)
    _check(lib().adadsf_decode_step(ctypes.byref(model.cfg), ctypes.byref(model.struct), _p(ids), B,
                                    _p(hidden_out), _p(kept_out), _p(cache), cache.numel(), int(C_max), _p(ws),
                                    ws.numel(), _s(stream)))


def adadsf_sync_check(ws: torch.Tensor, stream=None) -> int:
    """Synchronises and returns the status of the device error word (cleared)."""
    return lib().adadsf_sync_check(_p(ws), ws.numel(), _s(stream))


def adadsf_selftest_bounded_wait(ws: torch.Tensor, timeout_us: int, stream=None):
    _check(lib().adadsf_selftest_bounded_wait(_p(ws), ws.numel(), int(timeout_us), _s(stream)))


def adadsf_profile_begin(max_launches: int = 65536):
    """Start bracketing every library launch with CUDA events."""
    _check(lib().adadsf_profile_begin(int(max_launches)))


def adadsf_profile_end(max_records: int = 65536) -> list:
    """Stop profiling; returns [(kernel name, dense, ms, flops, bytes), ...] in launch order."""
    buf = (LaunchRecord * max_records)()
    n = lib().adadsf_profile_end(buf, max_records)
    if n < 0:
        raise AdadsfError(ERR_CUDA, adadsf_last_error())
    return [(adadsf_kernel_name(r.kind), bool(r.dense), r.ms, r.flops, r.bytes) for r in buf[:min(n, max_records)]]


def adadsf_kernel_name(kind: int) -> str:
    return lib().adadsf_kernel_name(int(kind)).decode()
