"""Feature-preserving alignment of one sparse layer's router (Sec. 3.5), on
synthetic data: the layer-local form of Eq. 9 with the router trained
through the score gate of the gated variant (Sec. 3.4: the router scores
stay on the differentiable path in training). Every step of the method runs in the
library's kernels (the gated and ungated layer forwards, the Eq. 9 value and
gradient, the router's parameter gradient); this module only sequences the
calls and applies the plain SGD update to the router tensors.

The layer input x and the dense layer's output h_dense are held fixed
(teacher forcing from the dense model, as Eq. 9 compares the two models
layer by layer), so the step's gradient is that of the layer's own L_hid.
"""
from __future__ import annotations

from typing import Optional

import torch

from . import adadsf as A

ROUTER_KEYS = ("router_w1", "router_b1", "router_w2", "router_b2")


def router_alignment_step(shape_cfg: A.ModelCfg, w: dict, x: torch.Tensor, h_dense: torch.Tensor, K: int,
                          lr: float, stream=None, ws: Optional[torch.Tensor] = None):
    """One SGD step on the router of layer weights `w` (device tensors; the
    router tensors are updated in place) against L_hid of Eq. 9 between the
    gated sparse layer's output on x (B, T, d) and h_dense (B, T, d).
    shape_cfg: the layer's config (the gate flag is set here). Returns the
    layer's L_hid before the step (mean over the B T tokens)."""
    B, T, d = x.shape
    cfg_g = A.ModelCfg.from_buffer_copy(shape_cfg)
    cfg_g.flags = int(cfg_g.flags) | A.FLAG_GATE_SIGMOID
    cfg_p = A.ModelCfg.from_buffer_copy(shape_cfg)
    cfg_p.flags = int(cfg_p.flags) & ~A.FLAG_GATE_SIGMOID
    if ws is None:
        ws = A.workspace(A.adadsf_layer_workspace_size(cfg_g, B, T, K), x.device)
    idx = torch.empty((B, K), dtype=torch.int32, device=x.device)
    y_g = x.clone()
    A.adadsf_sparse_layer_forward(cfg_g, w, y_g, K, idx, None, ws, stream)
    y_p = x.clone()
    idx_p = torch.empty_like(idx)
    A.adadsf_sparse_layer_forward(cfg_p, w, y_p, K, idx_p, None, ws, stream)
    acc = torch.zeros(2, dtype=torch.float64, device=x.device)
    grad_y = torch.empty((B * T, d), dtype=torch.float32, device=x.device)
    A.adadsf_align_hidden(y_g, h_dense, acc, grad_y, stream=stream)
    rows = (torch.arange(B, device=x.device, dtype=torch.int32)[:, None] * T + idx).reshape(-1).contiguous()
    g = A.adadsf_router_backward(cfg_g, w, x, y_p, rows, grad_y, stream=stream)
    # the mean over tokens: scale by 1 / (B T); plain SGD on the router tensors
    h = shape_cfg.router_hidden
    scale = lr / float(B * T)
    sizes = {"router_w1": h * d, "router_b1": h, "router_w2": h, "router_b2": 1}
    off = 0
    for k in ROUTER_KEYS:
        n = sizes[k]
        w[k].sub_((g[off:off + n] * scale).view(w[k].shape).to(w[k].dtype))
        off += n
    return float(acc[0] / acc[1])
