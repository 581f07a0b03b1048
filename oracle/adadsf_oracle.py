"""AdaDSF depth-sparse forward: plain fp64 CPU oracle.

TEST INFRASTRUCTURE ONLY. Only the test suite, the smoke check of the build
entry and the benchmark's CPU-baseline leg may import this module; the product
path never calls it and shares no code with it.

Every function is the plain definition of one step of the paper's method, in
float64 NumPy, with no blocking, fusion or reordering beyond what the definition
states. Matrix products (``@``), ``np.lexsort`` and ``scipy.special.erf`` serve as
library primitives.

Sources (paper "Adaptive Depth Sparse Framework", AdaDSF):
  * Sec. 3.1, Eq. 1   scaled dot-product attention softmax(QK^T/sqrt(d_k))V
  * Sec. 3.1, Eq. 2   FFN W2 sigma(W1 x + b1) + b2
  * Sec. 3.1, Eq. 3   a decoder layer composes attention and FFN with a
                      residual; the concrete (pre-norm) layer forms are those of
                      the GPT-NeoX and Qwen2.5 backbones the paper evaluates
                      (Sec. 4.1, "Models")
  * Sec. 3.3, Eq. 4   s_i = cosine similarity of layer input and output
  * Sec. 3.3, Eqs. 5-8  similarity -> layer-wise retention ratio r_i
  * Sec. 3.4          router scores, Top-K_i with K_i = floor(r_i * s), binary
                      mask, unselected tokens bypass through the residual path

Readings where the paper is silent (each one is listed in the design notes):
  * router = Linear(d, h) -> SiLU -> Linear(h, 1) on the raw residual stream;
  * kept tokens attend causally to kept tokens only, with rotary positions
    taken from their original token index;
  * Top-K ties go to the lower position; -0.0 equals +0.0; NaN ranks below -inf;
  * Eq. 8 can give r_i > 1; the default clamps to 1 and re-spreads the excess
    over the other layers in proportion to r'_i (``raw=True`` skips this);
  * K_i = floor(r_i * T + 1e-9), clamped to [0, T];
  * the similarity statistic is the mean over tokens of the per-token cosine
    (``mode="flat"``: cosine of the flattened tensors);
  * NeoX layer: x + Attn(LN1 x) + MLP(LN2 x); Qwen layer: h = x + Attn(RMS1 x),
    h + MLP(RMS2 h). The layer's residual delta is written to kept rows only.
  * router scores only select by default (kept rows get x + delta, so r = 1 is
    the dense layer); the score-gated variant (``p["gate"] == "sigmoid"``)
    scales each kept row's delta by sigmoid(score), which keeps the score
    pathway differentiable as Sec. 3.4 asks of training (Mixture-of-Depths
    style). The gate applies to the layer's whole delta; inside the layer
    (Qwen's h, the norms) nothing changes.
"""
from __future__ import annotations

import numpy as np
from scipy.special import erf

NEOX = 0
QWEN = 1


# --------------------------------------------------------------------------
# elementwise pieces
# --------------------------------------------------------------------------
def silu(x):
    """SiLU(x) = x * sigmoid(x)."""
    return x / (1.0 + np.exp(-x))


def sigmoid(x):
    """Logistic function 1 / (1 + e^-x)."""
    return 1.0 / (1.0 + np.exp(-np.asarray(x, dtype=np.float64)))


def gelu(x):
    """Exact GELU, x * Phi(x), with Phi the standard normal CDF."""
    return 0.5 * x * (1.0 + erf(x / np.sqrt(2.0)))


def layer_norm(x, g, b, eps):
    """LayerNorm over the last axis: biased variance, affine gain and bias."""
    mu = x.mean(axis=-1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)
    return (x - mu) / np.sqrt(var + eps) * g + b


def rms_norm(x, g, eps):
    """RMSNorm over the last axis: x / sqrt(mean(x^2) + eps) * g."""
    return x / np.sqrt((x * x).mean(axis=-1, keepdims=True) + eps) * g


def rope(v, pos, rotary_dim, theta):
    """Rotary embedding ("rotate half" convention) of the first ``rotary_dim``
    features of each row of v (n, head_dim) at integer positions pos (n,).
    Feature i < rotary_dim/2 pairs with i + rotary_dim/2 and both turn by the
    angle pos * theta^(-2i/rotary_dim)."""
    half = rotary_dim // 2
    inv = theta ** (-(np.arange(half, dtype=np.float64) * 2.0) / rotary_dim)
    ang = np.asarray(pos, dtype=np.float64)[:, None] * inv[None, :]
    c, s = np.cos(ang), np.sin(ang)
    out = np.array(v, dtype=np.float64, copy=True)
    a = v[:, :half]
    b = v[:, half:rotary_dim]
    out[:, :half] = a * c - b * s
    out[:, half:rotary_dim] = b * c + a * s
    return out


def linear(x, w, b=None, act=None):
    """Affine map of Eq. 2, x W^T + b (W stored [out, in]), optionally followed
    by the exact GELU."""
    y = np.asarray(x, dtype=np.float64) @ np.asarray(w, dtype=np.float64).T
    if b is not None:
        y = y + b
    if act == "gelu":
        y = gelu(y)
    return y


# --------------------------------------------------------------------------
# Eq. 1 -- attention among the given rows, causal in row order
# --------------------------------------------------------------------------
def causal_attention(q, k, v, n_heads, n_kv_heads, head_dim):
    """softmax(Q K^T / sqrt(d_k)) V per head (Eq. 1); row i sees rows j <= i.
    q (n, n_heads*hd), k and v (n, n_kv_heads*hd); query head h reads
    key/value head h // (n_heads / n_kv_heads)."""
    n = q.shape[0]
    out = np.zeros((n, n_heads * head_dim), dtype=np.float64)
    if n == 0:
        return out
    group = n_heads // n_kv_heads
    allowed = np.tril(np.ones((n, n), dtype=bool))
    for h in range(n_heads):
        g = h // group
        qh = q[:, h * head_dim:(h + 1) * head_dim]
        kh = k[:, g * head_dim:(g + 1) * head_dim]
        vh = v[:, g * head_dim:(g + 1) * head_dim]
        s = (qh @ kh.T) / np.sqrt(head_dim)
        s = np.where(allowed, s, -np.inf)
        s = s - s.max(axis=1, keepdims=True)
        p = np.exp(s)
        p = p / p.sum(axis=1, keepdims=True)
        out[:, h * head_dim:(h + 1) * head_dim] = p @ vh
    return out


# --------------------------------------------------------------------------
# Transformer layer on a packed set of tokens (Eqs. 1-3 in the backbone forms)
# --------------------------------------------------------------------------
def _attention_branch(a, pos, W, p):
    hd, H, Hkv = p["head_dim"], p["n_heads"], p["n_kv_heads"]
    qd, kvd = H * hd, Hkv * hd
    qkv = a @ W["w_qkv"].T + W["b_qkv"]
    q, k, v = qkv[:, :qd], qkv[:, qd:qd + kvd], qkv[:, qd + kvd:qd + 2 * kvd]
    q = np.concatenate([rope(q[:, h * hd:(h + 1) * hd], pos, p["rotary_dim"], p["rope_theta"])
                        for h in range(H)], axis=1) if len(pos) else q
    k = np.concatenate([rope(k[:, h * hd:(h + 1) * hd], pos, p["rotary_dim"], p["rope_theta"])
                        for h in range(Hkv)], axis=1) if len(pos) else k
    o = causal_attention(q, k, v, H, Hkv, hd)
    out = o @ W["w_o"].T
    if "b_o" in W:
        out = out + W["b_o"]
    return out


def block_delta(xp, pos, W, p):
    """Residual delta of one decoder layer applied to the packed rows xp (n, d)
    at original positions pos (n,): layer(xp) - xp."""
    eps = p["norm_eps"]
    if p["arch"] == NEOX:
        attn = _attention_branch(layer_norm(xp, W["ln1_w"], W["ln1_b"], eps), pos, W, p)
        m = layer_norm(xp, W["ln2_w"], W["ln2_b"], eps)
        mlp = gelu(m @ W["w_up"].T + W["b_up"]) @ W["w_down"].T + W["b_down"]
        return attn + mlp
    attn = _attention_branch(rms_norm(xp, W["ln1_w"], eps), pos, W, p)
    h = xp + attn
    m = rms_norm(h, W["ln2_w"], eps)
    mlp = (silu(m @ W["w_gate"].T) * (m @ W["w_up"].T)) @ W["w_down"].T
    return (h + mlp) - xp


# --------------------------------------------------------------------------
# Sec. 3.4 -- router and Top-K
# --------------------------------------------------------------------------
def router_scores(x, W):
    """Per-token importance score of the lightweight MLP router (Sec. 3.4):
    w2 . SiLU(W1 x + b1) + b2, for x (..., d)."""
    hdn = silu(x @ W["router_w1"].T + W["router_b1"])
    return hdn @ W["router_w2"] + W["router_b2"][0]


def topk_keep(scores, K):
    """Positions of the Top-K scores of one sequence (Sec. 3.4), ascending.
    Order: higher score first, equal scores by lower position; NaN ranks below
    every number; -0.0 and +0.0 compare equal."""
    scores = np.asarray(scores, dtype=np.float64)
    T = scores.shape[0]
    K = int(K)
    if K <= 0:
        return np.zeros(0, dtype=np.int64)
    nan = np.isnan(scores)
    key = np.where(nan, 0.0, scores)
    # lexsort: last key is primary
    order = np.lexsort((np.arange(T), -key, nan.astype(np.int8)))
    return np.sort(order[:K]).astype(np.int64)


# --------------------------------------------------------------------------
# Sec. 3.4 -- one sparse layer
# --------------------------------------------------------------------------
def sparse_layer_forward(x, W, p, K, idx=None):
    """Depth-sparse layer (Sec. 3.4) on x (B, T, d).

    Scores every token with the router, keeps the Top-K of each sequence
    (or the given ``idx`` (B, K)), runs the layer on the kept tokens only and
    adds its residual delta to those rows (scaled by sigmoid(score) when
    ``p["gate"] == "sigmoid"``); every other row is copied unchanged.
    Returns (x_out, idx (B, K), scores (B, T))."""
    x = np.asarray(x, dtype=np.float64)
    B, T, d = x.shape
    scores = router_scores(x, W)
    if idx is None:
        idx = np.stack([topk_keep(scores[b], K) for b in range(B)]) if B else np.zeros((0, K), np.int64)
    idx = np.asarray(idx, dtype=np.int64).reshape(B, -1)
    gated = p.get("gate", "none") == "sigmoid"
    out = x.copy()
    for b in range(B):
        sel = idx[b]
        if sel.size == 0:
            continue
        xp = x[b, sel]
        delta = block_delta(xp, sel, W, p)
        if gated:
            delta = sigmoid(scores[b, sel])[:, None] * delta
        out[b, sel] = xp + delta
    return out, idx, scores


# --------------------------------------------------------------------------
# Sec. 3.3, Eq. 4 -- similarity statistic
# --------------------------------------------------------------------------
COS_EPS = 1e-8


def cos_sim_stat(x_in, x_out, mode="token"):
    """Eq. 4 accumulated over a batch. Returns the additive partial sums:
    mode "token": (sum over rows of cos(x_in_row, x_out_row), number of rows),
                  cos = a.b / (max(|a|, eps) * max(|b|, eps));
    mode "flat":  (sum a.b, sum |a|^2, sum |b|^2) over all rows."""
    a = np.asarray(x_in, dtype=np.float64).reshape(-1, np.shape(x_in)[-1])
    b = np.asarray(x_out, dtype=np.float64).reshape(-1, np.shape(x_out)[-1])
    dot = (a * b).sum(axis=1)
    na2 = (a * a).sum(axis=1)
    nb2 = (b * b).sum(axis=1)
    if mode == "token":
        cos = dot / (np.maximum(np.sqrt(na2), COS_EPS) * np.maximum(np.sqrt(nb2), COS_EPS))
        return float(cos.sum()), float(a.shape[0])
    return float(dot.sum()), float(na2.sum()), float(nb2.sum())


def similarity(acc, mode="token"):
    """s_i from the accumulated partial sums of ``cos_sim_stat``."""
    if mode == "token":
        return acc[0] / acc[1]
    return acc[0] / (max(np.sqrt(acc[1]), COS_EPS) * max(np.sqrt(acc[2]), COS_EPS))


# --------------------------------------------------------------------------
# Sec. 3.3, Eqs. 5-8 -- retention allocation
# --------------------------------------------------------------------------
def allocate_ratios(s, t, tau=0.05, beta=10.0, raw=False):
    """Layer-wise retention ratios from the similarity vector s (length L).

    Eq. 5: w~_i = exp((s_i - max s)/tau), w = w~ / sum w~
    Eq. 6: z_i = beta * (mean(w) - w_i)
    Eq. 7: r'_i = 0.05 + 0.9 * sigmoid(z_i)
    Eq. 8: r_i = t L r'_i / sum_j r'_j
    Unless ``raw``, ratios above 1 are clamped to 1 and the remaining budget
    t L - (#clamped) is spread over the other layers in proportion to r'_i,
    repeated until no ratio exceeds 1 (t >= 1 gives all ones)."""
    s = np.asarray(s, dtype=np.float64)
    L = s.shape[0]
    wt = np.exp((s - s.max()) / tau)
    w = wt / wt.sum()
    z = beta * (w.mean() - w)
    rp = 0.05 + 0.9 / (1.0 + np.exp(-z))
    r = t * L / rp.sum() * rp
    if raw:
        return r, rp
    if t >= 1.0:
        return np.ones(L), rp
    fixed = np.zeros(L, dtype=bool)
    while True:
        over = (~fixed) & (r > 1.0)
        if not over.any():
            break
        fixed |= over
        budget = t * L - fixed.sum()
        r = np.where(fixed, 1.0, budget / rp[~fixed].sum() * rp)
    return r, rp


def kept_counts(r, T, rounding="floor"):
    """K_i = floor(r_i * T) (Sec. 3.4), with a 1e-9 guard against ratios that
    land a hair below an integer; ``rounding="round"`` rounds to nearest."""
    r = np.asarray(r, dtype=np.float64)
    if rounding == "floor":
        K = np.floor(r * T + 1e-9)
    else:
        K = np.floor(r * T + 0.5)
    return np.clip(K, 0, T).astype(np.int64)


# --------------------------------------------------------------------------
# whole model: embedding -> L sparse layers -> final norm
# --------------------------------------------------------------------------
def final_norm(x, Wm, p):
    if p["arch"] == NEOX:
        return layer_norm(x, Wm["final_w"], Wm["final_b"], p["norm_eps"])
    return rms_norm(x, Wm["final_w"], p["norm_eps"])


def sparse_model_forward(ids, Wm, layers, p, K, idx_force=None, stats_mode=None):
    """Embedding lookup, then each layer l as a sparse layer with K[l] kept
    tokens per sequence (or the kept sets idx_force[l]), then the final norm.
    With ``stats_mode`` the Eq. 4 partial sums of every layer's input/output
    pair are returned too. Returns (hidden, [idx_l], [stats_l])."""
    x = np.asarray(Wm["embed"], dtype=np.float64)[np.asarray(ids)]
    kept, stats = [], []
    for l, W in enumerate(layers):
        x_new, idx, _ = sparse_layer_forward(x, W, p, K[l], None if idx_force is None else idx_force[l])
        if stats_mode is not None:
            stats.append(cos_sim_stat(x, x_new, stats_mode))
        kept.append(idx)
        x = x_new
    return final_norm(x, Wm, p), kept, stats


def params_of(shape):
    """Plain dict of the backbone hyper-parameters the functions above read."""
    return {k: getattr(shape, k) for k in
            ("arch", "d", "n_heads", "n_kv_heads", "head_dim", "ffn", "rotary_dim",
             "rope_theta", "norm_eps")}


# --------------------------------------------------------------------------
# Sec. 4.1 (Tables 1-2) -- normalized FLOPs of the depth-sparse forward
# --------------------------------------------------------------------------
def block_flops(p, K):
    """Floating-point operations (2 per multiply-add) of one decoder layer on
    the K kept tokens of one sequence: the QKV, output and MLP projections
    (3 MLP matrices for SwiGLU, 2 for GELU) plus causal attention among the
    kept tokens (query i meets i + 1 keys in Q K^T and in P V)."""
    d, H, Hkv, hd, F_ = p["d"], p["n_heads"], p["n_kv_heads"], p["head_dim"], p["ffn"]
    q, kv = H * hd, Hkv * hd
    n_mlp = 3 if p["arch"] == QWEN else 2
    proj = 2.0 * K * ((q + 2 * kv) * d + d * q + n_mlp * d * F_)
    attn = 2.0 * H * hd * K * (K + 1)
    return proj + attn


def router_flops(p, T, h=64):
    """The router's multiply-adds on all T tokens of one sequence: W1 (h x d)
    and w2 (h)."""
    return 2.0 * T * h * (p["d"] + 1)


def normalized_flops(p, T, K, h=64):
    """Sparse-forward FLOPs over the dense model's, per sequence of T tokens:
    sum over layers of (router on all T tokens when the layer drops any,
    plus the layer on its K_l kept tokens) divided by the sum of the dense
    layers on T tokens. Embedding, final norm and LM head are left out (the
    same in both). K = T everywhere gives 1; K = 0 everywhere gives the
    routers' cost alone."""
    num = sum((router_flops(p, T, h) if k < T else 0.0) + block_flops(p, k) for k in K)
    return num / (len(K) * block_flops(p, T))


# --------------------------------------------------------------------------
# Autoregressive decode with a cache of kept tokens only (the paper is silent
# on generation; this is a Mixture-of-Depths style reading)
# --------------------------------------------------------------------------
def kept_threshold(scores, idx):
    """The lowest router score among a sequence's kept tokens (the K-th
    largest of Sec. 3.4's Top-K); +inf when nothing is kept (a layer that
    keeps no prompt token keeps no generated token either)."""
    s = np.asarray(scores, dtype=np.float64)[np.asarray(idx, dtype=np.int64)]
    return float(s.min()) if s.size else np.inf


def decode_keep(score, threshold):
    """Causal keep decision of a new token: kept iff its score beats the
    threshold strictly (a tie loses, as the later position loses ties in
    Top-K; NaN never wins)."""
    return bool(score > threshold)


def sparse_prefill(ids, Wm, layers, p, K, idx_force=None):
    """The sparse model on the prompt (sparse_model_forward) plus the state a
    decode needs per layer l and sequence b: the kept positions, the kept
    tokens' layer-l INPUT rows (their keys and values are functions of
    these), and the threshold of Sec. 3.4's Top-K. ``idx_force[l]`` (B, K_l)
    replaces layer l's Top-K (the threshold is then taken over the forced
    set). Returns (hidden, state) with state = {"pos": [l][b] list, "rows":
    [l][b] list, "thr": [l][b], "T": prompt length}."""
    ids = np.asarray(ids)
    x = np.asarray(Wm["embed"], dtype=np.float64)[ids]
    B, T = ids.shape
    st = {"pos": [], "rows": [], "thr": [], "T": T}
    for l, W in enumerate(layers):
        x_new, idx, sc = sparse_layer_forward(x, W, p, K[l], None if idx_force is None else idx_force[l])
        st["pos"].append([list(idx[b]) for b in range(B)])
        st["rows"].append([[x[b, t].copy() for t in idx[b]] for b in range(B)])
        st["thr"].append([kept_threshold(sc[b], idx[b]) for b in range(B)])
        x = x_new
    return final_norm(x, Wm, p), st


def decode_step(ids_new, Wm, layers, p, st, kept_force=None):
    """One generated token per sequence at position st["T"] (then st["T"] +=
    1). Layer by layer: the router scores the token's current hidden state;
    if it beats the layer's threshold the token is kept -- it attends
    causally to the layer's kept tokens (rotary at original positions), its
    residual delta is added, and it joins the layer's kept set (its input
    row is cached); otherwise it bypasses the layer unchanged. Computed from
    the definition: the layer is re-run on the kept rows plus the new one
    and the last row's delta is taken (attention is causal, so earlier kept
    rows are unaffected). ``kept_force`` (L, B) bool replaces the decisions
    (the scores and own decisions are still returned). Returns (hidden (B, d)
    after the final norm, kept (L, B) bool -- this function's own decisions
    --, scores (L, B) of the router at each layer)."""
    ids_new = np.asarray(ids_new).reshape(-1)
    B = ids_new.shape[0]
    t = st["T"]
    x = np.asarray(Wm["embed"], dtype=np.float64)[ids_new]
    kept = np.zeros((len(layers), B), dtype=bool)
    scores = np.zeros((len(layers), B))
    gated = p.get("gate", "none") == "sigmoid"
    for l, W in enumerate(layers):
        sc = router_scores(x, W)
        scores[l] = sc
        x_next = x.copy()
        for b in range(B):
            kept[l, b] = decode_keep(sc[b], st["thr"][l][b])
            if not (kept[l, b] if kept_force is None else kept_force[l][b]):
                continue
            rows = np.array(st["rows"][l][b] + [x[b]])
            pos = np.array(st["pos"][l][b] + [t])
            delta = block_delta(rows, pos, W, p)[-1]
            if gated:
                delta = sigmoid(sc[b]) * delta
            x_next[b] = x[b] + delta
            st["rows"][l][b].append(x[b].copy())
            st["pos"][l][b].append(t)
        x = x_next
    st["T"] = t + 1
    return final_norm(x, Wm, p), kept, scores


# --------------------------------------------------------------------------
# Sec. 3.5, Eqs. 9-11 -- feature-preserving alignment objective, and the
# router's gradient through the score gate (Sec. 3.4: router scores on the
# differentiable path)
# --------------------------------------------------------------------------
def softmax(z, axis=-1):
    """exp(z - max) / sum exp(z - max) along `axis`."""
    z = np.asarray(z, dtype=np.float64)
    e = np.exp(z - z.max(axis=axis, keepdims=True))
    return e / e.sum(axis=axis, keepdims=True)


def hidden_alignment(h_sparse, h_dense):
    """Eq. 9 for one layer, per token: || softmax(h_sparse) - softmax(h_dense) ||_2
    with the softmax over the hidden features of the token. Returns the
    per-token values (shape of the inputs without the last axis); the layer's
    loss is their mean."""
    return np.sqrt(((softmax(h_sparse) - softmax(h_dense)) ** 2).sum(axis=-1))


def hidden_alignment_grad(h_sparse, h_dense):
    """Gradient of each token's Eq. 9 value with respect to its h_sparse row
    (by the chain rule through the norm and the softmax): with p =
    softmax(h_sparse), q = softmax(h_dense), r = p - q, n = |r|,
    d n / d h = p * (r / n - p . r / n); zero where n = 0."""
    p = softmax(h_sparse)
    r = p - softmax(h_dense)
    n = np.sqrt((r * r).sum(axis=-1, keepdims=True))
    safe = np.where(n > 0, n, 1.0)
    u = r / safe
    g = p * (u - (p * u).sum(axis=-1, keepdims=True))
    return np.where(n > 0, g, 0.0)


def output_alignment(h_sparse, h_dense, w_head):
    """Eq. 10 per token: KL(P_dense || P_sparse) = sum_c P_dense(c) log(P_dense(c)
    / P_sparse(c)), P = softmax of the logits h W_head^T over the classes.
    Returns the per-token values; the loss is their mean."""
    ls = np.asarray(h_sparse, dtype=np.float64) @ np.asarray(w_head, dtype=np.float64).T
    ld = np.asarray(h_dense, dtype=np.float64) @ np.asarray(w_head, dtype=np.float64).T
    lps = ls - ls.max(axis=-1, keepdims=True)
    lps = lps - np.log(np.exp(lps).sum(axis=-1, keepdims=True))
    lpd = ld - ld.max(axis=-1, keepdims=True)
    lpd = lpd - np.log(np.exp(lpd).sum(axis=-1, keepdims=True))
    return (np.exp(lpd) * (lpd - lps)).sum(axis=-1)


def alignment_objective(l_align, l_hid_layers):
    """Eq. 11: L = L_align + (1/L) sum_l L_hid^(l), from the per-token means."""
    return float(l_align) + float(np.mean(l_hid_layers))


def router_grad(x, W, rows, delta, grad_y):
    """Gradient of a loss with respect to the router parameters of one gated
    layer (kept rows y = x + sigmoid(s) delta, Sec. 3.4), given the loss's
    gradient grad_y at the kept rows' outputs and the layer's ungated delta
    there; x and the layer's other weights are held fixed, and the Top-K
    choice itself carries no gradient. rows: the kept rows of x (n, d) as a
    flat index; delta, grad_y: (n_kept, d). Chain rule:
      ds = sigmoid'(s) (grad_y . delta),  s = w2 . SiLU(u) + b2,  u = W1 x + b1
      dw2 = sum ds SiLU(u), db2 = sum ds, du = ds w2 SiLU'(u),
      dW1 = sum du (x) x, db1 = sum du.
    Returns a dict with router_w1, router_b1, router_w2, router_b2."""
    xs = np.asarray(x, dtype=np.float64).reshape(-1, np.shape(x)[-1])[np.asarray(rows)]
    u = xs @ W["router_w1"].T + W["router_b1"]
    sg = 1.0 / (1.0 + np.exp(-u))
    su = u * sg
    s = su @ W["router_w2"] + W["router_b2"][0]
    sig = sigmoid(s)
    ds = sig * (1.0 - sig) * (np.asarray(grad_y, dtype=np.float64) * np.asarray(delta, dtype=np.float64)).sum(-1)
    dsilu = sg * (1.0 + u * (1.0 - sg))
    du = ds[:, None] * W["router_w2"][None, :] * dsilu
    return {"router_w1": du.T @ xs, "router_b1": du.sum(0), "router_w2": (ds[:, None] * su).sum(0),
            "router_b2": np.array([ds.sum()])}
