"""Pins of the fp64 oracle against facts that do not come from the oracle itself:
library routines it must agree with on special cases, closed forms, limits,
invariants the paper states or the mathematics fixes, and brute force.

Each group below names the passage of the paper it pins."""
import math
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as F
from scipy.spatial.distance import cosine as scipy_cosine_distance

from oracle import adadsf_oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _paper_constants():
    vals = {}
    with open(os.path.join(GOLDEN, "paper_constants.txt")) as f:
        for line in f:
            line = line.split("#")[0].strip()
            if line:
                k, v = line.split()
                vals.setdefault(k, []).append(float(v))
    return vals


PC = _paper_constants()
BETA = PC["beta"][0]
TAUS = PC["tau"]


def rng(seed=0):
    return np.random.default_rng(seed)


# ---------------------------------------------------------------- Eqs. 5-8
class TestAllocation:
    def test_budget_eq8(self):
        """Eq. 8 rescales so that sum r = t L."""
        g = rng(1)
        for L in (1, 2, 5, 12, 28):
            s = g.uniform(0.3, 1.0, L)
            for t in (0.25, 0.5, 0.9):
                r, _ = O.allocate_ratios(s, t, 0.05, BETA, raw=True)
                assert r.sum() == pytest.approx(t * L, rel=1e-12)

    def test_ratio_bounds_eq7(self):
        """Eq. 7 maps into (floor, floor + span) = (0.05, 0.95)."""
        lo, span = PC["ratio_floor"][0], PC["ratio_span"][0]
        g = rng(2)
        for _ in range(50):
            s = g.uniform(-1, 1, 16)
            _, rp = O.allocate_ratios(s, 0.5, 0.01, BETA, raw=True)
            assert (rp > lo).all() and (rp < lo + span).all()

    def test_uniform_similarity_gives_uniform_ratio(self):
        """Equal s_i: w = 1/L, z = 0, r' = 0.05 + 0.45 = 0.5, r = t."""
        for L in (1, 3, 12):
            r, rp = O.allocate_ratios(np.full(L, 0.7), 0.6, 0.05, BETA)
            assert np.allclose(rp, 0.5, rtol=0, atol=1e-15)
            assert np.allclose(r, 0.6, rtol=1e-14)

    def test_two_layer_closed_form(self):
        """L = 2: mean(w) = 1/2 so z_2 = -z_1 and r'_1 + r'_2 = 0.1 + 0.9 = 1;
        hence r_i = 2 t r'_i, with r'_1 = 0.05 + 0.9 sig(beta (1/2 - sig((s1 - s2)/tau)))."""
        g = rng(3)
        for _ in range(20):
            s = g.uniform(0, 1, 2)
            tau = g.choice(TAUS)
            t = g.uniform(0.1, 0.5)
            r, rp = O.allocate_ratios(s, t, tau, BETA, raw=True)
            assert rp.sum() == pytest.approx(1.0, abs=1e-14)
            sig = lambda v: 1.0 / (1.0 + math.exp(-v))
            w1 = sig((s[0] - s[1]) / tau)
            rp1 = 0.05 + 0.9 * sig(BETA * (0.5 - w1))
            assert rp[0] == pytest.approx(rp1, rel=1e-13)
            assert r == pytest.approx(2 * t * rp, rel=1e-13)

    def test_worked_example(self):
        """Values worked out by hand from Eqs. 5-8 (tau = 0.05, beta = 10, t = 0.5),
        quoted to 4 decimals; the paper prints no numeric example."""
        r, rp = O.allocate_ratios([0.9, 0.95, 0.99, 0.8], 0.5, 0.05, BETA, raw=True)
        assert np.round(rp, 4) == pytest.approx([0.7845, 0.4452, 0.0737, 0.8726], abs=1e-4)
        assert np.round(r, 4) == pytest.approx([0.7210, 0.4092, 0.0678, 0.8020], abs=1e-4)
        r, _ = O.allocate_ratios([0.1, 0.2, 0.3, 0.99], 0.5, 0.05, BETA, raw=True)
        assert np.round(r, 4) == pytest.approx([0.6542, 0.6542, 0.6542, 0.0375], abs=1e-4)
        r, _ = O.allocate_ratios([0.9, 0.95, 0.99, 0.8], 1.0, 0.05, BETA, raw=True)
        assert np.round(r, 4) == pytest.approx([1.4421, 0.8184, 0.1355, 1.6040], abs=1e-4)

    def test_one_hot_limit(self):
        """tau -> 0 with a unique maximum: w = e_max, z_max = beta (1/L - 1),
        z_other = beta / L (closed form)."""
        L = 4
        _, rp = O.allocate_ratios([0.1, 0.2, 0.3, 0.99], 0.5, 1e-4, BETA, raw=True)
        sig = lambda v: 1.0 / (1.0 + math.exp(-v))
        assert rp[3] == pytest.approx(0.05 + 0.9 * sig(BETA * (1 / L - 1)), rel=1e-12)
        assert rp[:3] == pytest.approx([0.05 + 0.9 * sig(BETA / L)] * 3, rel=1e-12)

    def test_high_temperature_limit(self):
        """tau -> infinity: weights become uniform, so r -> t."""
        r, _ = O.allocate_ratios([0.1, 0.5, 0.9, 0.3], 0.4, 1e9, BETA, raw=True)
        assert r == pytest.approx([0.4] * 4, rel=1e-7)

    def test_shift_invariance(self):
        """Eq. 5 subtracts max(s): s + c gives the same ratios."""
        g = rng(4)
        s = g.uniform(0.5, 1.0, 12)
        a, _ = O.allocate_ratios(s, 0.5, 0.05, BETA, raw=True)
        b, _ = O.allocate_ratios(s + 3.25, 0.5, 0.05, BETA, raw=True)
        assert np.allclose(a, b, rtol=1e-12)

    def test_more_similar_layer_gets_less_compute(self):
        """Sec. 3.3: layers with larger transformation (smaller s) receive more
        compute; so s_i > s_j implies r_i < r_j."""
        g = rng(5)
        s = g.permutation(np.linspace(0.6, 0.99, 10))
        r, _ = O.allocate_ratios(s, 0.5, 0.05, BETA, raw=True)
        order = np.argsort(s)
        assert (np.diff(r[order]) < 0).all()

    def test_smaller_tau_larger_variance(self):
        """Sec. 4.3 (Table 3 discussion): smaller tau yields a larger variance
        of the retention ratios."""
        s = np.array([0.80, 0.86, 0.90, 0.93, 0.95, 0.97, 0.98, 0.99])
        var = [np.var(O.allocate_ratios(s, 0.5, tau, BETA, raw=True)[0]) for tau in sorted(TAUS, reverse=True)]
        assert var[0] < var[1] < var[2]

    def test_clamp_redistributes(self):
        """Reading for r_i > 1: clamp to 1 and re-spread the budget in
        proportion to r'; the budget t L is kept and order is preserved."""
        s = [0.9, 0.95, 0.99, 0.8]
        r, rp = O.allocate_ratios(s, 0.75, 0.05, BETA)
        assert r.sum() == pytest.approx(3.0, rel=1e-12)
        assert (r <= 1.0).all()
        assert r[0] == 1.0 and r[3] == 1.0
        assert r[1] / r[2] == pytest.approx(rp[1] / rp[2], rel=1e-12)
        r, _ = O.allocate_ratios(s, 1.0, 0.05, BETA)
        assert (r == 1.0).all()

    def test_kept_counts_floor(self):
        """K_i = floor(r_i * s) (Sec. 3.4)."""
        assert O.kept_counts([0.5, 0.25, 0.999, 1.0, 0.0], 512).tolist() == [256, 128, 511, 512, 0]
        r = np.full(12, 0.5)
        r = 0.5 * 12 / r.sum() * r          # ratios that may land a hair below 0.5
        assert (O.kept_counts(r, 512) == 256).all()


# ---------------------------------------------------------------- Sec. 3.4 Top-K
def _brute_topk(scores, K):
    """Kept iff fewer than K tokens rank ahead of it (O(T^2) definition)."""
    T = len(scores)

    def ahead(u, t):
        su, st = scores[u], scores[t]
        nu, nt = math.isnan(su), math.isnan(st)
        if nu and nt:
            return u < t
        if nu != nt:
            return nt          # a number is ahead of NaN
        if su != st:
            return su > st
        return u < t

    return [t for t in range(T) if sum(ahead(u, t) for u in range(T) if u != t) < K]


class TestTopK:
    def test_hand_built_ties(self):
        """Ties -> lower position; -0.0 == +0.0; NaN below everything."""
        s = [1.0, 3.0, 3.0, 2.0, 3.0, -0.0, 0.0, float("nan")]
        expect = {0: [], 1: [1], 3: [1, 2, 4], 5: [0, 1, 2, 3, 4], 6: [0, 1, 2, 3, 4, 5],
                  7: [0, 1, 2, 3, 4, 5, 6], 8: list(range(8))}
        for K, e in expect.items():
            assert O.topk_keep(s, K).tolist() == e

    def test_brute_force(self):
        g = rng(6)
        for trial in range(60):
            T = int(g.integers(1, 40))
            s = g.normal(size=T)
            if trial % 3 == 0:
                s = np.round(s, 1)                     # many ties
            if trial % 5 == 0:
                s[g.integers(0, T, 3)] = np.nan
            if trial % 7 == 0:
                s[g.integers(0, T, 2)] = -np.inf
            K = int(g.integers(0, T + 1))
            assert O.topk_keep(s, K).tolist() == _brute_topk(list(s), K)


# ---------------------------------------------------------------- Eq. 4
class TestCosSim:
    def test_special_cases(self):
        g = rng(7)
        x = g.normal(size=(5, 33))
        assert O.similarity(O.cos_sim_stat(x, x)) == pytest.approx(1.0, abs=1e-15)
        assert O.similarity(O.cos_sim_stat(x, -x)) == pytest.approx(-1.0, abs=1e-15)
        assert O.similarity(O.cos_sim_stat(x, 2.5 * x)) == pytest.approx(1.0, abs=1e-15)
        a = np.zeros((2, 4)); a[:, 0] = 1
        b = np.zeros((2, 4)); b[:, 1] = 3
        assert O.similarity(O.cos_sim_stat(a, b)) == 0.0
        assert O.similarity(O.cos_sim_stat(x, x, "flat"), "flat") == pytest.approx(1.0, abs=1e-15)

    def test_matches_scipy(self):
        g = rng(8)
        a, b = g.normal(size=(7, 20)), g.normal(size=(7, 20))
        tot, n = O.cos_sim_stat(a, b)
        ref = sum(1.0 - scipy_cosine_distance(a[i], b[i]) for i in range(7))
        assert n == 7 and tot == pytest.approx(ref, rel=1e-13)
        d, na, nb = O.cos_sim_stat(a, b, "flat")
        assert O.similarity((d, na, nb), "flat") == pytest.approx(
            1.0 - scipy_cosine_distance(a.ravel(), b.ravel()), rel=1e-13)


# ---------------------------------------------------------------- Eqs. 1-3 building blocks
T64 = torch.float64


class TestPieces:
    def test_gelu_silu(self):
        x = np.linspace(-6, 6, 101)
        assert O.gelu(x) == pytest.approx(F.gelu(torch.tensor(x, dtype=T64)).numpy(), rel=1e-13, abs=1e-15)
        assert O.silu(x) == pytest.approx(F.silu(torch.tensor(x, dtype=T64)).numpy(), rel=1e-13, abs=1e-15)
        assert O.gelu(np.array([1.0]))[0] == pytest.approx(0.8413447460685429, rel=1e-15)  # Phi(1)

    def test_norms(self):
        g = rng(9)
        x, w, b = g.normal(size=(6, 40)), g.normal(size=40), g.normal(size=40)
        ref = F.layer_norm(torch.tensor(x), (40,), torch.tensor(w), torch.tensor(b), 1e-5).numpy()
        assert O.layer_norm(x, w, b, 1e-5) == pytest.approx(ref, rel=1e-12, abs=1e-13)
        y = O.rms_norm(x, np.ones(40), 0.0)
        assert np.sqrt((y * y).mean(axis=1)) == pytest.approx(np.ones(6), rel=1e-13)
        if hasattr(F, "rms_norm"):
            ref = F.rms_norm(torch.tensor(x), (40,), torch.tensor(w), 1e-6).numpy()
            assert O.rms_norm(x, w, 1e-6) == pytest.approx(ref, rel=1e-12, abs=1e-13)

    def test_rope_complex_form(self):
        """Rotate-half RoPE = multiplying (a_i + i b_i) by exp(i pos theta^(-2i/r))."""
        g = rng(10)
        hd, rot, theta = 16, 8, 1e4
        v = g.normal(size=(5, hd))
        pos = np.array([0, 1, 7, 100, 4095])
        out = O.rope(v, pos, rot, theta)
        half = rot // 2
        for n in range(5):
            for i in range(half):
                z = complex(v[n, i], v[n, i + half]) * np.exp(1j * pos[n] * theta ** (-2 * i / rot))
                assert out[n, i] == pytest.approx(z.real, abs=1e-12)
                assert out[n, i + half] == pytest.approx(z.imag, abs=1e-12)
        assert out[:, rot:] == pytest.approx(v[:, rot:], abs=0)
        assert out[0] == pytest.approx(v[0], abs=1e-15)          # position 0 is the identity

    def test_rope_relative(self):
        """q.k after RoPE depends on the position difference only."""
        g = rng(11)
        q, k = g.normal(size=(1, 32)), g.normal(size=(1, 32))
        a = O.rope(q, [9], 32, 1e6) @ O.rope(k, [3], 32, 1e6).T
        b = O.rope(q, [1009], 32, 1e6) @ O.rope(k, [1003], 32, 1e6).T
        assert a == pytest.approx(b, rel=1e-10)

    @pytest.mark.parametrize("H,Hkv", [(4, 4), (6, 2)])
    def test_attention_vs_sdpa(self, H, Hkv):
        g = rng(12)
        n, hd = 9, 16
        q, k, v = g.normal(size=(n, H * hd)), g.normal(size=(n, Hkv * hd)), g.normal(size=(n, Hkv * hd))
        out = O.causal_attention(q, k, v, H, Hkv, hd)
        tq = torch.tensor(q).view(n, H, hd).transpose(0, 1)
        tk = torch.tensor(k).view(n, Hkv, hd).transpose(0, 1).repeat_interleave(H // Hkv, 0)
        tv = torch.tensor(v).view(n, Hkv, hd).transpose(0, 1).repeat_interleave(H // Hkv, 0)
        ref = F.scaled_dot_product_attention(tq, tk, tv, is_causal=True).transpose(0, 1).reshape(n, H * hd)
        assert out == pytest.approx(ref.numpy(), rel=1e-12, abs=1e-13)

    def test_attention_special_cases(self):
        g = rng(13)
        v = g.normal(size=(6, 8))
        k = np.tile(g.normal(size=(1, 8)), (6, 1))          # identical keys
        out = O.causal_attention(g.normal(size=(6, 8)), k, v, 1, 1, 8)
        for i in range(6):                                   # uniform mean of the prefix
            assert out[i] == pytest.approx(v[:i + 1].mean(axis=0), rel=1e-12)
        one = O.causal_attention(g.normal(size=(1, 8)), g.normal(size=(1, 8)), v[:1], 1, 1, 8)
        assert one == pytest.approx(v[:1], rel=1e-15)         # softmax of one score


# ---------------------------------------------------------------- Sec. 3.4 layer
def _params(arch, d=32, H=4, Hkv=4, hd=8, F_=48, rot=4, theta=1e4):
    return {"arch": arch, "d": d, "n_heads": H, "n_kv_heads": Hkv, "head_dim": hd, "ffn": F_,
            "rotary_dim": rot, "rope_theta": theta, "norm_eps": 1e-5}


def _weights(p, seed, rh=8, zero=()):
    g = rng(seed)
    d, q, kv, F_ = p["d"], p["n_heads"] * p["head_dim"], p["n_kv_heads"] * p["head_dim"], p["ffn"]
    W = {"router_w1": g.normal(0, 0.3, (rh, d)), "router_b1": g.normal(0, 0.3, rh),
         "router_w2": g.normal(0, 0.3, rh), "router_b2": g.normal(0, 0.3, 1),
         "ln1_w": 1 + g.normal(0, 0.1, d), "ln2_w": 1 + g.normal(0, 0.1, d),
         "w_qkv": g.normal(0, 0.2, (q + 2 * kv, d)), "b_qkv": g.normal(0, 0.2, q + 2 * kv),
         "w_o": g.normal(0, 0.2, (d, q)), "w_up": g.normal(0, 0.2, (F_, d)), "w_down": g.normal(0, 0.2, (d, F_))}
    if p["arch"] == O.NEOX:
        W.update({"ln1_b": g.normal(0, 0.1, d), "ln2_b": g.normal(0, 0.1, d), "b_o": g.normal(0, 0.2, d),
                  "b_up": g.normal(0, 0.2, F_), "b_down": g.normal(0, 0.2, d)})
    else:
        W["w_gate"] = g.normal(0, 0.2, (F_, d))
    for z in zero:
        W[z] = np.zeros_like(W[z])
    return W


class TestLayer:
    def test_router_closed_form(self):
        """d=2, h=1: score = 2 * SiLU(3) + 0.5 with SiLU(3) = 3 / (1 + e^-3)."""
        W = {"router_w1": np.array([[1.0, 0.0]]), "router_b1": np.array([0.0]),
             "router_w2": np.array([2.0]), "router_b2": np.array([0.5])}
        s = O.router_scores(np.array([[3.0, 7.0]]), W)
        assert s[0] == pytest.approx(2 * 3 / (1 + math.exp(-3)) + 0.5, rel=1e-15)

    @pytest.mark.parametrize("arch", [O.NEOX, O.QWEN])
    def test_r1_is_dense_and_r0_identity(self, arch):
        """K = T: every token kept -> the dense layer on the whole sequence;
        K = 0: every token bypasses -> identity, byte for byte."""
        p = _params(arch, Hkv=2 if arch == O.QWEN else 4)
        W = _weights(p, 14)
        x = rng(15).normal(size=(2, 11, 32))
        out, idx, _ = O.sparse_layer_forward(x, W, p, 11)
        for b in range(2):
            dense = x[b] + O.block_delta(x[b], np.arange(11), W, p)
            assert out[b] == pytest.approx(dense, rel=1e-13, abs=1e-13)
        out0, idx0, _ = O.sparse_layer_forward(x, W, p, 0)
        assert idx0.shape == (2, 0) and np.array_equal(out0.view(np.uint64), x.view(np.uint64))

    @pytest.mark.parametrize("arch", [O.NEOX, O.QWEN])
    def test_skipped_rows_untouched_and_kept_rows_follow_router(self, arch):
        p = _params(arch)
        W = _weights(p, 16)
        x = rng(17).normal(size=(3, 13, 32))
        out, idx, sc = O.sparse_layer_forward(x, W, p, 5)
        for b in range(3):
            assert idx[b].tolist() == _brute_topk(list(sc[b]), 5)
            skip = np.setdiff1d(np.arange(13), idx[b])
            assert np.array_equal(out[b, skip].view(np.uint64), x[b, skip].view(np.uint64))
            assert not np.allclose(out[b, idx[b]], x[b, idx[b]])

    @pytest.mark.parametrize("arch", [O.NEOX, O.QWEN])
    def test_position_shift_invariance(self, arch):
        """Positions enter only through RoPE, whose scores depend on position
        differences: shifting every kept position by c leaves the delta unchanged,
        while permuting the gaps changes it."""
        p = _params(arch)
        W = _weights(p, 18)
        xp = rng(19).normal(size=(6, 32))
        pos = np.array([0, 2, 3, 7, 8, 12])
        a = O.block_delta(xp, pos, W, p)
        b = O.block_delta(xp, pos + 37, W, p)
        c = O.block_delta(xp, np.array([0, 1, 2, 3, 4, 5]), W, p)
        assert a == pytest.approx(b, rel=1e-9, abs=1e-11)
        assert not np.allclose(a, c)

    def test_neox_closed_form_zero_projections(self):
        """W_qkv = 0 and W_up = 0: every value row is b_v, so attention returns
        b_v whatever the scores; delta = W_o b_v + b_o + W_down GELU(b_up) + b_down."""
        p = _params(O.NEOX)
        W = _weights(p, 20, zero=("w_qkv", "w_up"))
        xp = rng(21).normal(size=(5, 32))
        bv = W["b_qkv"][64:96]
        expect = W["w_o"] @ bv + W["b_o"] + W["w_down"] @ O.gelu(W["b_up"]) + W["b_down"]
        got = O.block_delta(xp, np.arange(5), W, p)
        for i in range(5):
            assert got[i] == pytest.approx(expect, rel=1e-12, abs=1e-13)

    def test_qwen_closed_form_zero_projections(self):
        """W_qkv = 0, W_gate = 0: query head h returns value head h // 2 (= b_v of
        that head), h = x + W_o o and SiLU(0) = 0 kills the MLP, so delta = W_o o."""
        p = _params(O.QWEN, Hkv=2)
        W = _weights(p, 22, zero=("w_qkv", "w_gate"))
        xp = rng(23).normal(size=(4, 32))
        bv = W["b_qkv"][32 + 16:32 + 32]
        got = O.block_delta(xp, np.arange(4), W, p)
        for i in range(4):
            o = np.concatenate([bv[:8], bv[:8], bv[8:], bv[8:]])
            assert got[i] == pytest.approx(W["w_o"] @ o, rel=1e-12)

    @pytest.mark.parametrize("arch", [O.NEOX, O.QWEN])
    def test_causality(self, arch):
        """Changing the last kept token leaves the earlier outputs unchanged."""
        p = _params(arch)
        W = _weights(p, 24)
        xp = rng(25).normal(size=(7, 32))
        a = O.block_delta(xp, np.arange(7), W, p)
        xq = xp.copy(); xq[-1] += rng(27).normal(size=32)   # not a constant shift: LayerNorm ignores those
        b = O.block_delta(xq, np.arange(7), W, p)
        assert a[:-1] == pytest.approx(b[:-1], rel=1e-13, abs=1e-14)
        assert not np.allclose(a[-1], b[-1])

    def test_model_special_cases(self):
        """All K = 0: the model is final_norm(embedding); statistics are cos = 1.
        All K = T: the model is the dense stack."""
        p = _params(O.NEOX)
        g = rng(26)
        Wm = {"embed": g.normal(size=(50, 32)), "final_w": 1 + g.normal(0, .1, 32), "final_b": g.normal(0, .1, 32)}
        layers = [_weights(p, 30 + l) for l in range(3)]
        ids = g.integers(0, 50, size=(2, 9))
        h, kept, st = O.sparse_model_forward(ids, Wm, layers, p, [0, 0, 0], stats_mode="token")
        assert h == pytest.approx(O.layer_norm(Wm["embed"][ids], Wm["final_w"], Wm["final_b"], 1e-5), rel=1e-13)
        assert all(O.similarity(s_) == pytest.approx(1.0, abs=1e-14) for s_ in st)
        h, kept, _ = O.sparse_model_forward(ids, Wm, layers, p, [9, 9, 9])
        x = Wm["embed"][ids]
        for W in layers:
            x = np.stack([x[b] + O.block_delta(x[b], np.arange(9), W, p) for b in range(2)])
        assert h == pytest.approx(O.layer_norm(x, Wm["final_w"], Wm["final_b"], 1e-5), rel=1e-12)


# ---------------------------------------------------------------- Eqs. 1-3: how the layer composes
def _tiny(arch):
    """One head of width 2 on d = 2, FFN width 2, norm eps 0, full rotary."""
    return {"arch": arch, "d": 2, "n_heads": 1, "n_kv_heads": 1, "head_dim": 2, "ffn": 2,
            "rotary_dim": 2, "rope_theta": 1e4, "norm_eps": 0.0}


_ROUTER_ONLY = {"router_w1": np.ones((1, 2)), "router_b1": np.zeros(1), "router_w2": np.ones(1),
                "router_b2": np.zeros(1)}   # K = 0: the layer only scores its tokens


class TestComposition:
    """Hand-worked single-token layers. One token attends only to itself, so
    attention returns its value row exactly (softmax of one score) and rotary
    angles do not matter; every other step is worked out below with distinct
    norm gains and non-symmetric weights, so that swapping the two norms of
    GPT-NeoX, the gate and up roles of SwiGLU, or the input of Qwen's second
    RMSNorm changes the result."""

    def test_neox_parallel_branches(self):
        """x = (3, 1): mean 2, variance 1, so LayerNorm gives (1, -1) before the
        affine step.
        LN1: gain (2, 3), bias (0.5, -1)  -> n1 = (2.5, -4)
        LN2: gain (1, 0.5), bias (-1, 2)  -> n2 = (0, 1.5)
        attention: V = I n1 + 0 = (2.5, -4); W_o = [[1, 1], [0, 2]], b_o = (0.25, 0)
                   -> attn = (2.5 - 4 + 0.25, -8) = (-1.25, -8)
        MLP: up = I n2 + 0 = (0, 1.5); GELU -> (0, 1.5 Phi(1.5)) = (0, 1.3997891980967129)
             W_down = I, b_down = (0, 0.5) -> mlp = (0, 1.8997891980967129)
        delta = attn + mlp = (-1.25, -6.1002108019032871).
        With LN1 and LN2 swapped the result would be (4.2345, 3.4999)."""
        p = _tiny(O.NEOX)
        W = {"ln1_w": np.array([2.0, 3.0]), "ln1_b": np.array([0.5, -1.0]),
             "ln2_w": np.array([1.0, 0.5]), "ln2_b": np.array([-1.0, 2.0]),
             "w_qkv": np.vstack([np.array([[0.3, -0.7], [1.1, 0.2]]),       # q
                                 np.array([[-0.4, 0.9], [0.6, 0.5]]),       # k
                                 np.eye(2)]),                               # v
             "b_qkv": np.array([0.1, -0.2, 0.3, 0.05, 0.0, 0.0]),
             "w_o": np.array([[1.0, 1.0], [0.0, 2.0]]), "b_o": np.array([0.25, 0.0]),
             "w_up": np.eye(2), "b_up": np.zeros(2),
             "w_down": np.eye(2), "b_down": np.array([0.0, 0.5])}
        got = O.block_delta(np.array([[3.0, 1.0]]), np.array([5]), W, p)
        assert got[0] == pytest.approx([-1.25, -6.1002108019032871], rel=1e-14)

    def test_qwen_sequential_residual(self):
        """x = (1, -1): RMS 1.
        RMS1 gain (2, 3) -> n1 = (2, -3)
        attention: V = I n1 + (0.5, 0) = (2.5, -3); W_o = [[1, 0], [1, 1]]
                   -> attn = (2.5, -0.5); h = x + attn = (3.5, -1.5), RMS(h) = sqrt(7.25)
        RMS2 of h, gain (1, 2) -> n2 = (a, b), a = 3.5/sqrt(7.25) = 1.2998673672393630,
                                  b = 2 (-1.5)/sqrt(7.25) = -1.1141720290623112
        gate = W_gate n2, W_gate = [[1, 0], [0, 0.5]] -> (a, b/2)
        up   = W_up n2,   W_up   = [[0, 1], [2, 0]]   -> (b, 2a)
        act = SiLU(gate) * up = (SiLU(a) b, SiLU(b/2) 2a)
            = (-1.1380735080494927, -0.52749388389216593)
        W_down = I: delta = attn + act = (1.3619264919505073, -1.0274938838921659).
        Swapping gate and up gives act = (-0.3579, -1.3481); RMS2 of x instead
        of h gives n2 = (1, -2)."""
        p = _tiny(O.QWEN)
        W = {"ln1_w": np.array([2.0, 3.0]), "ln2_w": np.array([1.0, 2.0]),
             "w_qkv": np.vstack([np.array([[0.3, -0.7], [1.1, 0.2]]),
                                 np.array([[-0.4, 0.9], [0.6, 0.5]]),
                                 np.eye(2)]),
             "b_qkv": np.array([0.1, -0.2, 0.3, 0.05, 0.5, 0.0]),
             "w_o": np.array([[1.0, 0.0], [1.0, 1.0]]),
             "w_gate": np.array([[1.0, 0.0], [0.0, 0.5]]), "w_up": np.array([[0.0, 1.0], [2.0, 0.0]]),
             "w_down": np.eye(2)}
        got = O.block_delta(np.array([[1.0, -1.0]]), np.array([9]), W, p)
        assert got[0] == pytest.approx([1.3619264919505073, -1.0274938838921659], rel=1e-14)

    def test_qwen_final_norm(self):
        """All K = 0: the Qwen model returns RMSNorm(embedding) with the final
        gain. Row (3, 4): RMS = sqrt(12.5), normalised (0.84852813742385703,
        1.1313708498984760), gain (2, 0.5) -> (1.6970562748477141,
        0.56568542494923802)."""
        p = _tiny(O.QWEN)
        Wm = {"embed": np.array([[3.0, 4.0], [0.0, 0.0]]), "final_w": np.array([2.0, 0.5])}
        h, _, _ = O.sparse_model_forward(np.array([[0]]), Wm, [_ROUTER_ONLY], p, [0])
        assert h[0, 0] == pytest.approx([1.6970562748477141, 0.56568542494923802], rel=1e-14)
        ref = F.rms_norm(torch.tensor([[3.0, 4.0]], dtype=torch.float64), (2,),
                         torch.tensor([2.0, 0.5], dtype=torch.float64), eps=0.0)
        assert h[0] == pytest.approx(ref.numpy(), rel=1e-14)

    def test_neox_final_norm_matches_torch(self):
        p = _tiny(O.NEOX)
        p["norm_eps"] = 1e-5
        g = rng(40)
        Wm = {"embed": g.normal(size=(7, 2)), "final_w": 1 + g.normal(0, 0.3, 2), "final_b": g.normal(0, 0.3, 2)}
        ids = np.array([[3, 0, 6, 6]])
        h, _, _ = O.sparse_model_forward(ids, Wm, [_ROUTER_ONLY], p, [0])
        ref = F.layer_norm(torch.from_numpy(Wm["embed"][ids]), (2,), torch.from_numpy(Wm["final_w"]),
                           torch.from_numpy(Wm["final_b"]), eps=1e-5)
        assert h == pytest.approx(ref.numpy(), rel=1e-13)

    def test_linear_orientation_bias_and_gelu(self):
        """W stored [out, in]: x = (1, -1), W = [[1, 2], [0, 3]], b = (0, 0)
        -> x W^T = (-1, -3) (the transposed product would give (1, -1));
        GELU: (-Phi(-1), -3 Phi(-3)) = (-0.15865525393145705, -0.0040496940948902836).
        With bias (0.5, -1): (11.5, 16) for x = (1, 2), W = [[3, 4], [5, 6]]."""
        y = O.linear(np.array([[1.0, -1.0]]), np.array([[1.0, 2.0], [0.0, 3.0]]))
        assert y[0].tolist() == [-1.0, -3.0]
        g_ = O.linear(np.array([[1.0, -1.0]]), np.array([[1.0, 2.0], [0.0, 3.0]]), act="gelu")
        assert g_[0] == pytest.approx([-0.15865525393145705, -0.0040496940948902836], rel=1e-14)
        b = O.linear(np.array([[1.0, 2.0]]), np.array([[3.0, 4.0], [5.0, 6.0]]), np.array([0.5, -1.0]))
        assert b[0].tolist() == [11.5, 16.0]


# ---------------------------------------------------------------- Sec. 3.4: score-gated variant
class TestGate:
    """Kept rows get x + sigmoid(score) delta in the gated variant."""

    def test_hand_worked_single_token(self):
        """The NeoX single-token layer of TestComposition (delta =
        (-1.25, -6.1002108019032871)) with a router whose hidden unit is
        SiLU(0 . x + 1) = SiLU(1) = 0.73105857863000488 and score
        2 SiLU(1) - 0.5 = 0.96211715726000976; sigmoid of it is
        0.72354549497730215, so the gated delta is
        (-0.90443186872162769, -4.4137800441289991)."""
        p = _tiny(O.NEOX)
        p["gate"] = "sigmoid"
        W = {"router_w1": np.zeros((1, 2)), "router_b1": np.array([1.0]), "router_w2": np.array([2.0]),
             "router_b2": np.array([-0.5]),
             "ln1_w": np.array([2.0, 3.0]), "ln1_b": np.array([0.5, -1.0]),
             "ln2_w": np.array([1.0, 0.5]), "ln2_b": np.array([-1.0, 2.0]),
             "w_qkv": np.vstack([np.array([[0.3, -0.7], [1.1, 0.2]]), np.array([[-0.4, 0.9], [0.6, 0.5]]),
                                 np.eye(2)]),
             "b_qkv": np.array([0.1, -0.2, 0.3, 0.05, 0.0, 0.0]),
             "w_o": np.array([[1.0, 1.0], [0.0, 2.0]]), "b_o": np.array([0.25, 0.0]),
             "w_up": np.eye(2), "b_up": np.zeros(2),
             "w_down": np.eye(2), "b_down": np.array([0.0, 0.5])}
        x = np.array([[[3.0, 1.0]]])
        out, idx, sc = O.sparse_layer_forward(x, W, p, 1)
        assert sc[0, 0] == pytest.approx(0.96211715726000976, rel=1e-15)
        assert out[0, 0] - x[0, 0] == pytest.approx([-0.90443186872162769, -4.4137800441289991], rel=1e-14)

    @pytest.mark.parametrize("arch", [O.NEOX, O.QWEN])
    def test_constant_score_scales_every_delta(self, arch):
        """A router with w2 = 0 gives every token the score b2: score 0 halves
        every kept row's delta (sigmoid(0) = 1/2); a large score recovers the
        ungated layer; skipped rows stay untouched either way."""
        p = _params(arch, Hkv=2 if arch == O.QWEN else 4)
        W = _weights(p, 41)
        x = rng(42).normal(size=(2, 9, 32))
        idx = np.array([[0, 2, 3, 7], [1, 4, 5, 8]])
        plain, _, _ = O.sparse_layer_forward(x, W, p, 4, idx=idx)
        pg = dict(p, gate="sigmoid")
        for b2, factor in ((0.0, 0.5), (60.0, 1.0)):
            Wc = dict(W, router_w2=np.zeros_like(W["router_w2"]), router_b2=np.array([b2]))
            got, _, _ = O.sparse_layer_forward(x, Wc, pg, 4, idx=idx)
            assert got - x == pytest.approx(factor * (plain - x), rel=1e-12, abs=1e-14)
            for b in range(2):
                skip = np.setdiff1d(np.arange(9), idx[b])
                assert np.array_equal(got[b, skip].view(np.uint64), x[b, skip].view(np.uint64))

    def test_sigmoid(self):
        assert O.sigmoid(0.0) == 0.5
        assert O.sigmoid(np.log(3.0)) == pytest.approx(0.75, rel=1e-15)
        assert O.sigmoid(-np.log(3.0)) == pytest.approx(0.25, rel=1e-15)


# ---------------------------------------------------------------- Sec. 4.1: normalized FLOPs
class TestNormalizedFlops:
    P = {"arch": O.NEOX, "d": 4, "n_heads": 1, "n_kv_heads": 1, "head_dim": 4, "ffn": 8,
         "rotary_dim": 4, "rope_theta": 1e4, "norm_eps": 1e-5}

    def test_hand_counted(self):
        """d = 4, one head of 4, FFN 8, GELU MLP, T = 4, router width 2.
        Per token the projections take 12*4 (QKV) + 4*4 (output) + 2*4*8 (MLP)
        = 128 multiply-adds = 256 flops; causal attention on K tokens takes
        2 * 4 * K (K + 1) flops. K = 4: 1024 + 160 = 1184; K = 2: 512 + 48 = 560.
        The router on 4 tokens: 2 * 4 * 2 * (4 + 1) = 80.
        Layers K = (2, 4): (80 + 560 + 1184) / (2 * 1184) = 1824 / 2368."""
        assert O.block_flops(self.P, 4) == 1184
        assert O.block_flops(self.P, 2) == 560
        assert O.router_flops(self.P, 4, h=2) == 80
        assert O.normalized_flops(self.P, 4, [2, 4], h=2) == pytest.approx(1824 / 2368, rel=1e-15)

    def test_limits(self):
        """Every token kept: exactly 1 (no router counted, nothing dropped);
        none kept: the routers' share alone."""
        assert O.normalized_flops(self.P, 4, [4, 4, 4], h=2) == 1.0
        assert O.normalized_flops(self.P, 4, [0, 0], h=2) == pytest.approx(80 / 1184, rel=1e-15)

    def test_swiglu_counts_three_mlp_matrices(self):
        """The Qwen form adds the gate matrix: 2 * 4 * 8 more multiply-adds a token."""
        q = dict(self.P, arch=O.QWEN)
        assert O.block_flops(q, 4) - O.block_flops(self.P, 4) == 2 * 4 * 4 * 8


# ---------------------------------------------------------------- decode with a kept-token cache
class TestDecode:
    """Generation reading: a new token is kept at layer l iff its router score
    beats the lowest kept prompt score of that layer; kept tokens attend to
    the layer's kept tokens and join them."""

    def _model(self, arch, seed):
        p = _params(arch, Hkv=2 if arch == O.QWEN else 4)
        g = rng(seed)
        Wm = {"embed": g.normal(size=(30, 32)), "final_w": 1 + g.normal(0, .1, 32)}
        if arch == O.NEOX:
            Wm["final_b"] = g.normal(0, .1, 32)
        layers = [_weights(p, seed + 1 + l) for l in range(3)]
        return p, Wm, layers

    @pytest.mark.parametrize("arch", [O.NEOX, O.QWEN])
    def test_matches_sparse_forward_on_the_extended_sequence(self, arch):
        """Prompt of 10, two decoded tokens; per sequence, the decoded token's
        output equals the last row of the sparse model on the extended
        sequence with each layer's kept set = the prompt's kept set plus the
        new token where it was kept (causality makes the two the same)."""
        p, Wm, layers = self._model(arch, 50)
        ids = rng(51).integers(0, 30, size=(3, 12))
        K = [6, 3, 8]
        _, st = O.sparse_prefill(ids[:, :10], Wm, layers, p, K)
        decided = [[list(st["pos"][l][b]) for b in range(3)] for l in range(3)]
        n_kept = 0
        for t in (10, 11):
            h, kept, _ = O.decode_step(ids[:, t], Wm, layers, p, st)
            n_kept += kept.sum()
            for l in range(3):
                for b in range(3):
                    if kept[l, b]:
                        decided[l][b].append(t)
            for b in range(3):
                force = [np.array([decided[l][b]]) for l in range(3)]
                ref, _, _ = O.sparse_model_forward(ids[b:b + 1, :t + 1], Wm, layers, p,
                                                   [len(f[0]) for f in force], idx_force=force)
                assert h[b] == pytest.approx(ref[0, -1], rel=1e-12, abs=1e-12)
        assert 0 < n_kept < 2 * 3 * 3          # some kept, some skipped

    def test_always_kept_is_the_dense_model(self):
        """Thresholds -inf (every token kept) and a dense prompt: the decoded
        token's output is the dense model's last row on the extended sequence."""
        p, Wm, layers = self._model(O.NEOX, 60)
        ids = rng(61).integers(0, 30, size=(2, 8))
        _, st = O.sparse_prefill(ids[:, :7], Wm, layers, p, [7, 7, 7])
        st["thr"] = [[-np.inf] * 2 for _ in range(3)]
        h, kept, _ = O.decode_step(ids[:, 7], Wm, layers, p, st)
        assert kept.all()
        x = np.asarray(Wm["embed"])[ids]
        for W in layers:
            x = np.stack([x[b] + O.block_delta(x[b], np.arange(8), W, p) for b in range(2)])
        dense = O.layer_norm(x, Wm["final_w"], Wm["final_b"], p["norm_eps"])
        assert h == pytest.approx(dense[:, -1], rel=1e-12, abs=1e-12)

    def test_never_kept_bypasses_every_layer(self):
        p, Wm, layers = self._model(O.QWEN, 70)
        ids = rng(71).integers(0, 30, size=(2, 6))
        _, st = O.sparse_prefill(ids[:, :5], Wm, layers, p, [2, 2, 2])
        st["thr"] = [[np.inf] * 2 for _ in range(3)]
        h, kept, _ = O.decode_step(ids[:, 5], Wm, layers, p, st)
        assert not kept.any()
        assert h == pytest.approx(O.rms_norm(np.asarray(Wm["embed"])[ids[:, 5]], Wm["final_w"], p["norm_eps"]),
                                  rel=1e-14)
        assert [len(r) for r in st["rows"][0]] == [2, 2]          # nothing joined the cache

    def test_threshold_and_keep_rule(self):
        """The threshold is the K-th largest score; a tie loses (the later
        position loses Top-K ties); NaN never wins."""
        sc = np.array([0.5, 2.0, -1.0, 2.0, 0.7])
        idx = O.topk_keep(sc, 3)
        assert O.kept_threshold(sc, idx) == 0.7
        assert O.decode_keep(0.71, 0.7) and not O.decode_keep(0.7, 0.7)
        assert not O.decode_keep(float("nan"), 0.7) and not O.decode_keep(float("nan"), -np.inf)
        assert O.kept_threshold(sc, []) == np.inf              # nothing kept: nothing will be


# ---------------------------------------------------------------- Sec. 3.5, Eqs. 9-11; router gradient
class TestAlignment:
    def test_softmax_matches_scipy(self):
        from scipy.special import softmax as sp_softmax
        z = rng(80).normal(size=(5, 9)) * 4
        assert O.softmax(z) == pytest.approx(sp_softmax(z, axis=-1), rel=1e-14)

    def test_hidden_alignment_hand_value_and_limits(self):
        """h_s = (0, 0) -> p = (1/2, 1/2); h_d = (ln 3, 0) -> q = (3/4, 1/4);
        |p - q| = sqrt(2) / 4. Identical rows give 0; adding a constant to a
        row changes nothing (the softmax is shift invariant)."""
        hs = np.array([[0.0, 0.0]])
        hd = np.array([[math.log(3.0), 0.0]])
        assert O.hidden_alignment(hs, hd)[0] == pytest.approx(math.sqrt(2) / 4, rel=1e-15)
        x = rng(81).normal(size=(4, 16))
        assert O.hidden_alignment(x, x) == pytest.approx(np.zeros(4), abs=1e-15)
        y = rng(82).normal(size=(4, 16))
        assert O.hidden_alignment(x + 3.0, y - 1.5) == pytest.approx(O.hidden_alignment(x, y), rel=1e-12)

    def test_hidden_alignment_grad_matches_finite_differences_and_autograd(self):
        hs = rng(83).normal(size=(3, 7))
        hd = rng(84).normal(size=(3, 7))
        g = O.hidden_alignment_grad(hs, hd)
        eps = 1e-6
        fd = np.zeros_like(hs)
        for i in range(hs.shape[0]):
            for j in range(hs.shape[1]):
                a, b = hs.copy(), hs.copy()
                a[i, j] += eps
                b[i, j] -= eps
                fd[i, j] = (O.hidden_alignment(a, hd)[i] - O.hidden_alignment(b, hd)[i]) / (2 * eps)
        assert g == pytest.approx(fd, rel=1e-6, abs=1e-9)
        t = torch.tensor(hs, requires_grad=True)
        loss = torch.linalg.vector_norm(torch.softmax(t, -1) - torch.softmax(torch.tensor(hd), -1), dim=-1).sum()
        loss.backward()
        assert g == pytest.approx(t.grad.numpy(), rel=1e-12, abs=1e-15)

    def test_output_alignment(self):
        """W_head = I: logits are the hidden rows. P_s = (1/2, 1/2), P_d = (3/4, 1/4):
        KL = 3/4 ln(3/2) + 1/4 ln(1/2) = 0.13081203594113694. KL(P || P) = 0,
        KL >= 0, and agreement with scipy.special.rel_entr."""
        from scipy.special import rel_entr, softmax as sp_softmax
        kl = O.output_alignment(np.array([[0.0, 0.0]]), np.array([[math.log(3.0), 0.0]]), np.eye(2))
        assert kl[0] == pytest.approx(0.75 * math.log(1.5) + 0.25 * math.log(0.5), rel=1e-14)
        assert kl[0] == pytest.approx(0.13081203594113694, rel=1e-14)
        g = rng(85)
        W = g.normal(size=(30, 8))
        hs, hd = g.normal(size=(6, 8)), g.normal(size=(6, 8))
        assert O.output_alignment(hs, hs, W) == pytest.approx(np.zeros(6), abs=1e-14)
        got = O.output_alignment(hs, hd, W)
        ref = rel_entr(sp_softmax(hd @ W.T, axis=-1), sp_softmax(hs @ W.T, axis=-1)).sum(-1)
        assert got == pytest.approx(ref, rel=1e-12) and (got >= 0).all()

    def test_objective(self):
        assert O.alignment_objective(0.1, [0.2, 0.4]) == pytest.approx(0.4, rel=1e-15)

    @pytest.mark.parametrize("arch", [O.NEOX, O.QWEN])
    def test_router_grad_through_the_gated_layer(self, arch):
        """L(theta) = sum over kept rows of grad_y . y, y the gated layer's
        output with the kept set held fixed: its finite-difference gradient in
        every router parameter equals router_grad (delta = the ungated layer's
        delta); and torch autograd of the same expression agrees."""
        p = dict(_params(arch, Hkv=2 if arch == O.QWEN else 4), gate="sigmoid")
        W = _weights(p, 86)
        x = rng(87).normal(size=(2, 9, 32))
        idx = np.array([[0, 3, 4, 8], [1, 2, 6, 7]])
        rows = (np.arange(2)[:, None] * 9 + idx).ravel()
        G = rng(88).normal(size=(8, 32))
        plain, _, _ = O.sparse_layer_forward(x, W, dict(p, gate="none"), 4, idx=idx)
        delta = (plain - x).reshape(-1, 32)[rows]
        got = O.router_grad(x, W, rows, delta, G)

        def loss(Wr):
            y, _, _ = O.sparse_layer_forward(x, Wr, p, 4, idx=idx)
            return float((G * y.reshape(-1, 32)[rows]).sum())

        eps = 1e-6
        for name in ("router_w1", "router_b1", "router_w2", "router_b2"):
            fd = np.zeros_like(W[name])
            flat = fd.reshape(-1)
            for k in range(flat.size):
                a = {kk: vv.copy() for kk, vv in W.items()}
                b = {kk: vv.copy() for kk, vv in W.items()}
                a[name].reshape(-1)[k] += eps
                b[name].reshape(-1)[k] -= eps
                flat[k] = (loss(a) - loss(b)) / (2 * eps)
            assert got[name] == pytest.approx(fd, rel=1e-5, abs=1e-8), name
        # autograd of sum G . (x + sigmoid(s) delta) over the router parameters
        tw = {k: torch.tensor(W[k], requires_grad=True) for k in ("router_w1", "router_b1", "router_w2", "router_b2")}
        xs = torch.tensor(x.reshape(-1, 32)[rows])
        s = torch.nn.functional.silu(xs @ tw["router_w1"].T + tw["router_b1"]) @ tw["router_w2"] + tw["router_b2"][0]
        (torch.tensor(G) * (xs + torch.sigmoid(s)[:, None] * torch.tensor(delta))).sum().backward()
        for k, t in tw.items():
            assert got[k] == pytest.approx(t.grad.numpy(), rel=1e-12, abs=1e-14), k
