"""Host-side checks of the C ABI (no GPU needed): the library loads and exports
every declared entry point, the host-only allocation (Sec. 3.3, Eqs. 5-8)
matches the oracle, and argument errors are reported before any launch."""
import ctypes
import os
import re

import numpy as np
import pytest

from oracle import adadsf_oracle as O
from paper_2607_21291_gb300 import build as B
from paper_2607_21291_gb300 import synth as S

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def A():
    B.build()
    from paper_2607_21291_gb300 import adadsf
    adadsf.lib()
    return adadsf


def _declared():
    names = set()
    inc = os.path.join(ROOT, "include")
    for f in os.listdir(inc):
        if f.endswith(".h"):
            src = open(os.path.join(inc, f)).read()
            src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
            names |= set(re.findall(r"\b(adadsf_\w+)\s*\(", src))
    return sorted(names)


def test_exports_every_declared_symbol(A):
    names = _declared()
    assert len(names) >= 14
    raw = ctypes.CDLL(A.LIB_PATH)
    for n in names:
        assert hasattr(raw, n), n


def test_alloc_matches_oracle(A):
    g = np.random.default_rng(0)
    for L in (1, 2, 4, 12, 24, 28):
        for t in (0.25, 0.5, 0.75, 0.95, 1.0):
            for tau in (0.25, 0.1, 0.05):
                s = g.uniform(0.5, 1.0, L)
                for T in (128, 512, 4096):
                    r, K = A.adadsf_alloc_ratios(s, t, tau, 10.0, T)
                    ro, _ = O.allocate_ratios(s, t, tau, 10.0)
                    assert r == pytest.approx(ro, rel=1e-12, abs=1e-15)
                    assert K.tolist() == O.kept_counts(ro, T).tolist()
                    rr, _ = A.adadsf_alloc_ratios(s, t, tau, 10.0, T, A.ALLOC_RAW)
                    assert rr == pytest.approx(O.allocate_ratios(s, t, tau, 10.0, raw=True)[0], rel=1e-12)
                    _, Kr = A.adadsf_alloc_ratios(s, t, tau, 10.0, T, A.ALLOC_ROUND)
                    assert Kr.tolist() == O.kept_counts(ro, T, "round").tolist()


def test_similarity_matches_oracle(A):
    """Eq. 4's final step on the host: s_l from accumulated partial sums, in
    both aggregation modes, against the oracle's cos_sim_stat / similarity."""
    g = np.random.default_rng(3)
    tok, flat = [], []
    for l in range(5):
        a = g.standard_normal((40, 16))
        b = a + (0.2 + 0.3 * l) * g.standard_normal((40, 16))
        tok.append(O.cos_sim_stat(a, b))
        flat.append(O.cos_sim_stat(a, b, "flat"))
    assert A.adadsf_similarity(np.array(tok)) == pytest.approx([O.similarity(t) for t in tok], rel=1e-15)
    assert A.adadsf_similarity(np.array(flat), A.STATS_FLAT) == pytest.approx(
        [O.similarity(f, "flat") for f in flat], rel=1e-15)
    with pytest.raises(A.AdadsfError):
        A.adadsf_similarity(np.array([[1.0, 0.0]]))                # no tokens counted
    with pytest.raises(ValueError):
        A.adadsf_similarity(np.zeros(3))                           # not [L, 2]


def test_normalized_flops_matches_oracle(A):
    g = np.random.default_rng(4)
    for key in ("c1", "c2", "c3", "c4", "c5"):
        wl = S.WORKLOADS[key]
        shape = wl.shape
        for K in ([wl.T] * shape.n_layers, [0] * shape.n_layers,
                  g.integers(0, wl.T + 1, shape.n_layers).tolist()):
            got = A.adadsf_normalized_flops(A.make_cfg(shape), wl.T, K)
            assert got == pytest.approx(O.normalized_flops(O.params_of(shape), wl.T, K, shape.router_hidden),
                                        rel=1e-13)
    with pytest.raises(A.AdadsfError):
        A.adadsf_normalized_flops(A.make_cfg(S.PYTHIA_160M), 100, [101] * 12)


def test_alloc_rejects_bad_args(A):
    with pytest.raises(A.AdadsfError):
        A.adadsf_alloc_ratios([0.5, 0.6], 1.5)
    with pytest.raises(A.AdadsfError):
        A.adadsf_alloc_ratios([0.5, float("nan")], 0.5)
    with pytest.raises(A.AdadsfError):
        A.adadsf_alloc_ratios([0.5, 0.6], 0.5, tau=0.0)


def test_workspace_sizes(A):
    for key in ("c1", "c2", "c3", "c4", "c5"):
        wl = S.WORKLOADS[key]
        cfg = A.make_cfg(wl.shape)
        K = wl.T // 2
        n = A.adadsf_layer_workspace_size(cfg, wl.B, wl.T, K)
        assert n % 256 == 0 and n > wl.B * K * wl.shape.ffn * (2 if wl.shape.dtype == "bf16" else 4)
        m = A.adadsf_model_workspace_size(cfg, wl.B, wl.T, [K] * wl.shape.n_layers, True)
        assert m > n
    cfg = A.make_cfg(S.PYTHIA_160M)
    with pytest.raises(A.AdadsfError):
        A.adadsf_layer_workspace_size(cfg, 2, 100, 101)          # K > T
    bad = A.make_cfg(S.PYTHIA_160M.replace(head_dim=96))
    with pytest.raises(A.AdadsfError):
        A.adadsf_layer_workspace_size(bad, 2, 100, 50)
    assert "head_dim" in A.adadsf_last_error()


def test_flags_and_their_workspace(A):
    """FLAG_GATHERED_QKV is accepted with or without FLAG_FOLDED_NORMS; it
    adds exactly one fp32 sum of squares per token (B T floats, 256-byte
    aligned) to a bf16 Qwen layer's workspace, and only together with
    FLAG_FOLDED_NORMS (alone it is ignored); unknown flag bits are refused."""
    B, T, K = 4, 1000, 500
    for shape, grows in ((S.QWEN25_1_5B, True), (S.PYTHIA_160M, False)):
        sizes = {f: A.adadsf_layer_workspace_size(A.make_cfg(shape, f), B, T, K)
                 for f in (0, A.FLAG_FOLDED_NORMS, A.FLAG_GATHERED_QKV,
                           A.FLAG_FOLDED_NORMS | A.FLAG_GATHERED_QKV)}
        assert sizes[A.FLAG_FOLDED_NORMS] == sizes[0] == sizes[A.FLAG_GATHERED_QKV]
        extra = sizes[A.FLAG_FOLDED_NORMS | A.FLAG_GATHERED_QKV] - sizes[0]
        assert extra == ((B * T * 4 + 255) // 256 * 256 if grows else 0)
    with pytest.raises(A.AdadsfError):
        A.adadsf_layer_workspace_size(A.make_cfg(S.QWEN25_1_5B, 8), B, T, K)


def test_argument_errors_precede_launch(A):
    lib = A.lib()
    cfg = A.make_cfg(S.PYTHIA_160M)
    assert lib.adadsf_topk_select(None, 2, 10, 11, None, None, None) == A.ERR_INVALID_ARG
    assert lib.adadsf_topk_select(None, 2, 10, 0, None, None, None) == A.OK        # K = 0: nothing
    assert lib.adadsf_sparse_layer_forward(ctypes.byref(cfg), None, None, 2, 16, 0, None, None,
                                           None, 0, None) == A.OK                    # K = 0: nothing
    assert lib.adadsf_sparse_layer_forward(ctypes.byref(cfg), None, None, 2, 16, 8, None, None,
                                           None, 0, None) == A.ERR_INVALID_ARG
    assert lib.adadsf_linear(None, None, None, 4, 100, 64, A.BF16, 0, None, None, 0, None) == A.ERR_UNSUPPORTED
    assert lib.adadsf_router_select(ctypes.byref(cfg), None, None, 2, 16, 4, None, None, None, None, 0,
                                    None) == A.ERR_INVALID_ARG
    assert lib.adadsf_router_select_workspace_size(ctypes.byref(cfg), 4, 512) > 256 + 4 * (16 + 4)
    assert lib.adadsf_layer_stats(None, None, 4, 64, A.BF16, 0, None, None, 0, None) == A.ERR_INVALID_ARG


def test_decode_argument_errors_precede_launch(A):
    lib = A.lib()
    cfg = A.make_cfg(S.PYTHIA_160M)
    n = lib.adadsf_kv_cache_size(ctypes.byref(cfg), 2, 100)
    # header + counts + thresholds + rotary table + K and V of 12 layers
    assert n >= 12 * 2 * (2 * 12 * 100 * 64 * 2)
    assert lib.adadsf_kv_cache_size(ctypes.byref(cfg), 0, 100) == 0
    # the prompt must leave room in the cache
    assert lib.adadsf_prefill(ctypes.byref(cfg), None, None, 2, 100, None, None, None, None, n, 100, None, 0,
                              None) == A.ERR_INVALID_ARG
    assert "C_max" in A.adadsf_last_error()
    buf = ctypes.create_string_buffer(1024)
    base = (ctypes.addressof(buf) + 255) & ~255
    assert lib.adadsf_prefill(ctypes.byref(cfg), None, None, 2, 50, None, None, None, base, 256, 100, None, 0,
                              None) == A.ERR_WORKSPACE_TOO_SMALL
    assert lib.adadsf_decode_step(ctypes.byref(cfg), None, None, 2, None, None, None, n, 100, None, 0,
                                  None) == A.ERR_INVALID_ARG
    assert lib.adadsf_decode_workspace_size(ctypes.byref(cfg), 2, 100) > 0
