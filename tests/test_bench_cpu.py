"""Host-side pieces of bench.py: the reference arm's JSON line (the fp64
oracle timed on the host cores) on a tiny stand-in workload, its rank
handling, and the lookup of recorded ncu traffic by kernel-source hash."""
import json
import os
import sys
import types

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
from paper_2607_21291_gb300 import synth as S  # noqa: E402

TINY = S.Workload("tiny-neox-B2-T24", S.PYTHIA_160M.replace(name="tiny", d=64, n_heads=2, n_kv_heads=2,
                                                            head_dim=32, ffn=128, n_layers=3, vocab=97,
                                                            rotary_dim=8),
                  2, 24, (0.5,), (2, 24))


def _args(**kw):
    a = dict(workload="c2", retention=None, warmup=3, steps=2)
    a.update(kw)
    return types.SimpleNamespace(**a)


def test_reference_arm_line(monkeypatch, capsys):
    monkeypatch.setitem(bench.S.WORKLOADS, "c2", TINY)
    bench.run_reference(_args(), 0, 1)
    lines = [l for l in capsys.readouterr().out.splitlines() if l.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["metric"] == bench.METRIC
    assert d["unit"] == "tokens/s" and d["value"] > 0 and d["higher_is_better"] is True
    assert d["n_gpus"] == 1 and d["steps"] == 2 and d["warmup"] == 3
    # one (sequence, layer) pair per step, extrapolated to all layers
    assert d["extrapolated"] is True
    assert d["ms_per_step"] == pytest.approx(TINY.T / (d["value"] * 3) * 1e3)
    # the workload's definition is the GPU arm's, key for key
    assert d["config"] == bench.shared_config(TINY, 0.5, 1)
    K = d["retention_plan"]["K_per_layer"]
    assert len(K) == 3 and all(0 <= k <= TINY.T for k in K)
    assert sum(K) == pytest.approx(0.5 * 3 * TINY.T, abs=3)
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["value"] == d["value"] and cb["cores"] >= 1 and cb["sample"]
    assert d["e2e"] == {"value": d["value"], "unit": "tokens/s", "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}


def test_reference_arm_other_ranks_do_no_work(monkeypatch, capsys):
    monkeypatch.setitem(bench.S.WORKLOADS, "c2", TINY)
    bench.run_reference(_args(), 1, 2)
    assert capsys.readouterr().out == ""


def test_reference_kept_counts_follow_oracle_allocation(monkeypatch, capsys):
    """The reference arm's K_l are the oracle's Eqs. 5-8 on the oracle's own
    Eq. 4 statistics, recomputed here from its printed similarities."""
    from oracle import adadsf_oracle as O
    monkeypatch.setitem(bench.S.WORKLOADS, "c2", TINY)
    bench.run_reference(_args(), 0, 1)
    d = json.loads(capsys.readouterr().out.strip().splitlines()[-1])
    s = d["retention_plan"]["similarity"]
    r, _ = O.allocate_ratios(s, 0.5, bench.TAU, bench.BETA)
    assert d["retention_plan"]["K_per_layer"] == O.kept_counts(r, TINY.T).tolist()


def test_layer_order_spreads_over_depth():
    for L in (1, 3, 12, 24, 28):
        o = bench.layer_order(L)
        assert sorted(o) == list(range(L))
        if L >= 12:     # any third of the order touches every third of the depth
            first = o[:L // 3]
            assert min(first) < L // 3 and max(first) >= 2 * L // 3


def test_counter_draws_match_on_any_subset():
    """The GPU arm draws whole tensors, the reference arm embedding rows: the
    same values either way."""
    import torch
    shape = TINY.shape
    E = S.bench_embed(shape, bench.WEIGHT_SEED)
    ids = S.counter_ids(bench.EVAL_SEED, 2, TINY.T, shape.vocab)
    assert int(ids.min()) >= 0 and int(ids.max()) < shape.vocab
    assert torch.equal(S.bench_embed_rows(shape, bench.WEIGHT_SEED, ids), E[ids.long()])


def test_host_threads():
    n = bench.host_threads()
    assert isinstance(n, int) and n >= 1


def test_recorded_traffic_needs_matching_sources(monkeypatch, tmp_path):
    (tmp_path / "profiles").mkdir()
    (tmp_path / "profiles" / "g.md").write_text(
        "header\ntraffic wl-a gemm 1.5e7 0123456789ab\ntraffic wl-b gemm 2.0e7 ba9876543210\n")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    monkeypatch.setattr(bench, "kernel_source_hash", lambda kind="": "0123456789ab")
    assert bench.recorded_traffic("gemm", "wl-a") == 1.5e7
    assert bench.recorded_traffic("gemm", "wl-b") is None     # taken on other sources
    assert bench.recorded_traffic("attention", "wl-a") is None
