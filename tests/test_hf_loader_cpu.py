"""The Hugging Face-layout checkpoint loader on small synthetic checkpoints
written here (GPT-NeoX single file, Qwen2 sharded with an index): names,
shapes, bf16 decoding, the regrouping of GPT-NeoX's per-head interleaved QKV
rows, and the loaded weights driving the oracle's layer."""
import json
import os
import struct

import numpy as np
import pytest

from oracle import adadsf_oracle as O
from paper_2607_21291_gb300 import hf_loader as HF
from paper_2607_21291_gb300 import synth as S


def _bf16_bits(a):
    return (S.round_to(np.asarray(a, np.float32), "bf16").view(np.uint32) >> 16).astype(np.uint16)


def write_safetensors(path, tensors, dtype="F32"):
    """Minimal writer of the safetensors container (header + raw bytes)."""
    header, blobs, off = {"__metadata__": {"format": "pt"}}, [], 0
    for name, a in tensors.items():
        raw = (_bf16_bits(a) if dtype == "BF16" else np.asarray(a, np.float32)).tobytes()
        header[name] = {"dtype": dtype, "shape": list(np.shape(a)), "data_offsets": [off, off + len(raw)]}
        blobs.append(raw)
        off += len(raw)
    h = json.dumps(header).encode()
    h += b" " * ((8 - len(h) % 8) % 8)
    with open(path, "wb") as f:
        f.write(struct.pack("<Q", len(h)))
        f.write(h)
        for b in blobs:
            f.write(b)


NEOX_CFG = {"model_type": "gpt_neox", "hidden_size": 64, "num_attention_heads": 2, "intermediate_size": 128,
            "num_hidden_layers": 2, "vocab_size": 50, "rotary_pct": 0.25, "rotary_emb_base": 10000,
            "layer_norm_eps": 1e-5, "use_parallel_residual": True, "hidden_act": "gelu"}
QWEN_CFG = {"model_type": "qwen2", "hidden_size": 64, "num_attention_heads": 4, "num_key_value_heads": 2,
            "intermediate_size": 96, "num_hidden_layers": 2, "vocab_size": 40, "rope_theta": 1e6,
            "rms_norm_eps": 1e-6, "hidden_act": "silu", "rope_scaling": None}


def _neox_ckpt(tmp_path, dtype):
    g = np.random.default_rng(0)
    d, H, hd, F, L, V = 64, 2, 32, 128, 2, 50
    t, per_head = {}, []
    for l in range(L):
        p = f"gpt_neox.layers.{l}."
        q, k, v = (g.normal(0, 0.1, (H, hd, d)) for _ in range(3))
        bq, bk, bv = (g.normal(0, 0.1, (H, hd)) for _ in range(3))
        # the checkpoint's fused rows: per head, its q rows, then k, then v
        t[p + "attention.query_key_value.weight"] = np.concatenate(
            [np.concatenate([q[h], k[h], v[h]], 0) for h in range(H)], 0)
        t[p + "attention.query_key_value.bias"] = np.concatenate(
            [np.concatenate([bq[h], bk[h], bv[h]]) for h in range(H)])
        per_head.append((q, k, v, bq, bk, bv))
        for n in ("input_layernorm", "post_attention_layernorm"):
            t[p + n + ".weight"] = 1 + g.normal(0, 0.1, d)
            t[p + n + ".bias"] = g.normal(0, 0.1, d)
        t[p + "attention.dense.weight"] = g.normal(0, 0.1, (d, d))
        t[p + "attention.dense.bias"] = g.normal(0, 0.1, d)
        t[p + "mlp.dense_h_to_4h.weight"] = g.normal(0, 0.1, (F, d))
        t[p + "mlp.dense_h_to_4h.bias"] = g.normal(0, 0.1, F)
        t[p + "mlp.dense_4h_to_h.weight"] = g.normal(0, 0.1, (d, F))
        t[p + "mlp.dense_4h_to_h.bias"] = g.normal(0, 0.1, d)
    t["gpt_neox.embed_in.weight"] = g.normal(0, 0.1, (V, d))
    t["gpt_neox.final_layer_norm.weight"] = 1 + g.normal(0, 0.1, d)
    t["gpt_neox.final_layer_norm.bias"] = g.normal(0, 0.1, d)
    write_safetensors(tmp_path / "model.safetensors", t, dtype)
    (tmp_path / "config.json").write_text(json.dumps(NEOX_CFG))
    return t, per_head


@pytest.mark.parametrize("dtype", ["F32", "BF16"])
def test_neox_names_shapes_and_qkv_regrouping(tmp_path, dtype):
    t, per_head = _neox_ckpt(tmp_path, dtype)
    shape, layers, extra = HF.load(str(tmp_path), dtype="bf16" if dtype == "BF16" else "f32")
    assert (shape.arch, shape.d, shape.n_heads, shape.n_kv_heads, shape.head_dim, shape.ffn, shape.n_layers,
            shape.vocab, shape.rotary_dim) == (S.NEOX, 64, 2, 2, 32, 128, 2, 50, 8)
    rd = (lambda a: S.round_to(np.asarray(a, np.float32), "bf16")) if dtype == "BF16" else \
         (lambda a: np.asarray(a, np.float32))
    for l, (q, k, v, bq, bk, bv) in enumerate(per_head):
        W = layers[l]
        assert set(S.layer_weight_shapes(shape)) <= set(W)
        # library layout: all query rows, then all key rows, then all value rows
        assert np.array_equal(W["w_qkv"], rd(np.concatenate([q.reshape(-1, 64), k.reshape(-1, 64),
                                                             v.reshape(-1, 64)], 0)))
        assert np.array_equal(W["b_qkv"], rd(np.concatenate([bq.ravel(), bk.ravel(), bv.ravel()])))
        assert np.array_equal(W["w_down"], rd(t[f"gpt_neox.layers.{l}.mlp.dense_4h_to_h.weight"]))
        assert np.array_equal(W["ln2_b"], rd(t[f"gpt_neox.layers.{l}.post_attention_layernorm.bias"]))
        assert W["router_w1"].shape == (64, 64) and W["router_b2"].shape == (1,)
    assert np.array_equal(extra["embed"], rd(t["gpt_neox.embed_in.weight"]))


def test_neox_regrouped_qkv_matches_checkpoint_semantics(tmp_path):
    """GPT-NeoX applies its fused projection, views each row as
    [head][3 * head_dim] and takes q, k, v as the three thirds of each head.
    The oracle reading the regrouped weights sees the same q, k, v."""
    t, _ = _neox_ckpt(tmp_path, "F32")
    shape, layers, _ = HF.load(str(tmp_path), dtype="f32")
    x = np.random.default_rng(1).normal(size=(5, 64))
    fused = x @ t["gpt_neox.layers.1.attention.query_key_value.weight"].T + \
        t["gpt_neox.layers.1.attention.query_key_value.bias"]
    per = fused.reshape(5, 2, 96)
    q_ck, k_ck, v_ck = per[..., :32], per[..., 32:64], per[..., 64:]
    W = layers[1]
    mine = x @ W["w_qkv"].astype(np.float64).T + W["b_qkv"]
    assert mine[:, :64].reshape(5, 2, 32) == pytest.approx(q_ck, rel=1e-6, abs=1e-6)
    assert mine[:, 64:128].reshape(5, 2, 32) == pytest.approx(k_ck, rel=1e-6, abs=1e-6)
    assert mine[:, 128:].reshape(5, 2, 32) == pytest.approx(v_ck, rel=1e-6, abs=1e-6)


def test_qwen_sharded_with_router_file(tmp_path):
    g = np.random.default_rng(2)
    d, H, Hkv, hd, F, L, V = 64, 4, 2, 16, 96, 2, 40
    t = {"model.embed_tokens.weight": g.normal(0, 0.1, (V, d)), "model.norm.weight": 1 + g.normal(0, .1, d)}
    for l in range(L):
        p = f"model.layers.{l}."
        t[p + "input_layernorm.weight"] = 1 + g.normal(0, 0.1, d)
        t[p + "post_attention_layernorm.weight"] = 1 + g.normal(0, 0.1, d)
        for n, rows in (("q", H * hd), ("k", Hkv * hd), ("v", Hkv * hd)):
            t[p + f"self_attn.{n}_proj.weight"] = g.normal(0, 0.1, (rows, d))
            t[p + f"self_attn.{n}_proj.bias"] = g.normal(0, 0.1, rows)
        t[p + "self_attn.o_proj.weight"] = g.normal(0, 0.1, (d, H * hd))
        for n, shp in (("gate", (F, d)), ("up", (F, d)), ("down", (d, F))):
            t[p + f"mlp.{n}_proj.weight"] = g.normal(0, 0.1, shp)
    names = sorted(t)
    half = len(names) // 2
    shards = {"model-00001-of-00002.safetensors": names[:half], "model-00002-of-00002.safetensors": names[half:]}
    for f, ns in shards.items():
        write_safetensors(tmp_path / f, {n: t[n] for n in ns})
    (tmp_path / "model.safetensors.index.json").write_text(
        json.dumps({"weight_map": {n: f for f, ns in shards.items() for n in ns}}))
    (tmp_path / "config.json").write_text(json.dumps(QWEN_CFG))
    rt = {}
    for l in range(L):
        rt.update({f"router.{l}.w1": g.normal(0, 0.1, (64, d)), f"router.{l}.b1": g.normal(0, 0.1, 64),
                   f"router.{l}.w2": g.normal(0, 0.1, 64), f"router.{l}.b2": g.normal(0, 0.1, 1)})
    write_safetensors(tmp_path / "router.safetensors", rt)
    shape, layers, extra = HF.load(str(tmp_path), dtype="f32", router=str(tmp_path / "router.safetensors"))
    assert (shape.arch, shape.n_heads, shape.n_kv_heads, shape.head_dim, shape.rotary_dim, shape.rope_theta) == \
        (S.QWEN, 4, 2, 16, 16, 1e6)
    f32 = lambda a: np.asarray(a, np.float32)
    W = layers[1]
    p = "model.layers.1."
    assert np.array_equal(W["w_qkv"], f32(np.concatenate([t[p + f"self_attn.{n}_proj.weight"] for n in "qkv"])))
    assert np.array_equal(W["b_qkv"], f32(np.concatenate([t[p + f"self_attn.{n}_proj.bias"] for n in "qkv"])))
    assert np.array_equal(W["w_gate"], f32(t[p + "mlp.gate_proj.weight"]))
    assert np.array_equal(W["router_w1"], f32(rt["router.1.w1"]))
    assert np.array_equal(extra["final_w"], f32(t["model.norm.weight"]))
    # the loaded model runs through the oracle (dense, K = T): finite output
    h, _, _ = O.sparse_model_forward(np.array([[1, 5, 7, 39]]), {k: v.astype(np.float64) for k, v in extra.items()},
                                     [{k: v.astype(np.float64) for k, v in w.items()} for w in layers],
                                     O.params_of(shape), [4, 2])
    assert h.shape == (1, 4, 64) and np.isfinite(h).all()


def test_unsupported_configs_are_refused():
    with pytest.raises(ValueError):
        HF.shape_from_config(dict(NEOX_CFG, use_parallel_residual=False))
    with pytest.raises(ValueError):
        HF.shape_from_config(dict(QWEN_CFG, rope_scaling={"type": "yarn", "factor": 4.0}))
    with pytest.raises(ValueError):
        HF.shape_from_config({"model_type": "llama", "hidden_size": 64, "num_attention_heads": 4})
