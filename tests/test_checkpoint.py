"""Checkpoint loading on the host: the hand-written safetensors reader (single
file and sharded index, bf16 / fp16 / fp32) against tensors written here, and
the HF config.json mapping of the Llama-family variants and the
mixture-of-experts families (DeepSeek-MoE, Mixtral with its tensor renaming)
the kernels implement."""
import json
import struct

import numpy as np
import pytest

torch = pytest.importorskip("torch")

import synth_inputs as si  # noqa: E402
from paper_2608_19889_gb300 import checkpoint as ck  # noqa: E402


def _write_safetensors(path, tensors):
    """Minimal writer: header of dtype / shape / byte offsets, then the data."""
    header, blobs, off = {}, [], 0
    for name, t in tensors.items():
        if t.dtype == torch.bfloat16:
            raw, dt = t.view(torch.int16).numpy().astype("<i2").tobytes(), "BF16"
        elif t.dtype == torch.float16:
            raw, dt = t.numpy().astype("<f2").tobytes(), "F16"
        else:
            raw, dt = t.numpy().astype("<f4").tobytes(), "F32"
        header[name] = {"dtype": dt, "shape": list(t.shape), "data_offsets": [off, off + len(raw)]}
        blobs.append(raw)
        off += len(raw)
    header["__metadata__"] = {"format": "pt"}
    h = json.dumps(header).encode()
    with open(path, "wb") as f:
        f.write(struct.pack("<Q", len(h)))
        f.write(h)
        for b in blobs:
            f.write(b)


def test_reader_returns_the_written_tensors_in_every_dtype(tmp_path):
    g = torch.Generator().manual_seed(0)
    ts = {"a.bf16": torch.randn(3, 5, generator=g).to(torch.bfloat16),
          "b.f16": torch.randn(7, generator=g).to(torch.float16),
          "c.f32": torch.randn(2, 2, 2, generator=g)}
    _write_safetensors(tmp_path / "x.safetensors", ts)
    got = ck.read_safetensors(str(tmp_path / "x.safetensors"))
    assert set(got) == set(ts)
    assert got["a.bf16"].dtype == torch.bfloat16 and torch.equal(got["a.bf16"], ts["a.bf16"])
    assert got["b.f16"].dtype == torch.float32 and torch.equal(got["b.f16"], ts["b.f16"].float())  # exact widening
    assert torch.equal(got["c.f32"], ts["c.f32"])


def test_sharded_checkpoint_reads_every_tensor_once(tmp_path):
    m = dict(L=2, D=64, H=4, G=2, d=16, F=96, V=50, tie=False, bias=True, theta=1e4, eps=1e-5)
    w = si.make_weights(m)
    names = sorted(w)
    shards = {"model-00001-of-00002.safetensors": names[: len(names) // 2],
              "model-00002-of-00002.safetensors": names[len(names) // 2:]}
    weight_map = {}
    for shard, ns in shards.items():
        _write_safetensors(tmp_path / shard, {n: w[n] for n in ns})
        weight_map.update({n: shard for n in ns})
    with open(tmp_path / "model.safetensors.index.json", "w") as f:
        json.dump({"metadata": {}, "weight_map": weight_map}, f)
    got = ck.read_checkpoint(str(tmp_path))
    assert set(got) == set(si.weight_shapes(m))
    assert all(torch.equal(got[n], w[n]) for n in names)


def test_truncated_tensor_is_rejected(tmp_path):
    _write_safetensors(tmp_path / "x.safetensors", {"a": torch.zeros(4)})
    raw = bytearray((tmp_path / "x.safetensors").read_bytes())
    (n,) = struct.unpack("<Q", raw[:8])
    hdr = json.loads(raw[8:8 + n])
    hdr["a"]["shape"] = [5]  # 20 bytes expected, 16 stored
    h = json.dumps(hdr).encode()
    (tmp_path / "y.safetensors").write_bytes(struct.pack("<Q", len(h)) + h + raw[8 + n:])
    with pytest.raises(ValueError):
        ck.read_safetensors(str(tmp_path / "y.safetensors"))


LLAMA31 = {"model_type": "llama", "num_hidden_layers": 32, "hidden_size": 4096, "num_attention_heads": 32,
           "num_key_value_heads": 8, "intermediate_size": 14336, "vocab_size": 128256, "rope_theta": 500000.0,
           "rms_norm_eps": 1e-5, "tie_word_embeddings": False, "hidden_act": "silu",
           "rope_scaling": {"rope_type": "llama3", "factor": 8.0, "low_freq_factor": 1.0, "high_freq_factor": 4.0,
                            "original_max_position_embeddings": 8192}}


def test_llama_config_with_rope_scaling():
    s = ck.shape_from_hf_config(LLAMA31)
    assert (s["L"], s["D"], s["H"], s["G"], s["d"], s["F"], s["V"]) == (32, 4096, 32, 8, 128, 14336, 128256)
    assert s["tie"] is False and s["bias"] is False and s["theta"] == 5e5 and s["eps"] == 1e-5
    assert (s["rope_factor"], s["rope_low"], s["rope_high"], s["rope_orig"]) == (8.0, 1.0, 4.0, 8192)
    assert "window" not in s and s.get("act", "silu") == "silu"


def test_qwen2_has_qkv_bias_and_mistral_its_window():
    q = dict(LLAMA31, model_type="qwen2", rope_scaling=None, tie_word_embeddings=True, use_sliding_window=False,
             sliding_window=32768)
    s = ck.shape_from_hf_config(q)
    assert s["bias"] is True and s["tie"] is True and "window" not in s
    m = dict(LLAMA31, model_type="mistral", rope_scaling=None, sliding_window=4096)
    assert ck.shape_from_hf_config(m)["window"] == 4096
    assert "window" not in ck.shape_from_hf_config(dict(m, sliding_window=None))
    qw = dict(q, use_sliding_window=True, sliding_window=4096)
    assert ck.shape_from_hf_config(dict(qw, max_window_layers=0))["window"] == 4096  # every layer windowed
    assert "window" not in ck.shape_from_hf_config(dict(qw, max_window_layers=32))  # no layer windowed


def test_gelu_gate_and_unsupported_configs():
    assert ck.shape_from_hf_config(dict(LLAMA31, rope_scaling=None, hidden_act="gelu_pytorch_tanh"))["act"] == \
        "gelu_tanh"
    for bad in (dict(LLAMA31, model_type="gpt2"), dict(LLAMA31, hidden_act="relu"),
                dict(LLAMA31, rope_scaling={"rope_type": "yarn", "factor": 4.0}), dict(LLAMA31, mlp_bias=True),
                dict(LLAMA31, model_type="qwen2", use_sliding_window=True, sliding_window=4096,
                     max_window_layers=28)):
        with pytest.raises(ValueError):
            ck.shape_from_hf_config(bad)


def test_head_dim_defaults_to_width_over_heads():
    c = {k: v for k, v in LLAMA31.items() if k != "rope_scaling"}
    assert ck.shape_from_hf_config(c)["d"] == 128
    assert ck.shape_from_hf_config(dict(c, head_dim=64))["d"] == 64


def test_rope_parameters_of_newer_configs_and_default_rope_type():
    """Transformers v5 configs keep the rotary settings under
    rope_parameters; a 'default' rope type means no frequency scaling; a
    config with no rotary base at all is refused rather than defaulted."""
    top = {k: v for k, v in LLAMA31.items() if k not in ("rope_theta", "rope_scaling")}
    v5 = dict(top, rope_parameters={"rope_type": "llama3", "rope_theta": 500000.0, "factor": 8.0,
                                    "low_freq_factor": 1.0, "high_freq_factor": 4.0,
                                    "original_max_position_embeddings": 8192})
    s = ck.shape_from_hf_config(v5)
    assert s["theta"] == 5e5 and (s["rope_factor"], s["rope_orig"]) == (8.0, 8192)
    plain = ck.shape_from_hf_config(dict(top, rope_parameters={"rope_type": "default", "rope_theta": 1e6}))
    assert plain["theta"] == 1e6 and "rope_factor" not in plain
    old_default = ck.shape_from_hf_config(dict(LLAMA31, rope_scaling={"rope_type": "default"}))
    assert "rope_factor" not in old_default
    with pytest.raises(ValueError):
        ck.shape_from_hf_config(top)


# ------------------------------------------------------ mixture of experts
DEEPSEEK_MOE_16B = {  # the config.json keys of a DeepSeek-MoE-16B-shaped model
    "model_type": "deepseek", "num_hidden_layers": 28, "hidden_size": 2048, "num_attention_heads": 16,
    "num_key_value_heads": 16, "intermediate_size": 10944, "vocab_size": 102400, "rope_theta": 10000.0,
    "rms_norm_eps": 1e-6, "tie_word_embeddings": False, "attention_bias": False, "hidden_act": "silu",
    "n_routed_experts": 64, "num_experts_per_tok": 6, "moe_intermediate_size": 1408, "n_shared_experts": 2,
    "first_k_dense_replace": 1, "moe_layer_freq": 1, "norm_topk_prob": False, "scoring_func": "softmax",
    "topk_method": "greedy"}
MIXTRAL = {
    "model_type": "mixtral", "num_hidden_layers": 2, "hidden_size": 64, "num_attention_heads": 4,
    "num_key_value_heads": 2, "intermediate_size": 96, "vocab_size": 50, "rope_theta": 1e6, "rms_norm_eps": 1e-5,
    "num_local_experts": 4, "num_experts_per_tok": 2, "sliding_window": None, "tie_word_embeddings": False}


def test_deepseek_moe_config_is_the_moe_workloads_shape():
    s = ck.shape_from_hf_config(DEEPSEEK_MOE_16B)
    want = dict(si.MODEL_SHAPES["moe16b"])
    assert {k: s[k] for k in want} == want


@pytest.mark.parametrize("key,value", [("moe_layer_freq", 2), ("scoring_func", "sigmoid"),
                                       ("topk_method", "group_limited_greedy")])
def test_deepseek_routing_the_kernels_do_not_implement_is_refused(key, value):
    with pytest.raises(ValueError):
        ck.shape_from_hf_config(dict(DEEPSEEK_MOE_16B, **{key: value}))


def test_qwen3_has_qk_norm_and_moe_families_without_kernels_are_refused():
    q3 = {"model_type": "qwen3", "num_hidden_layers": 2, "hidden_size": 64, "num_attention_heads": 4,
          "num_key_value_heads": 2, "head_dim": 32, "intermediate_size": 96, "vocab_size": 50, "rope_theta": 1e6,
          "attention_bias": False}
    s = ck.shape_from_hf_config(q3)
    assert s["qk_norm"] and not s["bias"] and s["d"] == 32
    for mt in ("qwen2_moe", "deepseek_v2"):
        with pytest.raises(ValueError):
            ck.shape_from_hf_config(dict(q3, model_type=mt))


def test_mixtral_config_and_tensor_names():
    s = ck.shape_from_hf_config(MIXTRAL)
    assert (s["n_experts"], s["top_k"], s["moe_F"], s["n_shared"], s["first_dense"], s["norm_topk"]) == \
        (4, 2, 96, 0, 0, True)
    assert "window" not in s and ck.shape_from_hf_config(dict(MIXTRAL, sliding_window=4096))["window"] == 4096
    lib = si.make_weights(s)
    inv = {"gate_proj": "w1", "up_proj": "w3", "down_proj": "w2"}
    mixtral = {}
    for name, t in lib.items():  # the library's names written the way a Mixtral checkpoint stores them
        p = name.split(".")
        if ".mlp.gate." in name:
            name = ".".join(p[:3] + ["block_sparse_moe", "gate", "weight"])
        elif ".mlp.experts." in name:
            name = ".".join(p[:3] + ["block_sparse_moe", "experts", p[5], inv[p[6]], "weight"])
        mixtral[name] = t
    assert not any(".mlp." in k for k in mixtral)
    back = ck.hf_to_library_names(s, "mixtral", mixtral)
    assert set(back) == set(lib) == set(si.weight_shapes(s))
    assert all(torch.equal(back[k], lib[k]) for k in lib)
    with pytest.raises(ValueError):
        ck.hf_to_library_names(s, "mixtral", {"model.layers.0.block_sparse_moe.experts.0.w9.weight": lib[
            "model.embed_tokens.weight"]})


def test_softmax_of_the_top_k_logits_is_the_renormalised_top_k():
    """Mixtral routes by the softmax of its top-k router logits; the library
    (and the oracle) take the softmax over all experts, keep the top k and,
    with norm_topk, divide by their sum. The two are the same weights."""
    from oracle import decoder as od
    rng = np.random.Generator(np.random.PCG64(3))
    h, Wr = rng.normal(size=(9, 16)), rng.normal(size=(8, 16))
    idx, w, _ = od.moe_route(h, Wr, 2, norm_topk=True)
    logits = h @ Wr.T
    top = np.take_along_axis(logits, idx, axis=-1)
    direct = np.exp(top - top.max(-1, keepdims=True))
    direct /= direct.sum(-1, keepdims=True)
    assert np.allclose(w, direct, rtol=1e-13, atol=1e-15)
    assert np.all(idx == np.argsort(-logits, axis=-1, kind="stable")[:, :2])  # the same experts too


PHI3 = {"model_type": "phi3", "num_hidden_layers": 2, "hidden_size": 64, "num_attention_heads": 4,
        "num_key_value_heads": 2, "intermediate_size": 96, "vocab_size": 50, "rope_theta": 10000.0,
        "rms_norm_eps": 1e-5, "sliding_window": 2047, "tie_word_embeddings": False, "hidden_act": "silu"}


def test_phi3_fused_matrices_split_into_the_librarys_tensors():
    s = ck.shape_from_hf_config(PHI3)
    assert (s["d"], s["window"], s["bias"]) == (16, 2047, False)
    lib = si.make_weights(s)
    fused = {}
    for name, t in lib.items():  # the library's tensors fused the way a Phi-3 checkpoint stores them
        if ".self_attn.q_proj." in name:
            p = name.replace("q_proj", "{}")
            fused[p.format("qkv_proj")] = torch.cat([lib[p.format(x)] for x in ("q_proj", "k_proj", "v_proj")])
        elif ".mlp.gate_proj." in name:
            p = name.replace("gate_proj", "{}")
            fused[p.format("gate_up_proj")] = torch.cat([lib[p.format("gate_proj")], lib[p.format("up_proj")]])
        elif not any(x in name for x in (".k_proj.", ".v_proj.", ".up_proj.")):
            fused[name] = t
    back = ck.hf_to_library_names(s, "phi3", fused)
    assert set(back) == set(lib) == set(si.weight_shapes(s))
    assert all(torch.equal(back[k], lib[k]) for k in lib)
    bad = dict(fused)
    bad["model.layers.0.mlp.gate_up_proj.weight"] = bad["model.layers.0.mlp.gate_up_proj.weight"][:-1]
    with pytest.raises(ValueError):
        ck.hf_to_library_names(s, "phi3", bad)
    with pytest.raises(ValueError):
        ck.shape_from_hf_config(dict(PHI3, rope_scaling={"type": "longrope", "short_factor": [1.0], "long_factor": [1.0]}))
    with pytest.raises(ValueError):
        ck.shape_from_hf_config(dict(PHI3, partial_rotary_factor=0.5))
