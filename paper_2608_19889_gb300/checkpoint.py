"""Loading a Hugging Face checkpoint directory into the C ABI's inputs.

The model definition and "a standard safetensors checkpoint" go in (Fig. 1;
appendix "A Complete Model Definition"). This module reads the two files a
checkpoint directory holds for that:

* `config.json` -> the shape dict that `make_config` takes (HF key names);
* `*.safetensors` (one file, or shards listed by
  `model.safetensors.index.json`) -> {HF tensor name: torch tensor}, parsed
  here directly: an 8-byte little-endian header length, a JSON header of
  {name: {dtype, shape, data_offsets}}, then the raw little-endian bytes.

Only what `axon_model_create` accepts is returned: bf16 and fp32 tensors pass
through; fp16 tensors are widened to fp32 (exact). Host memory only; the
create call copies and repacks on the device.

Mixture-of-experts checkpoints: DeepSeek-MoE configs map onto the library's
expert fields and use its tensor names as they are; Mixtral configs map with
norm_topk (Mixtral's router takes the softmax of the top-k logits, which is
the top-k softmax probabilities divided by their sum) and their
`block_sparse_moe.*` tensors are renamed (`hf_to_library_names`). Phi-3
checkpoints store q/k/v as one `qkv_proj` and gate/up as one `gate_up_proj`
matrix; they are split by rows into the library's separate tensors (the
kernels fuse them again in their own layout at create).
"""
from __future__ import annotations

import json
import os
import struct

import numpy as np

_DTYPES = {"BF16": (np.uint16, 2), "F16": (np.float16, 2), "F32": (np.float32, 4)}


def read_safetensors(path: str, names=None) -> dict:
    """{name: torch tensor} of one .safetensors file (bf16 / fp16 / fp32),
    optionally restricted to `names`."""
    import torch
    with open(path, "rb") as f:
        (n,) = struct.unpack("<Q", f.read(8))
        header = json.loads(f.read(n).decode("utf-8"))
        base = 8 + n
        out = {}
        for name, meta in header.items():
            if name == "__metadata__" or (names is not None and name not in names):
                continue
            dt = meta["dtype"]
            if dt not in _DTYPES:
                raise ValueError(f"{path}: tensor {name} has unsupported dtype {dt}")
            np_t, size = _DTYPES[dt]
            start, end = meta["data_offsets"]
            shape = tuple(int(s) for s in meta["shape"])
            count = int(np.prod(shape)) if shape else 1
            if end - start != count * size:
                raise ValueError(f"{path}: tensor {name}: {end - start} bytes for shape {shape}")
            f.seek(base + start)
            arr = np.frombuffer(f.read(end - start), dtype=np.dtype(np_t).newbyteorder("<")).reshape(shape)
            if dt == "BF16":
                t = torch.from_numpy(arr.astype(np.uint16).view(np.int16).copy()).view(torch.bfloat16)
            else:  # fp16 widens exactly; fp32 passes through
                t = torch.from_numpy(arr.astype(np.float32))
            out[name] = t
    return out


def read_checkpoint(directory: str) -> dict:
    """Every tensor of a checkpoint directory: `model.safetensors`, or the
    shards named by `model.safetensors.index.json`."""
    index = os.path.join(directory, "model.safetensors.index.json")
    if os.path.exists(index):
        with open(index) as f:
            weight_map = json.load(f)["weight_map"]
        out = {}
        for shard in sorted(set(weight_map.values())):
            names = {k for k, v in weight_map.items() if v == shard}
            out.update(read_safetensors(os.path.join(directory, shard), names))
        return out
    single = os.path.join(directory, "model.safetensors")
    if not os.path.exists(single):
        raise FileNotFoundError(f"{directory}: no model.safetensors or model.safetensors.index.json")
    return read_safetensors(single)


def _moe_fields(c: dict, mt: str) -> dict:
    """Mixture-of-experts fields of the shape dict (empty for dense models)."""
    if mt == "deepseek":
        if int(c.get("moe_layer_freq", 1)) != 1:
            raise ValueError("MoE layers at a stride (moe_layer_freq > 1) are not implemented")
        if c.get("scoring_func", "softmax") != "softmax" or c.get("topk_method", "greedy") != "greedy":
            raise ValueError("only softmax scoring with greedy top-k routing is implemented")
        if not c.get("n_routed_experts"):
            return {}
        return dict(n_experts=int(c["n_routed_experts"]), top_k=int(c["num_experts_per_tok"]),
                    moe_F=int(c["moe_intermediate_size"]), n_shared=int(c.get("n_shared_experts") or 0),
                    first_dense=int(c.get("first_k_dense_replace", 0)), norm_topk=bool(c.get("norm_topk_prob", False)))
    if mt == "mixtral":
        return dict(n_experts=int(c["num_local_experts"]), top_k=int(c["num_experts_per_tok"]),
                    moe_F=int(c["intermediate_size"]), n_shared=0, first_dense=0, norm_topk=True)
    return {}


def shape_from_hf_config(c: dict) -> dict:
    """The shape dict of `make_config` from an HF config.json of a
    Llama-family decoder (Llama, Mistral, Qwen2, Qwen3, SmolLM, ...) or of a
    DeepSeek-MoE or Mixtral mixture of experts. Raises on a model this
    library does not implement."""
    mt = c.get("model_type", "llama")
    if mt not in ("llama", "mistral", "qwen2", "qwen3", "deepseek", "mixtral", "phi3"):
        raise ValueError(f"model_type {mt!r} is not a Llama-family decoder this library implements")
    H = int(c["num_attention_heads"])
    D = int(c["hidden_size"])
    # Transformers v5 keeps the rotary settings under rope_parameters; older
    # configs keep rope_theta and rope_scaling at the top level
    rp = c.get("rope_parameters") or {}
    theta = rp.get("rope_theta", c.get("rope_theta"))
    if theta is None:
        raise ValueError("no rope_theta in the config (neither top level nor rope_parameters)")
    shape = dict(L=int(c["num_hidden_layers"]), D=D, H=H, G=int(c.get("num_key_value_heads", H)),
                 d=int(c.get("head_dim") or D // H), F=int(c["intermediate_size"]), V=int(c["vocab_size"]),
                 tie=bool(c.get("tie_word_embeddings", False)),
                 bias=bool(c.get("attention_bias", mt == "qwen2")),
                 theta=float(theta), eps=float(c.get("rms_norm_eps", 1e-6)))
    if c.get("mlp_bias"):
        raise ValueError("MLP biases are not implemented")
    if mt == "qwen3":
        shape["qk_norm"] = True  # per-head RMSNorm of q and k (q_norm / k_norm gains)
    if mt == "phi3" and float(c.get("partial_rotary_factor", 1.0)) != 1.0:
        raise ValueError("partial rotary embeddings are not implemented")
    shape.update(_moe_fields(c, mt))
    act = c.get("hidden_act", "silu")
    if act in ("gelu_pytorch_tanh", "gelu_new"):
        shape["act"] = "gelu_tanh"
    elif act != "silu":
        raise ValueError(f"hidden_act {act!r} is not implemented")
    window = c.get("sliding_window")
    if window and mt in ("mistral", "mixtral", "phi3"):
        shape["window"] = int(window)
    elif window and c.get("use_sliding_window", False):
        # Qwen2 windows the layers from max_window_layers on
        first = int(c.get("max_window_layers", 0))
        if 0 < first < shape["L"]:
            raise ValueError("a sliding window on only some layers is not implemented")
        if first <= 0:
            shape["window"] = int(window)
    rs = c.get("rope_scaling") or (rp if rp.get("rope_type", "default") != "default" else None)
    if rs:
        kind = rs.get("rope_type", rs.get("type"))
        if kind == "default":
            return shape
        if kind != "llama3":
            raise ValueError(f"rope_scaling {kind!r} is not implemented")
        shape.update(rope_factor=float(rs["factor"]), rope_low=float(rs["low_freq_factor"]),
                     rope_high=float(rs["high_freq_factor"]),
                     rope_orig=int(rs["original_max_position_embeddings"]))
    return shape


def load_model(directory: str, max_batch: int, max_context: int, **config_kw):
    """(model handle, shape dict) from a checkpoint directory: the config is
    read, the tensors are read to host memory, and axon_model_create copies
    them to the device. config_kw go to make_config (layout, precision, ...)."""
    from . import axon_model_create, make_config
    with open(os.path.join(directory, "config.json")) as f:
        hf = json.load(f)
    shape = shape_from_hf_config(hf)
    weights = hf_to_library_names(shape, hf.get("model_type", "llama"), read_checkpoint(directory))
    if shape["tie"]:
        weights.pop("lm_head.weight", None)
    cfg = make_config(shape, max_batch=max_batch, max_context=max_context, **config_kw)
    return axon_model_create(cfg, weights), shape


def hf_to_library_names(shape: dict, model_type: str, weights: dict) -> dict:
    """Rename a checkpoint's tensors to the names axon_model_create reads:
    Mixtral's router and experts (block_sparse_moe.gate -> mlp.gate,
    experts.{e}.w1 / w3 / w2 -> mlp.experts.{e}.gate_proj / up_proj /
    down_proj); every other family already uses them."""
    if model_type == "phi3":
        return _split_phi3(shape, weights)
    if model_type != "mixtral":
        return weights
    leaf = {"w1": "gate_proj", "w3": "up_proj", "w2": "down_proj"}
    out = {}
    for name, t in weights.items():
        parts = name.split(".")
        if ".block_sparse_moe." in name:
            i = parts.index("block_sparse_moe")
            rest = parts[i + 1:]
            if len(rest) == 4 and rest[0] == "experts" and rest[2] in leaf:
                rest = ["experts", rest[1], leaf[rest[2]], rest[3]]
            elif rest != ["gate", "weight"]:  # the router keeps its leaf name
                raise ValueError(f"unexpected mixture-of-experts tensor {name}")
            name = ".".join(parts[:i] + ["mlp"] + rest)
        out[name] = t
    return out


def _split_phi3(shape: dict, weights: dict) -> dict:
    """Phi-3's fused matrices split by rows: qkv_proj [(H + 2G) d, D] into
    q_proj, k_proj, v_proj (in that order); gate_up_proj [2F, D] into
    gate_proj (first F rows) and up_proj."""
    H, G, d, F = shape["H"], shape["G"], shape["d"], shape["F"]
    out = {}
    for name, t in weights.items():
        if name.endswith(".self_attn.qkv_proj.weight"):
            if tuple(t.shape)[0] != (H + 2 * G) * d:
                raise ValueError(f"{name}: {tuple(t.shape)} rows, expected {(H + 2 * G) * d}")
            p = name[: -len("qkv_proj.weight")]
            out[p + "q_proj.weight"] = t[: H * d].contiguous()
            out[p + "k_proj.weight"] = t[H * d:(H + G) * d].contiguous()
            out[p + "v_proj.weight"] = t[(H + G) * d:].contiguous()
        elif name.endswith(".mlp.gate_up_proj.weight"):
            if tuple(t.shape)[0] != 2 * F:
                raise ValueError(f"{name}: {tuple(t.shape)} rows, expected {2 * F}")
            p = name[: -len("gate_up_proj.weight")]
            out[p + "gate_proj.weight"] = t[:F].contiguous()
            out[p + "up_proj.weight"] = t[F:].contiguous()
        else:
            out[name] = t
    return out
