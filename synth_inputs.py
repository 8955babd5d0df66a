"""Seeded synthetic inputs shared by the tests, the smoke check and the benchmark.

This module holds no part of the decoder's arithmetic: it only draws weights,
token ids, context lengths and paged block tables from fixed seeds, in the
shapes of the 135M-, 0.5B-, 8B- and 32B-class Llama-family decoders the Axon
paper benchmarks (Sec. Results). Trained checkpoints are not used; weights are
random-init.

Recipe
  * matrices, embeddings and biases: N(0, 0.02) drawn in float32 by a torch
    generator seeded per tensor, rounded to bf16 (round-to-nearest-even);
  * RMSNorm gains: 1 + N(0, 0.02), rounded to bf16;
  * token ids: numpy PCG64(seed), uniform integers in [0, V);
  * context lengths: numpy PCG64(seed), uniform integers in [lo, hi];
  * paged block table: a numpy PCG64(seed) permutation of the pool handed out
    to sequences in order, so logical blocks land in shuffled pool blocks.
"""
from __future__ import annotations

import zlib

import numpy as np
import torch

# Shape classes of the paper's decoder benchmarks (HF config keys in comments).
MODEL_SHAPES = {
    # num_hidden_layers, hidden_size, heads, kv_heads, head_dim, intermediate, vocab
    "tiny": dict(L=2, D=64, H=4, G=2, d=16, F=96, V=320, tie=False, bias=True, theta=1e4, eps=1e-5),
    "135m": dict(L=30, D=576, H=9, G=3, d=64, F=1536, V=49152, tie=True, bias=False, theta=1e4, eps=1e-5),
    "0.5b": dict(L=24, D=896, H=14, G=2, d=64, F=4864, V=151936, tie=True, bias=True, theta=1e6, eps=1e-6),
    "8b": dict(L=32, D=4096, H=32, G=8, d=128, F=14336, V=128256, tie=False, bias=False, theta=5e5, eps=1e-5),
    "32b": dict(L=64, D=5120, H=40, G=8, d=128, F=27648, V=152064, tie=False, bias=True, theta=1e6, eps=1e-6),
    # DeepSeek-MoE-16B-shaped: 28 layers, the first dense, the rest with 64
    # routed experts (6 per token, weights not renormalised) and 2 shared
    # experts of width 1408 each; multi-head attention, head_dim 128
    "moe16b": dict(L=28, D=2048, H=16, G=16, d=128, F=10944, V=102400, tie=False, bias=False, theta=1e4,
                   eps=1e-6, n_experts=64, top_k=6, moe_F=1408, n_shared=2, first_dense=1, norm_topk=False),
    # Mistral-shaped 7B: the Llama block with a 4096-token sliding window
    "7b_swa": dict(L=32, D=4096, H=32, G=8, d=128, F=14336, V=32000, tie=False, bias=False, theta=1e4, eps=1e-5,
                   window=4096),
}

# Workloads: prompt batch and length, decode steps, cache layout.
WORKLOADS = {
    "135m_b1_s16_n16": dict(model="135m", B=1, S=16, n_new=16, layout="contiguous"),
    "0.5b_b1_s512_n128": dict(model="0.5b", B=1, S=512, n_new=128, layout="contiguous"),
    "8b_b1_s1024_n256": dict(model="8b", B=1, S=1024, n_new=256, layout="contiguous"),
    "8b_b8_s1024_n256": dict(model="8b", B=8, S=1024, n_new=256, layout="contiguous"),
    "8b_paged_b64_ctx512-4096_n128": dict(model="8b", B=64, ctx=(512, 4096), n_new=128, layout="paged"),
    "32b_b1_s2048_n256": dict(model="32b", B=1, S=2048, n_new=256, layout="contiguous"),
    "32b_b16_s2048_n256": dict(model="32b", B=16, S=2048, n_new=256, layout="contiguous"),
    # the paper's mixture-of-experts data point (DeepSeek-MoE 16B, Sec. Results)
    "moe16b_b1_s512_n128": dict(model="moe16b", B=1, S=512, n_new=128, layout="contiguous"),
    # prompt twice the window: the window bounds prefill attention and every decode step's keys
    "7b_swa_b1_s8192_n256": dict(model="7b_swa", B=1, S=8192, n_new=256, layout="contiguous"),
}

SEED_WEIGHTS, SEED_IDS, SEED_CTX, SEED_BLOCKS = 0, 1, 2, 3


def weight_shapes(m: dict) -> dict:
    """HF Llama parameter names and shapes ([out, in] for matrices); with
    qk_norm, the per-head q and k RMSNorm gains of Qwen3-family layers; with
    n_experts > 0, layers from first_dense on carry a mixture-of-experts MLP
    in the DeepSeek-MoE naming (router mlp.gate, routed mlp.experts.{e}.*,
    shared mlp.shared_experts.*)."""
    L, D, H, G, d, F, V = (m[k] for k in ("L", "D", "H", "G", "d", "F", "V"))
    shapes = {"model.embed_tokens.weight": (V, D)}
    for l in range(L):
        p = f"model.layers.{l}."
        shapes[p + "input_layernorm.weight"] = (D,)
        shapes[p + "self_attn.q_proj.weight"] = (H * d, D)
        shapes[p + "self_attn.k_proj.weight"] = (G * d, D)
        shapes[p + "self_attn.v_proj.weight"] = (G * d, D)
        if m["bias"]:
            shapes[p + "self_attn.q_proj.bias"] = (H * d,)
            shapes[p + "self_attn.k_proj.bias"] = (G * d,)
            shapes[p + "self_attn.v_proj.bias"] = (G * d,)
        if m.get("qk_norm"):
            shapes[p + "self_attn.q_norm.weight"] = (d,)
            shapes[p + "self_attn.k_norm.weight"] = (d,)
        shapes[p + "self_attn.o_proj.weight"] = (D, H * d)
        shapes[p + "post_attention_layernorm.weight"] = (D,)
        if m.get("n_experts", 0) and l >= m.get("first_dense", 0):
            E, Fe, ns = m["n_experts"], m["moe_F"], m.get("n_shared", 0)
            shapes[p + "mlp.gate.weight"] = (E, D)
            for e in range(E):
                q = f"{p}mlp.experts.{e}."
                shapes[q + "gate_proj.weight"] = (Fe, D)
                shapes[q + "up_proj.weight"] = (Fe, D)
                shapes[q + "down_proj.weight"] = (D, Fe)
            if ns:
                q = p + "mlp.shared_experts."
                shapes[q + "gate_proj.weight"] = (ns * Fe, D)
                shapes[q + "up_proj.weight"] = (ns * Fe, D)
                shapes[q + "down_proj.weight"] = (D, ns * Fe)
            continue
        shapes[p + "mlp.gate_proj.weight"] = (F, D)
        shapes[p + "mlp.up_proj.weight"] = (F, D)
        shapes[p + "mlp.down_proj.weight"] = (D, F)
    shapes["model.norm.weight"] = (D,)
    if not m["tie"]:
        shapes["lm_head.weight"] = (V, D)
    return shapes


def gpt2_weight_shapes(c: dict) -> dict:
    """HF GPT-2 parameter names and shapes (the appendix's complete model):
    `transpose=true` matrices stored [in, out]; keys L, D, V, P (positions)."""
    L, D, V, P = int(c["L"]), int(c["D"]), int(c["V"]), int(c["P"])
    s = {"transformer.wte.weight": (V, D), "transformer.wpe.weight": (P, D)}
    for l in range(L):
        p = f"transformer.h.{l}."
        for ln in ("ln_1", "ln_2"):
            s[p + ln + ".weight"] = (D,)
            s[p + ln + ".bias"] = (D,)
        s[p + "attn.c_attn.weight"] = (D, 3 * D)
        s[p + "attn.c_attn.bias"] = (3 * D,)
        s[p + "attn.c_proj.weight"] = (D, D)
        s[p + "attn.c_proj.bias"] = (D,)
        s[p + "mlp.c_fc.weight"] = (D, 4 * D)
        s[p + "mlp.c_fc.bias"] = (4 * D,)
        s[p + "mlp.c_proj.weight"] = (4 * D, D)
        s[p + "mlp.c_proj.bias"] = (D,)
    s["transformer.ln_f.weight"] = (D,)
    s["transformer.ln_f.bias"] = (D,)
    return s


def make_gpt2_weights(c: dict, seed: int = SEED_WEIGHTS, device="cpu") -> dict:
    """bf16 GPT-2 tensors by HF name: LayerNorm gains 1 + N(0, 0.02), every
    other tensor (matrices, embeddings, biases) N(0, 0.02)."""
    out = {}
    for name, shape in gpt2_weight_shapes(c).items():
        g = torch.Generator(device=device)
        g.manual_seed(_tensor_seed(seed, name))
        t = torch.empty(shape, dtype=torch.float32, device=device)
        t.normal_(0.0, 0.02, generator=g)
        if ".ln_" in name and name.endswith(".weight"):
            t += 1.0
        out[name] = t.to(torch.bfloat16)
    return out


def _tensor_seed(seed: int, name: str) -> int:
    return (seed * 1_000_003 + zlib.crc32(name.encode())) & 0x7FFF_FFFF_FFFF


def make_weights(m: dict, seed: int = SEED_WEIGHTS, device="cpu") -> dict:
    """bf16 tensors by HF name, drawn on `device` (a CUDA generator is used
    for large models; values differ between devices, never within one)."""
    out = {}
    for name, shape in weight_shapes(m).items():
        g = torch.Generator(device=device)
        g.manual_seed(_tensor_seed(seed, name))
        t = torch.empty(shape, dtype=torch.float32, device=device)
        t.normal_(0.0, 0.02, generator=g)
        if name.endswith(("layernorm.weight", "q_norm.weight", "k_norm.weight")) or name == "model.norm.weight":
            t += 1.0
        out[name] = t.to(torch.bfloat16)
    return out


def weights_as_f32_numpy(w: dict) -> dict:
    """Exact float32 widening of bf16 weights, for the oracle."""
    return {k: v.detach().float().cpu().numpy() for k, v in w.items()}


def make_ids(B: int, S: int, V: int, seed: int = SEED_IDS) -> np.ndarray:
    return np.random.Generator(np.random.PCG64(seed)).integers(0, V, size=(B, S), dtype=np.int64).astype(np.int32)


def make_context_lens(B: int, lo: int, hi: int, seed: int = SEED_CTX) -> np.ndarray:
    return np.random.Generator(np.random.PCG64(seed)).integers(lo, hi + 1, size=B, dtype=np.int64).astype(np.int32)


def make_block_table(capacities, block_size: int, max_blocks: int, num_blocks: int,
                     seed: int = SEED_BLOCKS) -> np.ndarray:
    """Shuffled block table: sequence b gets ceil(capacities[b] / block_size)
    pool blocks taken in turn from a seeded permutation of the pool. Unused
    entries are -1."""
    need = [-(-int(c) // block_size) for c in capacities]
    if sum(need) > num_blocks:
        raise ValueError("block pool too small")
    perm = np.random.Generator(np.random.PCG64(seed)).permutation(num_blocks)
    bt = np.full((len(need), max_blocks), -1, dtype=np.int32)
    at = 0
    for b, n in enumerate(need):
        bt[b, :n] = perm[at:at + n]
        at += n
    return bt
