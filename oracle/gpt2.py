"""Plain float64 CPU oracle of the GPT-2 causal LM, the complete model the
Axon paper writes out (appendix "A Complete Model Definition").

TEST INFRASTRUCTURE ONLY, like the rest of this package: the product path
never imports it, and it imports nothing from the product.

What it computes, read from that appendix and the built-ins it names:

* token embedding plus a learned position embedding at position
  past_length + i (`NN.embedding` of the token ids and of `position_ids ...
  past_length`);
* per layer a pre-norm block: LayerNorm `ln_1`; one fused projection
  `c_attn` to q, k and v (with bias, weight stored [in, out] -- the listing's
  `transpose=true`); multi-head causal attention over the cache (every head
  its own key/value head, scale 1/sqrt(d)); `c_proj` with bias; residual;
  LayerNorm `ln_2`; MLP `c_fc` (4D, bias) -> gelu_new -> `c_proj` (bias);
  residual;
* final LayerNorm `ln_f` and the LM head tied to the token embedding.

The paper prints no formulas; the readings taken are in READINGS.
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np

from .decoder import ContiguousKV, causal_attention, gelu_tanh

READINGS = [
    "LayerNorm: y = (x - mean(x)) / sqrt(var(x) + eps) * g + b over the last "
    "axis, var the biased (1/D) variance, eps inside the square root.",
    "`transpose=true` linears store W as [in, out]: y = x W + b.",
    "c_attn's output splits into q, k, v in that order, D columns each.",
    "Learned positions: position p adds row p of the position table; the "
    "i-th new token of a sequence sits at past_length + i.",
    "Attention: H heads, each with its own key/value head (G = H), scale "
    "1/sqrt(D/H), causal mask keeping keys at positions <= the query's.",
    "MLP: gelu_new(x W_fc + b_fc) W_proj + b_proj, gelu_new the tanh form.",
    "LM head: ln_f(x) wte^T (tied), no bias.",
]


@dataclass(frozen=True)
class GPT2Config:
    """GPT-2 config.json keys read through `Config.dim @@key`."""

    L: int  # n_layer
    D: int  # n_embd
    H: int  # n_head
    V: int  # vocab_size
    P: int  # n_positions
    eps: float = 1e-5  # layer_norm_epsilon

    @property
    def d(self) -> int:
        return self.D // self.H

    @staticmethod
    def from_dict(c: dict) -> "GPT2Config":
        return GPT2Config(L=int(c["L"]), D=int(c["D"]), H=int(c["H"]), V=int(c["V"]), P=int(c["P"]),
                          eps=float(c.get("eps", 1e-5)))


def layernorm(x, g, b, eps):
    """NN.layernorm (appendix GPT-2 definition, `ln_1`, `ln_2`, `ln_f`):
    centre each vector on the last axis, scale it to unit variance, then
    apply the gain g and bias b."""
    x = np.asarray(x, dtype=np.float64)
    mu = np.mean(x, axis=-1, keepdims=True)
    var = np.mean((x - mu) ** 2, axis=-1, keepdims=True)
    return (x - mu) / np.sqrt(var + eps) * np.asarray(g, dtype=np.float64) + np.asarray(b, dtype=np.float64)


def linear_t(x, W, b):
    """NN.linear with `transpose=true` (weight stored [in, out]) and bias."""
    return np.asarray(x, dtype=np.float64) @ np.asarray(W, dtype=np.float64) + np.asarray(b, dtype=np.float64)


class GPT2Oracle:
    """The GPT-2 causal LM over HF-named weights (float64)."""

    def __init__(self, cfg: GPT2Config, weights):
        self.cfg = cfg
        self.W = {k: np.asarray(v, dtype=np.float64) for k, v in weights.items()}

    def new_cache(self, B, Tmax):
        c = self.cfg
        return ContiguousKV(c.L, B, Tmax, c.H, c.d)

    def forward(self, ids, cache, past_lens):
        """New tokens ids [B, S] after past_lens[b] cached tokens; writes
        their K, V into the cache and returns logits [B, S, V]."""
        c, W = self.cfg, self.W
        ids = np.asarray(ids, dtype=np.int64)
        B, S = ids.shape
        pos = np.asarray(past_lens, dtype=np.int64).reshape(B)[:, None] + np.arange(S)[None, :]
        x = W["transformer.wte.weight"][ids] + W["transformer.wpe.weight"][pos]
        for l in range(c.L):
            p = f"transformer.h.{l}."
            h = layernorm(x, W[p + "ln_1.weight"], W[p + "ln_1.bias"], c.eps)
            qkv = linear_t(h, W[p + "attn.c_attn.weight"], W[p + "attn.c_attn.bias"])
            q = qkv[..., : c.D].reshape(B, S, c.H, c.d)
            k = qkv[..., c.D: 2 * c.D].reshape(B, S, c.H, c.d)
            v = qkv[..., 2 * c.D:].reshape(B, S, c.H, c.d)
            o = np.empty((B, S, c.H, c.d))
            for b in range(B):
                cache.write(l, b, pos[b], k[b], v[b])
                Kb, Vb = cache.read(l, b, int(pos[b, -1]) + 1)
                o[b] = causal_attention(q[b], Kb, Vb, pos[b], c.H, c.H)
            x = x + linear_t(o.reshape(B, S, c.D), W[p + "attn.c_proj.weight"], W[p + "attn.c_proj.bias"])
            h2 = layernorm(x, W[p + "ln_2.weight"], W[p + "ln_2.bias"], c.eps)
            u = gelu_tanh(linear_t(h2, W[p + "mlp.c_fc.weight"], W[p + "mlp.c_fc.bias"]))
            x = x + linear_t(u, W[p + "mlp.c_proj.weight"], W[p + "mlp.c_proj.bias"])
        hf = layernorm(x, W["transformer.ln_f.weight"], W["transformer.ln_f.bias"], c.eps)
        return hf @ W["transformer.wte.weight"].T

    def prefill(self, ids, cache):
        B = np.asarray(ids).shape[0]
        return self.forward(ids, cache, np.zeros(B, dtype=np.int64))

    def decode_step(self, tokens, cache, context_lens):
        return self.forward(np.asarray(tokens, dtype=np.int64).reshape(-1, 1), cache, context_lens)[:, 0, :]
