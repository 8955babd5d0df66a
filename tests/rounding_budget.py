"""Rounding budget of the 16-bit modes: the float64 forward with 16-bit
rounding applied at chosen points, to see which rounding point the logit
error comes from.

Test infrastructure (run by hand for the 8B-width table, and by
tests/test_rounding_budget.py at toy width): the forward is composed from
the oracle's elementary operations (RMSNorm, linear, RoPE, softmax, SwiGLU)
in the decoder order of the oracle's own forward, with a rounding hook at
each point where the GPU path stores a 16-bit value:

  a   the normalised GEMM operand x*g (the kernels scale the accumulator by
      the inverse RMS, so x*g is what gets rounded), one term
  q   the rotated query;  k, v  the cache entries (keys after RoPE)
  P   the unnormalised probabilities exp(s - max) entering P.V (the row sum
      that divides the result stays in fp32, as in the kernels)
  o   the attention output (the O projection's operand)
  u   the SwiGLU output (the down projection's operand)

With no point rounded it is the oracle's prefill exactly; rounding is
round-to-nearest-even through torch's bf16 / fp16 conversion.

    python tests/rounding_budget.py --width 8b --layers 2 --seq 48
"""
from __future__ import annotations

import argparse
import math
import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(HERE))

from oracle import decoder as od  # noqa: E402

POINTS = ("a", "q", "k", "v", "P", "o", "u")


def rounder(kind):
    """float64 array -> the same values rounded to bf16 or fp16; kind
    "bf16x2" / "fp16x2": two terms, hi = round(x) plus round(x - hi)."""
    import torch
    dt = {"bf16": torch.bfloat16, "fp16": torch.float16}[kind.replace("x2", "")]

    def r1(x):
        return torch.from_numpy(np.ascontiguousarray(x, dtype=np.float64)).to(dt).to(torch.float64).numpy()

    if kind.endswith("x2"):
        return lambda x: r1(x) + r1(np.asarray(x, dtype=np.float64) - r1(x))
    return r1


def forward(cfg: od.DecoderConfig, W: dict, ids, rounded=(), kind="fp16"):
    """Prompt pass of B sequences from an empty cache with 16-bit rounding at
    the points named in `rounded`, all of one kind, or with `kind` a dict
    {point: kind}. Returns logits [B, S, V]."""
    kinds = kind if isinstance(kind, dict) else {pt: kind for pt in POINTS}
    rnds = {pt: rounder(k) for pt, k in kinds.items()}

    def at(point, x):
        return rnds[point](x) if point in rounded else x

    def norm(x, g):
        if "a" not in rounded:
            return od.rmsnorm(x, g, cfg.eps)
        r = 1.0 / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + cfg.eps)
        return rnds["a"](x * g) * r

    ids = np.asarray(ids, dtype=np.int64)
    B, S = ids.shape
    pos = np.arange(S)[None, :].repeat(B, 0)
    x = W["model.embed_tokens.weight"][ids]
    H, G, d = cfg.H, cfg.G, cfg.d
    for l in range(cfg.L):
        p = f"model.layers.{l}."
        h = norm(x, W[p + "input_layernorm.weight"])
        b = (lambda n: W[p + f"self_attn.{n}_proj.bias"]) if cfg.bias else (lambda n: None)
        q = od.linear(h, W[p + "self_attn.q_proj.weight"], b("q")).reshape(B, S, H, d)
        k = od.linear(h, W[p + "self_attn.k_proj.weight"], b("k")).reshape(B, S, G, d)
        v = od.linear(h, W[p + "self_attn.v_proj.weight"], b("v")).reshape(B, S, G, d)
        if cfg.qk_norm:
            q = od.rmsnorm(q, W[p + "self_attn.q_norm.weight"], cfg.eps)
            k = od.rmsnorm(k, W[p + "self_attn.k_norm.weight"], cfg.eps)
        q = at("q", od.rope(q, pos[:, :, None], cfg.theta, cfg.rope_scaling()))
        k = at("k", od.rope(k, pos[:, :, None], cfg.theta, cfg.rope_scaling()))
        v = at("v", v)
        o = np.empty((B, S, H, d))
        t = np.arange(S)
        keep = t[None, :] <= t[:, None]
        if cfg.window:
            keep &= t[None, :] > t[:, None] - cfg.window
        for bb in range(B):
            for hh in range(H):
                gg = hh // (H // G)
                s = np.where(keep, q[bb, :, hh] @ k[bb, :, gg].T / math.sqrt(d), -np.inf)
                # flash form, as the kernels: the 16-bit probabilities
                # exp(s - max) enter P.V, the row sum stays unrounded
                e = np.exp(s - s.max(axis=-1, keepdims=True))
                o[bb, :, hh] = (at("P", e) @ v[bb, :, gg]) / e.sum(axis=-1, keepdims=True)
        o = at("o", o.reshape(B, S, H * d))
        x = x + od.linear(o, W[p + "self_attn.o_proj.weight"])
        h2 = norm(x, W[p + "post_attention_layernorm.weight"])
        if cfg.is_moe_layer(l):
            raise NotImplementedError("mixture-of-experts layers")
        u = at("u", od.swiglu(od.linear(h2, W[p + "mlp.gate_proj.weight"]),
                              od.linear(h2, W[p + "mlp.up_proj.weight"]), cfg.act))
        x = x + od.linear(u, W[p + "mlp.down_proj.weight"])
    head = W["model.embed_tokens.weight"] if cfg.tie else W["lm_head.weight"]
    return od.linear(norm(x, W["model.norm.weight"]), head)


def table(cfg, W, ids, kinds=("fp16", "bf16")):
    """{kind: {point or 'all': (rms, max) of the logit error}}: each point
    alone, and every point but a together (the two-term operand modes keep a
    exact to about 2^-22)."""
    ref = forward(cfg, W, ids)
    out = {}
    for kind in kinds:
        row = {}
        for pt in POINTS + ("all",):
            sel = tuple(x for x in POINTS if x != "a") if pt == "all" else (pt,)
            e = forward(cfg, W, ids, sel, kind) - ref
            row[pt] = (float(np.sqrt(np.mean(e * e))), float(np.max(np.abs(e))))
        out[kind] = row
    return out


def main():
    import synth_inputs as si
    ap = argparse.ArgumentParser()
    ap.add_argument("--width", default="8b", choices=sorted(si.MODEL_SHAPES))
    ap.add_argument("--layers", type=int, default=2)
    ap.add_argument("--seq", type=int, default=48)
    args = ap.parse_args()
    shape = dict(si.MODEL_SHAPES[args.width], L=args.layers)
    W = {k: np.asarray(v, dtype=np.float64) for k, v in si.weights_as_f32_numpy(si.make_weights(shape)).items()}
    ids = si.make_ids(1, args.seq, shape["V"])
    cfg = od.DecoderConfig.from_dict(shape)
    res = table(cfg, W, ids)
    print("| rounded to | " + " | ".join(POINTS) + " | all but a |")
    print("|---" * (len(POINTS) + 2) + "|")
    for kind, row in res.items():
        print(f"| {kind} | " + " | ".join(f"{row[p][0]:.1e} / {row[p][1]:.1e}" for p in POINTS + ("all",)) + " |")
    # whole modes: every point rounded as the mode stores it
    ref = forward(cfg, W, ids)
    modes = {"bf16 (one term everywhere)": "bf16",
             "bf16, two terms everywhere but the KV cache": {**{pt: "bf16x2" for pt in POINTS}, "k": "bf16",
                                                             "v": "bf16"},
             "fp16, two-term a (the fp16 prefill)": {**{pt: "fp16" for pt in POINTS}, "a": "fp16x2"}}
    for name, kind in modes.items():
        e = forward(cfg, W, ids, POINTS, kind) - ref
        print(f"{name}: rms {np.sqrt(np.mean(e * e)):.1e}, max {np.max(np.abs(e)):.1e}")


if __name__ == "__main__":
    main()
