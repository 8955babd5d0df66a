"""Pins for the GPT-2 oracle (the appendix's complete model): LayerNorm
closed forms and invariances, the [in, out] weight convention, a pure-Python
loop restatement of the whole forward, the zero-layer closed form, causality,
cached decode against full recompute, and learned positions."""
import math

import numpy as np
import pytest

import synth_inputs as si
from oracle import gpt2 as og

RNG = np.random.default_rng(77)


def tiny(L=2, D=8, H=2, V=16, P=12, seed=0):
    c = dict(L=L, D=D, H=H, V=V, P=P)
    w = si.weights_as_f32_numpy(si.make_gpt2_weights(c, seed=seed))
    # larger weights so that every term matters at tiny widths
    w = {k: (v if ".ln_" in k else v * 20.0) for k, v in w.items()}
    return og.GPT2Config.from_dict(c), w


def test_layernorm_unit_variance_zero_mean_and_constant_vector():
    x = RNG.normal(size=(5, 32)) * 3 + 7
    y = og.layernorm(x, np.ones(32), np.zeros(32), 1e-12)
    assert np.allclose(y.mean(-1), 0, atol=1e-12)
    assert np.allclose(y.var(-1), 1, atol=1e-9)
    b = RNG.normal(size=32)
    assert np.allclose(og.layernorm(np.full((2, 32), 4.2), RNG.normal(size=32), b, 1e-5), b, atol=1e-12)


def test_layernorm_ignores_shift_and_positive_scale():
    x = RNG.normal(size=(3, 16))
    g, b = RNG.normal(size=16), RNG.normal(size=16)
    y = og.layernorm(x, g, b, 1e-12)
    assert np.allclose(og.layernorm(x + 5.0, g, b, 1e-12), y, atol=1e-10)
    assert np.allclose(og.layernorm(x * 9.0, g, b, 1e-12), y, atol=1e-10)
    assert not np.allclose(og.layernorm(x * 9.0, g, b, 1.0), og.layernorm(x, g, b, 1.0))  # eps inside the root


def test_transposed_linear_reads_in_out():
    x = RNG.normal(size=(2, 3))
    W = RNG.normal(size=(3, 5))
    b = RNG.normal(size=5)
    y = og.linear_t(x, W, b)
    for r in range(2):
        for j in range(5):
            assert abs(y[r, j] - (sum(x[r, i] * W[i, j] for i in range(3)) + b[j])) < 1e-13


def _bf(cfg, W, ids):
    """Loop restatement with the math module: every position from scratch."""
    D, H, V = cfg.D, cfg.H, cfg.V
    d = D // H

    def ln(v, g, b):
        mu = sum(v) / len(v)
        var = sum((t - mu) ** 2 for t in v) / len(v)
        return [(v[i] - mu) / math.sqrt(var + cfg.eps) * float(g[i]) + float(b[i]) for i in range(len(v))]

    def lin(v, Wm, b):
        return [sum(v[i] * float(Wm[i, j]) for i in range(len(v))) + float(b[j]) for j in range(Wm.shape[1])]

    def gelu(z):
        return 0.5 * z * (1.0 + math.tanh(math.sqrt(2.0 / math.pi) * (z + 0.044715 * z ** 3)))

    xs = [[float(W["transformer.wte.weight"][t, i]) + float(W["transformer.wpe.weight"][s, i]) for i in range(D)]
          for s, t in enumerate(ids)]
    for l in range(cfg.L):
        p = f"transformer.h.{l}."
        qkv = [lin(ln(x, W[p + "ln_1.weight"], W[p + "ln_1.bias"]), W[p + "attn.c_attn.weight"],
                   W[p + "attn.c_attn.bias"]) for x in xs]
        new = []
        for s in range(len(xs)):
            o = []
            for h in range(H):
                q = qkv[s][h * d:(h + 1) * d]
                sc = [sum(q[j] * qkv[t][D + h * d + j] for j in range(d)) / math.sqrt(d) for t in range(s + 1)]
                mx = max(sc)
                e = [math.exp(c - mx) for c in sc]
                z = sum(e)
                o += [sum(e[t] / z * qkv[t][2 * D + h * d + j] for t in range(s + 1)) for j in range(d)]
            a = lin(o, W[p + "attn.c_proj.weight"], W[p + "attn.c_proj.bias"])
            x1 = [xs[s][i] + a[i] for i in range(D)]
            u = [gelu(t) for t in lin(ln(x1, W[p + "ln_2.weight"], W[p + "ln_2.bias"]), W[p + "mlp.c_fc.weight"],
                                      W[p + "mlp.c_fc.bias"])]
            m = lin(u, W[p + "mlp.c_proj.weight"], W[p + "mlp.c_proj.bias"])
            new.append([x1[i] + m[i] for i in range(D)])
        xs = new
    E = W["transformer.wte.weight"]
    out = []
    for x in xs:
        h = ln(x, W["transformer.ln_f.weight"], W["transformer.ln_f.bias"])
        out.append([sum(h[i] * float(E[v, i]) for i in range(D)) for v in range(V)])
    return out


@pytest.mark.parametrize("H", [1, 2, 4])
def test_gpt2_oracle_matches_bruteforce_loops(H):
    cfg, W = tiny(H=H)
    ids = [3, 15, 0, 7, 7, 2]
    o = og.GPT2Oracle(cfg, W)
    got = o.prefill(np.array([ids]), o.new_cache(1, 12))[0]
    assert np.allclose(got, np.array(_bf(cfg, W, ids)), rtol=1e-12, atol=1e-12)


def test_zero_layers_is_final_layernorm_then_tied_head():
    cfg, W = tiny(L=0)
    ids = np.array([[1, 4, 9]])
    o = og.GPT2Oracle(cfg, W)
    got = o.prefill(ids, o.new_cache(1, 4))[0]
    E = W["transformer.wte.weight"].astype(np.float64)
    x = E[ids[0]] + W["transformer.wpe.weight"][:3].astype(np.float64)
    mu = x.mean(-1, keepdims=True)
    y = (x - mu) / np.sqrt(((x - mu) ** 2).mean(-1, keepdims=True) + cfg.eps)
    y = y * W["transformer.ln_f.weight"] + W["transformer.ln_f.bias"]
    assert np.allclose(got, y @ E.T, rtol=1e-12, atol=1e-12)


def test_causality_and_cached_decode_equal_full_recompute():
    cfg, W = tiny()
    o = og.GPT2Oracle(cfg, W)
    ids = np.array([[5, 1, 2, 11, 3, 8, 0, 14], [2, 2, 9, 4, 1, 1, 7, 6]])
    full = o.prefill(ids, o.new_cache(2, 12))
    for k in (1, 4):
        assert np.allclose(o.prefill(ids[:, :k], o.new_cache(2, 12)), full[:, :k], rtol=1e-12, atol=1e-12)
    cache = o.new_cache(2, 12)
    o.prefill(ids[:, :3], cache)
    for t in range(3, 8):
        assert np.allclose(o.decode_step(ids[:, t], cache, np.array([t, t])), full[:, t], rtol=1e-12, atol=1e-12)


def test_learned_position_row_is_past_length_plus_offset():
    # zero layers: position p enters only through row p of the position table
    cfg, W = tiny(L=0)
    o = og.GPT2Oracle(cfg, W)
    E = W["transformer.wte.weight"].astype(np.float64)
    P = W["transformer.wpe.weight"].astype(np.float64)
    got = o.forward(np.array([[4, 9]]), o.new_cache(1, 12), [3])[0]
    for i, (t, p) in enumerate([(4, 3), (9, 4)]):
        x = E[t] + P[p]
        y = (x - x.mean()) / np.sqrt(((x - x.mean()) ** 2).mean() + cfg.eps)
        y = y * W["transformer.ln_f.weight"] + W["transformer.ln_f.bias"]
        assert np.allclose(got[i], y @ E.T, rtol=1e-12, atol=1e-12)
    W0 = dict(W)
    W0["transformer.wpe.weight"] = np.zeros_like(P)
    o0 = og.GPT2Oracle(cfg, W0)
    assert np.allclose(o0.forward(np.array([[4]]), o0.new_cache(1, 12), [0]),
                       o0.forward(np.array([[4]]), o0.new_cache(1, 12), [7]), rtol=1e-13, atol=1e-13)
