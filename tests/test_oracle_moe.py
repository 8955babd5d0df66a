"""Pins of the oracle's mixture-of-experts MLP (MoE.softmax_topk_router and
the grouped experts): a pure-Python loop restatement on tiny shapes, the
special cases that reduce to the dense SwiGLU MLP, invariance under a
relabelling of the experts, the tie rule of the top-k, teacher-forced
routing, and the decoder-level properties (cached decode = full recompute,
leading dense layers)."""
import math

import numpy as np
import pytest

import synth_inputs as si
from oracle import decoder as od

BASE = dict(L=2, D=8, H=2, G=1, d=4, F=12, V=16, tie=False, bias=False, theta=100.0, eps=1e-5,
            n_experts=4, top_k=2, moe_F=6, n_shared=1, first_dense=1, norm_topk=False)


def tiny(**over):
    m = dict(BASE, **over)
    w = si.weights_as_f32_numpy(si.make_weights(m, seed=3))
    w = {k: (v if k.endswith("layernorm.weight") or k == "model.norm.weight" else v * 20.0) for k, v in w.items()}
    return m, od.DecoderConfig.from_dict(m), w


def _bf_moe(h, W, p, m):
    """Element-by-element restatement with Python loops and the math module."""
    D, E, k = m["D"], m["n_experts"], m["top_k"]
    Wr = W[p + "mlp.gate.weight"]
    out = []
    for row in h:
        logits = [sum(float(row[i]) * float(Wr[e, i]) for i in range(D)) for e in range(E)]
        mx = max(logits)
        ex = [math.exp(v - mx) for v in logits]
        tot = sum(ex)
        prob = [v / tot for v in ex]
        chosen, left = [], list(range(E))
        for _ in range(k):  # repeated maximum, lowest index first among equals
            best = left[0]
            for e in left:
                if prob[e] > prob[best]:
                    best = e
            chosen.append(best)
            left.remove(best)
        wts = [prob[e] for e in chosen]
        if m["norm_topk"]:
            s = sum(wts)
            wts = [v / s for v in wts]

        def mlp(prefix, width):
            g = [sum(float(row[i]) * float(W[prefix + "gate_proj.weight"][f, i]) for i in range(D)) for f in range(width)]
            u = [sum(float(row[i]) * float(W[prefix + "up_proj.weight"][f, i]) for i in range(D)) for f in range(width)]
            a = [g[f] / (1.0 + math.exp(-g[f])) * u[f] for f in range(width)]
            return [sum(a[f] * float(W[prefix + "down_proj.weight"][o, f]) for f in range(width)) for o in range(D)]

        y = [0.0] * D
        for e, wt in zip(chosen, wts):
            ye = mlp(f"{p}mlp.experts.{e}.", m["moe_F"])
            y = [y[o] + wt * ye[o] for o in range(D)]
        if m["n_shared"]:
            ys = mlp(p + "mlp.shared_experts.", m["n_shared"] * m["moe_F"])
            y = [y[o] + ys[o] for o in range(D)]
        out.append(y)
    return np.array(out)


@pytest.mark.parametrize("norm_topk,n_shared,top_k", [(False, 1, 2), (True, 0, 3), (False, 0, 1)])
def test_moe_mlp_matches_bruteforce_loops(norm_topk, n_shared, top_k):
    m, cfg, W = tiny(norm_topk=norm_topk, n_shared=n_shared, top_k=top_k)
    o = od.Oracle(cfg, W)
    h = np.random.Generator(np.random.PCG64(5)).standard_normal((5, m["D"]))
    got = o.moe_mlp(h, "model.layers.1.")
    assert np.allclose(got, _bf_moe(h, W, "model.layers.1.", m), rtol=1e-12, atol=1e-12)


def test_one_expert_top1_is_the_dense_swiglu_mlp():
    m, cfg, W = tiny(n_experts=1, top_k=1, n_shared=0)
    o = od.Oracle(cfg, W)
    h = np.random.Generator(np.random.PCG64(6)).standard_normal((4, m["D"]))
    e = "model.layers.1.mlp.experts.0."
    dense = od.linear(od.swiglu(od.linear(h, W[e + "gate_proj.weight"]), od.linear(h, W[e + "up_proj.weight"])),
                      W[e + "down_proj.weight"])
    assert np.allclose(o.moe_mlp(h, "model.layers.1."), dense, rtol=1e-13, atol=1e-13)


@pytest.mark.parametrize("norm_topk", [True, False])
def test_identical_experts_give_the_dense_mlp_times_the_weight_sum(norm_topk):
    m, cfg, W = tiny(norm_topk=norm_topk, n_shared=0)
    p = "model.layers.1.mlp.experts."
    for e in range(1, m["n_experts"]):
        for n in ("gate_proj", "up_proj", "down_proj"):
            W[f"{p}{e}.{n}.weight"] = W[f"{p}0.{n}.weight"]
    o = od.Oracle(cfg, W)
    h = np.random.Generator(np.random.PCG64(7)).standard_normal((6, m["D"]))
    dense = od.linear(od.swiglu(od.linear(h, W[p + "0.gate_proj.weight"]), od.linear(h, W[p + "0.up_proj.weight"])),
                      W[p + "0.down_proj.weight"])
    got = o.moe_mlp(h, "model.layers.1.")
    idx, w, prob = o.last_routing["model.layers.1."]
    scale = np.ones((6, 1)) if norm_topk else np.sort(prob, -1)[:, ::-1][:, :m["top_k"]].sum(-1, keepdims=True)
    assert np.allclose(got, dense * scale, rtol=1e-12, atol=1e-12)


def test_relabelling_the_experts_changes_nothing():
    m, cfg, W = tiny()
    perm = [2, 0, 3, 1]
    W2 = dict(W)
    p = "model.layers.1.mlp."
    W2[p + "gate.weight"] = W[p + "gate.weight"][perm]
    for new, old in enumerate(perm):
        for n in ("gate_proj", "up_proj", "down_proj"):
            W2[f"{p}experts.{new}.{n}.weight"] = W[f"{p}experts.{old}.{n}.weight"]
    h = np.random.Generator(np.random.PCG64(8)).standard_normal((5, m["D"]))
    a = od.Oracle(cfg, W).moe_mlp(h, "model.layers.1.")
    b = od.Oracle(cfg, W2).moe_mlp(h, "model.layers.1.")
    assert np.allclose(a, b, rtol=1e-12, atol=1e-12)


def test_topk_ties_take_the_lowest_index():
    p = np.array([[0.1, 0.3, 0.3, 0.2, 0.3], [0.25, 0.25, 0.25, 0.25, 0.0]])
    assert od.topk_lowest(p, 2).tolist() == [[1, 2], [0, 1]]
    idx, w, _ = od.moe_route(np.zeros((1, 3)), np.zeros((4, 3)), 2, True)  # equal logits
    assert idx.tolist() == [[0, 1]] and np.allclose(w, 0.5)


def test_forced_routing_with_the_routers_own_choice_is_unchanged():
    m, cfg, W = tiny()
    o = od.Oracle(cfg, W)
    h = np.random.Generator(np.random.PCG64(9)).standard_normal((5, m["D"]))
    a = o.moe_mlp(h, "model.layers.1.")
    idx = o.last_routing["model.layers.1."][0]
    b = o.moe_mlp(h, "model.layers.1.", forced=idx)
    assert np.array_equal(a, b)
    other = (idx + 1) % m["n_experts"]
    assert not np.allclose(o.moe_mlp(h, "model.layers.1.", forced=other), a)


def test_moe_decoder_cached_decode_equals_full_recompute_and_first_layer_is_dense():
    m, cfg, W = tiny(L=3)
    assert not cfg.is_moe_layer(0) and cfg.is_moe_layer(1) and cfg.is_moe_layer(2)
    assert "model.layers.0.mlp.gate_proj.weight" in W and "model.layers.0.mlp.gate.weight" not in W
    o = od.Oracle(cfg, W)
    ids = np.array([[5, 1, 2, 11, 3, 8, 0, 14]])
    full = o.prefill(ids, o.new_contiguous_cache(1, 8))
    cache = o.new_contiguous_cache(1, 8)
    o.prefill(ids[:, :4], cache)
    for t in range(4, 8):
        step = o.decode_step(ids[:, t], cache, np.array([t]))
        assert np.allclose(step, full[:, t], rtol=1e-11, atol=1e-11)
