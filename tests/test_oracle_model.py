"""Model-level pins for the oracle: a pure-Python loop restatement on tiny
shapes, the L=0 closed form, causality, KV-cached decode versus full
recompute, paged versus contiguous caches and batch independence."""
import math

import numpy as np
import pytest

import synth_inputs as si
from oracle import decoder as od


def tiny_model(L=2, D=8, H=4, G=2, d=4, F=12, V=16, tie=False, bias=True, theta=100.0, eps=1e-5, seed=0, window=0,
               act="silu", qk_norm=False):
    m = dict(L=L, D=D, H=H, G=G, d=d, F=F, V=V, tie=tie, bias=bias, theta=theta, eps=eps, window=window, act=act,
             qk_norm=qk_norm)
    w = si.weights_as_f32_numpy(si.make_weights(m, seed=seed))
    # Large-ish weights so that every term matters at tiny widths.
    w = {k: (v if k.endswith(("layernorm.weight", "q_norm.weight", "k_norm.weight")) or k == "model.norm.weight"
             else v * 20.0)
         for k, v in w.items()}
    return od.DecoderConfig.from_dict(m), w


# ----------------------------------------------------- brute-force restatement
def _bf_forward(cfg, W, ids):
    """Element-by-element restatement with Python loops and the math module:
    full recompute of every position from scratch, no cache, no numpy
    vectorisation."""
    L, D, H, G, d, F, V = cfg.L, cfg.D, cfg.H, cfg.G, cfg.d, cfg.F, cfg.V
    S = len(ids)

    def rms(vec, g):
        ms = sum(t * t for t in vec) / len(vec)
        r = 1.0 / math.sqrt(ms + cfg.eps)
        return [vec[i] * r * float(g[i]) for i in range(len(vec))]

    def lin(vec, Wm, b=None):
        out = []
        for o in range(Wm.shape[0]):
            acc = 0.0
            for k in range(Wm.shape[1]):
                acc += vec[k] * float(Wm[o, k])
            if b is not None:
                acc += float(b[o])
            out.append(acc)
        return out

    def rot(vec, p):
        half = d // 2
        out = [0.0] * d
        for j in range(half):
            ang = p * cfg.theta ** (-2.0 * j / d)
            out[j] = vec[j] * math.cos(ang) - vec[j + half] * math.sin(ang)
            out[j + half] = vec[j + half] * math.cos(ang) + vec[j] * math.sin(ang)
        return out

    xs = [[float(W["model.embed_tokens.weight"][t, i]) for i in range(D)] for t in ids]
    for l in range(L):
        p = f"model.layers.{l}."
        qs, ks, vs = [], [], []
        for s in range(S):
            h = rms(xs[s], W[p + "input_layernorm.weight"])
            q = lin(h, W[p + "self_attn.q_proj.weight"], W.get(p + "self_attn.q_proj.bias"))
            k = lin(h, W[p + "self_attn.k_proj.weight"], W.get(p + "self_attn.k_proj.bias"))
            v = lin(h, W[p + "self_attn.v_proj.weight"], W.get(p + "self_attn.v_proj.bias"))
            qh = [q[hh * d:(hh + 1) * d] for hh in range(H)]
            kh = [k[g * d:(g + 1) * d] for g in range(G)]
            if cfg.qk_norm:
                qh = [rms(v_, W[p + "self_attn.q_norm.weight"]) for v_ in qh]
                kh = [rms(v_, W[p + "self_attn.k_norm.weight"]) for v_ in kh]
            qs.append([rot(v_, s) for v_ in qh])
            ks.append([rot(v_, s) for v_ in kh])
            vs.append([v[g * d:(g + 1) * d] for g in range(G)])
        new_x = []
        for s in range(S):
            o = []
            for hh in range(H):
                g = hh * G // H
                # visible keys: t <= s, and with a window W only the last W of them
                vis = [t for t in range(s + 1) if cfg.window == 0 or s - t < cfg.window]
                sc = [sum(qs[s][hh][j] * ks[t][g][j] for j in range(d)) / math.sqrt(d) for t in vis]
                mx = max(sc)
                e = [math.exp(c - mx) for c in sc]
                z = sum(e)
                for j in range(d):
                    o.append(sum(e[i] / z * vs[t][g][j] for i, t in enumerate(vis)))
            a = lin(o, W[p + "self_attn.o_proj.weight"])
            x1 = [xs[s][i] + a[i] for i in range(D)]
            h2 = rms(x1, W[p + "post_attention_layernorm.weight"])
            gt = lin(h2, W[p + "mlp.gate_proj.weight"])
            up = lin(h2, W[p + "mlp.up_proj.weight"])
            if cfg.act == "gelu_tanh":
                c = math.sqrt(2.0 / math.pi)
                u = [0.5 * gt[i] * (1.0 + math.tanh(c * (gt[i] + 0.044715 * gt[i] ** 3))) * up[i] for i in range(F)]
            else:
                u = [gt[i] / (1.0 + math.exp(-gt[i])) * up[i] for i in range(F)]
            dn = lin(u, W[p + "mlp.down_proj.weight"])
            new_x.append([x1[i] + dn[i] for i in range(D)])
        xs = new_x
    head = W["model.embed_tokens.weight"] if cfg.tie else W["lm_head.weight"]
    return [lin(rms(x, W["model.norm.weight"]), head) for x in xs]


@pytest.mark.parametrize("tie,bias,H,G,window,act,qkn", [
    (False, True, 4, 2, 0, "silu", False), (True, False, 2, 2, 0, "silu", False),
    (False, False, 4, 1, 0, "silu", False), (False, True, 4, 2, 2, "silu", False), (True, False, 2, 2, 3, "silu", False),
    (False, True, 4, 2, 0, "gelu_tanh", False), (False, True, 4, 2, 0, "silu", True)])
def test_oracle_matches_bruteforce_loops(tie, bias, H, G, window, act, qkn):
    cfg, W = tiny_model(tie=tie, bias=bias, H=H, G=G, d=4, D=8, window=window, act=act, qk_norm=qkn)
    ids = [3, 15, 0, 7, 7]
    ref = np.array(_bf_forward(cfg, W, ids))
    o = od.Oracle(cfg, W)
    got = o.prefill(np.array([ids]), o.new_contiguous_cache(1, 8))[0]
    assert np.allclose(got, ref, rtol=1e-12, atol=1e-12)


def test_selected_rows_match_bruteforce_loops_at_those_positions():
    """prefill(rows=...) returns exactly the listed positions' logits (the
    large-shape GPU checks compare sampled rows through it)."""
    cfg, W = tiny_model()
    ids = [3, 15, 0, 7, 7, 2]
    ref = np.array(_bf_forward(cfg, W, ids))
    o = od.Oracle(cfg, W)
    rows = [4, 0, 5]
    got = o.prefill(np.array([ids]), o.new_contiguous_cache(1, 8), rows=rows)[0]
    assert got.shape == (3, cfg.V)
    assert np.allclose(got, ref[rows], rtol=1e-12, atol=1e-12)


# ------------------------------------------------------------- special cases
def test_zero_layers_is_norm_then_head():
    cfg, W = tiny_model(L=0)
    ids = np.array([[1, 4, 9]])
    o = od.Oracle(cfg, W)
    got = o.prefill(ids, o.new_contiguous_cache(1, 4))
    E = W["model.embed_tokens.weight"].astype(np.float64)
    x = E[ids[0]]
    r = 1.0 / np.sqrt(np.mean(x * x, -1, keepdims=True) + cfg.eps)
    want = (x * r * W["model.norm.weight"]) @ W["lm_head.weight"].astype(np.float64).T
    assert np.allclose(got[0], want, rtol=1e-13, atol=1e-13)
    # Tied head reads the embedding matrix.
    cfg_t, W_t = tiny_model(L=0, tie=True)
    ot = od.Oracle(cfg_t, W_t)
    got_t = ot.prefill(ids, ot.new_contiguous_cache(1, 4))
    Et = W_t["model.embed_tokens.weight"].astype(np.float64)
    xt = Et[ids[0]]
    rt = 1.0 / np.sqrt(np.mean(xt * xt, -1, keepdims=True) + cfg_t.eps)
    assert np.allclose(got_t[0], (xt * rt * W_t["model.norm.weight"]) @ Et.T, rtol=1e-13, atol=1e-13)


# ---------------------------------------------------------------- invariants
def test_appending_tokens_leaves_earlier_logits_unchanged():
    cfg, W = tiny_model()
    o = od.Oracle(cfg, W)
    ids = np.array([[5, 1, 2, 11, 3, 8]])
    full = o.prefill(ids, o.new_contiguous_cache(1, 8))
    for k in (1, 3, 5):
        part = o.prefill(ids[:, :k], o.new_contiguous_cache(1, 8))
        assert np.allclose(part, full[:, :k], rtol=1e-12, atol=1e-12)


def test_incremental_decode_equals_full_recompute():
    cfg, W = tiny_model()
    o = od.Oracle(cfg, W)
    ids = np.array([[5, 1, 2, 11, 3, 8, 0, 14], [2, 2, 9, 4, 1, 1, 7, 6]])
    full = o.prefill(ids, o.new_contiguous_cache(2, 8))
    cache = o.new_contiguous_cache(2, 8)
    o.prefill(ids[:, :3], cache)
    for t in range(3, 8):
        step = o.decode_step(ids[:, t], cache, np.array([t, t]))
        assert np.allclose(step, full[:, t], rtol=1e-12, atol=1e-12)


def test_sliding_window_decode_equals_full_recompute_and_differs_from_no_window():
    cfg, W = tiny_model(window=3)
    o = od.Oracle(cfg, W)
    ids = np.array([[5, 1, 2, 11, 3, 8, 0, 14]])
    full = o.prefill(ids, o.new_contiguous_cache(1, 8))
    cache = o.new_contiguous_cache(1, 8)
    o.prefill(ids[:, :2], cache)
    for t in range(2, 8):
        step = o.decode_step(ids[:, t], cache, np.array([t]))
        assert np.allclose(step, full[:, t], rtol=1e-12, atol=1e-12)
    cfg0, _ = tiny_model(window=0)
    o0 = od.Oracle(cfg0, W)
    none = o0.prefill(ids, o0.new_contiguous_cache(1, 8))
    assert np.allclose(none[:, :3], full[:, :3], rtol=1e-12, atol=1e-12)  # the window covers positions 0..2
    assert not np.allclose(none[:, 3:], full[:, 3:])


def test_rope_scaling_changes_only_positions_beyond_zero_and_factor_one_is_off():
    base = dict(L=2, D=8, H=4, G=2, d=4, F=12, V=16, tie=False, bias=True, theta=100.0, eps=1e-5)
    _, W = tiny_model()
    ids = np.array([[5, 1, 2, 11, 3, 8]])

    def run(extra):
        o = od.Oracle(od.DecoderConfig.from_dict(dict(base, **extra)), W)
        return o.prefill(ids, o.new_contiguous_cache(1, 8))

    plain = run({})
    assert np.allclose(run(dict(rope_factor=1.0, rope_low=1.0, rope_high=4.0, rope_orig=64)), plain,
                       rtol=1e-12, atol=1e-12)
    scaled = run(dict(rope_factor=8.0, rope_low=1.0, rope_high=4.0, rope_orig=64))
    assert np.allclose(scaled[:, 0], plain[:, 0], rtol=1e-12, atol=1e-12)  # position 0: no rotation at all
    assert not np.allclose(scaled[:, 1:], plain[:, 1:])


def test_qk_norm_makes_logits_invariant_to_the_scale_of_q_and_k_projections():
    # per-head RMSNorm of q and k removes any positive scale of their
    # projections (bias off, eps negligible against the scaled norms)
    cfg, W = tiny_model(qk_norm=True, bias=False, eps=1e-12)
    ids = np.array([[5, 1, 2, 11, 3, 8]])
    o = od.Oracle(cfg, W)
    base = o.prefill(ids, o.new_contiguous_cache(1, 8))
    W2 = dict(W)
    for l in range(cfg.L):
        W2[f"model.layers.{l}.self_attn.q_proj.weight"] = W[f"model.layers.{l}.self_attn.q_proj.weight"] * 7.0
        W2[f"model.layers.{l}.self_attn.k_proj.weight"] = W[f"model.layers.{l}.self_attn.k_proj.weight"] * 0.25
    o2 = od.Oracle(cfg, W2)
    assert np.allclose(o2.prefill(ids, o2.new_contiguous_cache(1, 8)), base, rtol=1e-10, atol=1e-10)
    cfg0, _ = tiny_model(qk_norm=False, bias=False, eps=1e-12)  # without it the scale matters
    a = od.Oracle(cfg0, W).prefill(ids, od.Oracle(cfg0, W).new_contiguous_cache(1, 8))
    b = od.Oracle(cfg0, W2).prefill(ids, od.Oracle(cfg0, W2).new_contiguous_cache(1, 8))
    assert not np.allclose(a, b)


def test_qk_norm_decode_equals_full_recompute():
    cfg, W = tiny_model(qk_norm=True)
    o = od.Oracle(cfg, W)
    ids = np.array([[5, 1, 2, 11, 3, 8, 0, 14]])
    full = o.prefill(ids, o.new_contiguous_cache(1, 8))
    cache = o.new_contiguous_cache(1, 8)
    o.prefill(ids[:, :3], cache)
    for t in range(3, 8):
        assert np.allclose(o.decode_step(ids[:, t], cache, np.array([t])), full[:, t], rtol=1e-12, atol=1e-12)


def test_paged_cache_is_bit_identical_to_contiguous():
    cfg, W = tiny_model()
    o = od.Oracle(cfg, W)
    B, S, bs = 2, 7, 2
    ids = np.array([[5, 1, 2, 11, 3, 8, 0], [2, 2, 9, 4, 1, 1, 7]])
    bt = si.make_block_table([S + 3, S + 3], bs, 6, 12, seed=3)
    c_cont = o.new_contiguous_cache(B, 12)
    c_page = o.new_paged_cache(12, bs, bt)
    a = o.prefill(ids, c_cont)
    b = o.prefill(ids, c_page)
    assert np.array_equal(a, b)
    lens = np.array([S, S])
    for t in range(3):
        tok = od.argmax_lowest(a[:, -1] if t == 0 else sa)
        sa = o.decode_step(tok, c_cont, lens)
        sb = o.decode_step(tok, c_page, lens)
        assert np.array_equal(sa, sb)
        lens = lens + 1
    # Cache contents sit at the slots the block table names.
    for b_ in range(B):
        for p in range(S + 3):
            blk, off = od.slot_of(bt, b_, p, bs)
            assert np.array_equal(c_page.K[1][blk, off], c_cont.K[1][b_, p])


def test_batch_rows_are_independent():
    cfg, W = tiny_model()
    o = od.Oracle(cfg, W)
    ids = np.array([[5, 1, 2, 11], [2, 2, 9, 4], [0, 13, 13, 1]])
    both = o.prefill(ids, o.new_contiguous_cache(3, 4))
    for b in range(3):
        one = o.prefill(ids[b:b + 1], o.new_contiguous_cache(1, 4))
        assert np.allclose(one[0], both[b], rtol=1e-13, atol=1e-13)


def test_generate_teacher_forced_matches_free_running_when_forced_on_own_tokens():
    cfg, W = tiny_model()
    o = od.Oracle(cfg, W)
    ids = np.array([[5, 1, 2]])
    toks, logits = o.generate(ids, 4, o.new_contiguous_cache(1, 8))
    toks2, logits2 = o.generate(ids, 4, o.new_contiguous_cache(1, 8), forced=toks)
    assert np.array_equal(toks, toks2) and np.allclose(logits, logits2, rtol=1e-14, atol=1e-14)


def test_varlen_equals_batched_forward_for_equal_lengths():
    """forward_varlen over equal-length chunks is the batched forward."""
    cfg, W = tiny_model()
    o = od.Oracle(cfg, W)
    ids = np.random.default_rng(3).integers(0, cfg.V, size=(3, 5))
    c1 = o.new_contiguous_cache(3, 16)
    ref = o.forward(ids, c1, [0, 0, 0])
    c2 = o.new_contiguous_cache(3, 16)
    got = o.forward_varlen([ids[b] for b in range(3)], c2, [0, 0, 0], last_only=False)
    for b in range(3):
        assert np.allclose(got[b], ref[b], rtol=0, atol=1e-12)


@pytest.mark.parametrize("window", [0, 2, 5])
def test_varlen_chunks_equal_one_prompt_and_mixed_decode(window):
    """Prompts cut into chunks of different lengths (one of them a single
    decode-like token) give the logits of the whole prompts, paged cache with
    shuffled blocks included; under a sliding window narrower and wider than
    the chunks too."""
    cfg, W = tiny_model(window=window)
    o = od.Oracle(cfg, W)
    rng = np.random.default_rng(4)
    lens = [7, 4, 9]
    prompts = [rng.integers(0, cfg.V, size=n) for n in lens]
    full = o.new_contiguous_cache(3, 16)
    ref = [o.forward(p[None], od.SeqSlot(full, b), [0])[0] for b, p in enumerate(prompts)]
    cut = [3, 3, 8]  # second sequence: last chunk is one token, like a decode step
    bt = np.random.default_rng(5).permutation(3 * 4).reshape(3, 4)
    for cache in (o.new_contiguous_cache(3, 16), o.new_paged_cache(12, 4, bt)):
        first = o.forward_varlen([p[:c] for p, c in zip(prompts, cut)], cache, [0, 0, 0], last_only=False)
        second = o.forward_varlen([p[c:] for p, c in zip(prompts, cut)], cache, cut, last_only=False)
        for b in range(3):
            assert np.allclose(first[b], ref[b][:cut[b]], rtol=0, atol=1e-12)
            assert np.allclose(second[b], ref[b][cut[b]:], rtol=0, atol=1e-12)
