"""Pins for the CPU oracle: closed forms, invariants, special cases and a
brute-force loop restatement on tiny shapes. None of these compares the
oracle with itself; each would fail on a plausible slip (dropped term, wrong
sign, transposed operand, wrong pairing or head mapping)."""
import math

import numpy as np
import pytest
from scipy.special import expit

from oracle import decoder as od

RNG = np.random.default_rng(1234)


# --------------------------------------------------------------------- RMSNorm
def test_rmsnorm_unit_rms_times_gain():
    x = RNG.normal(size=(5, 37)) * 3.0
    y = od.rmsnorm(x, np.ones(37), 0.0)
    assert np.allclose(np.sqrt(np.mean(y * y, axis=-1)), 1.0, rtol=0, atol=1e-13)
    # A constant gain c scales the RMS to |c| (a "1 + g" reading would give 1 + c).
    y2 = od.rmsnorm(x, np.full(37, 2.0), 0.0)
    assert np.allclose(np.sqrt(np.mean(y2 * y2, axis=-1)), 2.0, atol=1e-13)
    # Per-coordinate gain: y / g has unit RMS.
    g = RNG.uniform(0.5, 1.5, size=37)
    y3 = od.rmsnorm(x, g, 0.0)
    assert np.allclose(np.sqrt(np.mean((y3 / g) ** 2, axis=-1)), 1.0, atol=1e-13)


def test_rmsnorm_eps_inside_sqrt():
    # Constant vector a: a / sqrt(a^2 + eps), closed form.
    a, eps = 0.01, 1e-4
    y = od.rmsnorm(np.full((1, 8), a), np.ones(8), eps)
    assert np.allclose(y, a / math.sqrt(a * a + eps), atol=1e-15)
    assert np.all(od.rmsnorm(np.zeros((2, 4)), np.ones(4), 1e-6) == 0.0)


# ---------------------------------------------------------------------- linear
def test_linear_out_in_convention_bruteforce():
    x = RNG.normal(size=(3, 5))
    W = RNG.normal(size=(7, 5))  # [out, in]
    b = RNG.normal(size=7)
    y = od.linear(x, W, b)
    for i in range(3):
        for o in range(7):
            ref = sum(x[i, k] * W[o, k] for k in range(5)) + b[o]
            assert abs(y[i, o] - ref) < 1e-12


# ------------------------------------------------------------------------ RoPE
def test_rope_closed_form_pairs_and_frequencies():
    # d = 4, theta = 100: inv_freq = [1, 100^(-1/2)] = [1, 0.1]; pairs (0,2), (1,3).
    p = 3.0
    e0 = np.array([1.0, 0.0, 0.0, 0.0])
    e1 = np.array([0.0, 1.0, 0.0, 0.0])
    e2 = np.array([0.0, 0.0, 1.0, 0.0])
    assert np.allclose(od.rope(e0, p, 100.0), [math.cos(p), 0, math.sin(p), 0], atol=1e-15)
    assert np.allclose(od.rope(e1, p, 100.0), [0, math.cos(0.1 * p), 0, math.sin(0.1 * p)], atol=1e-15)
    assert np.allclose(od.rope(e2, p, 100.0), [-math.sin(p), 0, math.cos(p), 0], atol=1e-15)
    assert np.allclose(od.rope_inv_freq(8, 1e4), [1e4 ** (-j / 4) for j in range(4)], rtol=1e-15)


def test_rope_identity_at_zero_and_norm_preserving():
    x = RNG.normal(size=(6, 64))
    assert np.array_equal(od.rope(x, np.zeros(6), 1e6), x)
    y = od.rope(x, np.arange(6) * 997.0, 1e6)
    assert np.allclose(np.linalg.norm(y, axis=-1), np.linalg.norm(x, axis=-1), rtol=1e-13)


def test_rope_dot_depends_only_on_relative_position():
    q = RNG.normal(size=128)
    k = RNG.normal(size=128)
    for pq, pk, s in [(5, 2, 100), (0, 0, 4000), (1234, 17, 3)]:
        a = od.rope(q, pq, 5e5) @ od.rope(k, pk, 5e5)
        b = od.rope(q, pq + s, 5e5) @ od.rope(k, pk + s, 5e5)
        assert abs(a - b) < 1e-10 * (1 + abs(a))


# ------------------------------------------------------------ SiLU / softmax
LLAMA31 = (8.0, 1.0, 4.0, 8192)  # factor, low_freq_factor, high_freq_factor, original context


def test_rope_scaling_factor_one_is_no_scaling():
    f = od.rope_inv_freq(128, 5e5)
    for low, high in [(1.0, 4.0), (2.0, 3.0)]:
        assert np.allclose(od.rope_inv_freq(128, 5e5, (1.0, low, high, 8192)), f, rtol=1e-15, atol=0)


def test_rope_scaling_bands_at_their_closed_form_edges():
    d, theta = 128, 5e5
    factor, low, high, C = LLAMA31
    f = od.rope_inv_freq(d, theta)
    g = od.rope_inv_freq(d, theta, LLAMA31)
    # wavelength 2 pi theta^(2j/d) < C/high  <=>  j < (d/2) ln(C / (2 pi high)) / ln(theta)
    n_keep = math.ceil((d / 2) * math.log(C / (2 * math.pi * high)) / math.log(theta))
    n_stretch_from = math.floor((d / 2) * math.log(C / (2 * math.pi * low)) / math.log(theta)) + 1
    assert 0 < n_keep < n_stretch_from < d // 2
    assert np.array_equal(g[:n_keep], f[:n_keep])
    assert np.allclose(g[n_stretch_from:], f[n_stretch_from:] / factor, rtol=1e-15, atol=0)
    mid = g[n_keep:n_stretch_from] / f[n_keep:n_stretch_from]
    assert np.all((mid < 1.0) & (mid > 1.0 / factor))


def test_rope_scaling_ratio_is_continuous_and_monotone_in_wavelength():
    # 1024 frequencies: the ratio scaled / unscaled falls from 1 to 1/factor
    # without a jump at either band edge (a reversed blend jumps by 7/8)
    g = od.rope_inv_freq(2048, 5e5, LLAMA31)
    r = g / od.rope_inv_freq(2048, 5e5)
    assert r[0] == 1.0 and abs(r[-1] - 1 / 8) < 1e-15
    assert np.all(np.diff(r) <= 1e-15)
    assert np.max(np.abs(np.diff(r))) < 0.05


def test_silu_matches_library_logistic():
    z = np.linspace(-40, 40, 801)
    assert np.allclose(od.silu(z), z * expit(z), rtol=1e-14, atol=1e-300)
    assert od.silu(np.array([0.0]))[0] == 0.0
    assert np.isfinite(od.silu(np.array([-1000.0]))).all()
    g, u = RNG.normal(size=9), RNG.normal(size=9)
    assert np.allclose(od.swiglu(g, u), g * expit(g) * u, rtol=1e-14)


def test_gelu_tanh_against_exact_gelu_and_its_identities():
    from scipy.special import erf
    z = np.linspace(-8, 8, 4001)
    g = od.gelu_tanh(z)
    exact = 0.5 * z * (1 + erf(z / math.sqrt(2)))  # GELU from the normal CDF
    assert np.max(np.abs(g - exact)) < 1e-3  # the tanh form approximates it closely...
    assert np.max(np.abs(g - exact)) > 1e-5  # ...but is not it
    assert np.allclose(g - od.gelu_tanh(-z), z, atol=1e-13)  # gelu(z) - gelu(-z) = z
    assert od.gelu_tanh(0.0) == 0.0
    assert abs(od.gelu_tanh(1.0) - 0.5 * (1 + math.tanh(math.sqrt(2 / math.pi) * 1.044715))) < 1e-15


def test_gated_mlp_activation_choice():
    gate = RNG.normal(size=(3, 5))
    up = RNG.normal(size=(3, 5))
    assert np.allclose(od.swiglu(gate, up), gate * expit(gate) * up, atol=1e-15)
    assert np.allclose(od.swiglu(gate, up, "gelu_tanh"), od.gelu_tanh(gate) * up, atol=1e-15)


def test_softmax_rows_sum_to_one_and_shift_invariant():
    s = RNG.normal(size=(4, 33)) * 10
    a = od.softmax(s)
    assert np.allclose(a.sum(-1), 1.0, atol=1e-14)
    assert np.allclose(od.softmax(s + 123.0), a, atol=1e-15)
    assert np.allclose(od.softmax(np.zeros(5)), 0.2)


# ------------------------------------------------------------------- attention
def test_attention_single_key_returns_v():
    q = RNG.normal(size=(4, 8))
    K = RNG.normal(size=(1, 2, 8))
    V = RNG.normal(size=(1, 2, 8))
    o = od.attention_one_query(q, K, V, 4, 2)
    for h in range(4):
        assert np.allclose(o[h], V[0, h // 2])


def test_attention_equal_scores_average_v():
    q = np.zeros((2, 8))
    K = RNG.normal(size=(5, 1, 8))
    V = RNG.normal(size=(5, 1, 8))
    o = od.attention_one_query(q, K, V, 2, 1)
    assert np.allclose(o[0], V[:, 0].mean(0), atol=1e-15)


def test_attention_two_key_closed_form_scale():
    d = 16
    q = np.zeros((1, d))
    q[0, 0] = 1.0
    K = np.zeros((2, 1, d))
    K[0, 0, 0], K[1, 0, 0] = 3.0, -1.0
    V = np.zeros((2, 1, d))
    V[0, 0, 1], V[1, 0, 1] = 1.0, 0.0
    o = od.attention_one_query(q, K, V, 1, 1)
    w0 = 1.0 / (1.0 + math.exp(-(3.0 - (-1.0)) / math.sqrt(d)))  # scale 1/sqrt(d)
    assert abs(o[0, 1] - w0) < 1e-15


def test_gqa_head_mapping_contiguous_groups():
    H, G, d, T = 8, 2, 4, 3
    q = RNG.normal(size=(H, d))
    K = RNG.normal(size=(T, G, d))
    V = np.zeros((T, G, d))
    for g in range(G):
        V[:, g, :] = g + 1.0
    o = od.attention_one_query(q, K, V, H, G)
    for h in range(H):
        assert np.allclose(o[h], h // (H // G) + 1.0)  # head h -> KV head h // (H/G)


def test_gqa_with_H_equal_G_is_mha_and_repeat_kv():
    H, d, T = 3, 8, 6
    q = RNG.normal(size=(T, H, d))
    K = RNG.normal(size=(T, H, d))
    V = RNG.normal(size=(T, H, d))
    o = od.causal_attention(q, K, V, np.arange(T), H, H)
    # Repeat-kv restatement of GQA with G=1 for 3 heads.
    K1, V1 = K[:, :1], V[:, :1]
    og = od.causal_attention(q, K1, V1, np.arange(T), H, 1)
    for i in range(T):
        for h in range(H):
            s = np.array([q[i, h] @ K[t, h] / math.sqrt(d) for t in range(i + 1)])
            a = np.exp(s - s.max()); a /= a.sum()
            assert np.allclose(o[i, h], a @ V[: i + 1, h], atol=1e-13)
            s1 = np.array([q[i, h] @ K1[t, 0] / math.sqrt(d) for t in range(i + 1)])
            a1 = np.exp(s1 - s1.max()); a1 /= a1.sum()
            assert np.allclose(og[i, h], a1 @ V1[: i + 1, 0], atol=1e-13)


def test_causal_mask_ignores_future_keys():
    S, H, G, d = 5, 2, 1, 4
    q = RNG.normal(size=(S, H, d))
    K = RNG.normal(size=(S, G, d))
    V = RNG.normal(size=(S, G, d))
    o = od.causal_attention(q, K, V, np.arange(S), H, G)
    K2, V2 = K.copy(), V.copy()
    K2[3:] = 99.0
    V2[3:] = -99.0
    o2 = od.causal_attention(q, K2, V2, np.arange(S), H, G)
    assert np.array_equal(o[:3], o2[:3])
    assert not np.allclose(o[3:], o2[3:])


def test_window_one_sees_only_its_own_key():
    S, H, G, d = 6, 4, 2, 8
    q = RNG.normal(size=(S, H, d))
    K = RNG.normal(size=(S, G, d))
    V = RNG.normal(size=(S, G, d))
    o = od.causal_attention(q, K, V, np.arange(S), H, G, window=1)
    for i in range(S):
        for h in range(H):
            assert np.allclose(o[i, h], V[i, h // 2], atol=1e-15)


def test_window_covering_the_context_is_no_window():
    S, H, G, d = 7, 2, 1, 4
    q = RNG.normal(size=(S, H, d))
    K = RNG.normal(size=(S, G, d))
    V = RNG.normal(size=(S, G, d))
    full = od.causal_attention(q, K, V, np.arange(S), H, G)
    for w in (S, S + 5):
        assert np.array_equal(od.causal_attention(q, K, V, np.arange(S), H, G, window=w), full)


def test_window_two_reduces_to_two_key_attention():
    # query at position 4 with window 2 attends keys 3 and 4 only: the
    # single-query attention over exactly those keys
    S, H, G, d = 5, 2, 2, 8
    q = RNG.normal(size=(S, H, d))
    K = RNG.normal(size=(S, G, d))
    V = RNG.normal(size=(S, G, d))
    o = od.causal_attention(q, K, V, np.arange(S), H, G, window=2)
    assert np.allclose(o[4], od.attention_one_query(q[4], K[3:5], V[3:5], H, G), atol=1e-14)
    assert np.allclose(o[0], V[0][[0, 1]], atol=1e-15)  # position 0: only itself


def test_window_ignores_keys_that_slid_out():
    S, H, G, d, W = 9, 2, 1, 4, 3
    q = RNG.normal(size=(S, H, d))
    K = RNG.normal(size=(S, G, d))
    V = RNG.normal(size=(S, G, d))
    o = od.causal_attention(q, K, V, np.arange(S), H, G, window=W)
    K2, V2 = K.copy(), V.copy()
    K2[2], V2[2] = 50.0, -50.0  # visible to positions 2, 3, 4 only
    o2 = od.causal_attention(q, K2, V2, np.arange(S), H, G, window=W)
    assert np.array_equal(o[:2], o2[:2]) and np.array_equal(o[5:], o2[5:])
    assert not np.allclose(o[2:5], o2[2:5])


# ------------------------------------------------------------- integer helpers
def test_slot_of_and_argmax_ties():
    bt = np.array([[7, 2, 9], [0, 5, 1]])
    assert od.slot_of(bt, 0, 0, 16) == (7, 0)
    assert od.slot_of(bt, 0, 17, 16) == (2, 1)
    assert od.slot_of(bt, 1, 47, 16) == (1, 15)
    assert od.argmax_lowest(np.array([[1.0, 3.0, 3.0, 2.0]]))[0] == 1
    assert od.argmax_lowest(np.array([[-1.0, -1.0]]))[0] == 0
