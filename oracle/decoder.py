"""Plain float64 CPU oracle of the Llama-family decoder forward.

TEST INFRASTRUCTURE ONLY (see the package docstring): the product path never
imports this module, and this module imports nothing from the product.

What it computes follows the Axon paper (arxiv 2608.19889):

* the pre-norm residual block -- `h <- NN.rmsnorm@ln x; a <- attention h ...;
  return x + a` (Sec. "The Axon Language", Syntax paragraph);
* the core built-ins `NN.embedding`, `NN.linear` (weights `[out, in]`, default
  `bias=true` that Llama checkpoints leave out except on q/k/v), `NN.rmsnorm`
  (Sec. "Built-In Libraries", core built-ins listing; running example of the
  compiler stages for the `bias=true` default);
* `Attention.attention` with grouped-query heads, causal masks and the
  `1.0 / sqrt HD` scale (Sec. "Built-In Libraries", the tensor/math listing
  `scale_heads` and the attention-and-masking paragraph);
* `Positions.position_ids ... past_length=past_len` and the `Cache`
  built-ins, dynamic and static overlays with one interface (Sec.
  "Built-In Libraries", positions and cache management);
* `Act.swiglu` between `NN.linear@up` and `NN.linear@down` (appendix,
  function application and composition listing);
* the model skeleton -- embedding, a `for` loop over layers that threads the
  cache, final norm and a tied or untied LM head (appendix GPT-2 causal_lm
  listing);
* greedy generation, counting generated tokens (Sec. "Results", Measures).

The paper prints no formulas for these operations. Each place where it is
silent takes the reading listed in READINGS below.

Precision: every input (weights that are exact bf16 values, ids) is widened
to float64 and every product, sum and transcendental is float64. Nothing is
rounded back to bf16: the oracle is the exact-arithmetic target the GPU path
is compared against.
"""
from __future__ import annotations

import math
from dataclasses import dataclass

import numpy as np

READINGS = [
    "RMSNorm: y = x / sqrt(mean(x^2) + eps) * g; the gain multiplies the "
    "normalised vector (not 1+g); eps sits inside the square root.",
    "RoPE: rotate-half pairing (j, j + d/2), inv_freq_j = theta^(-2j/d), "
    "angle = position * inv_freq_j; no frequency scaling unless configured "
    "(next entry).",
    "Positions: the i-th new token of sequence b has position past_b + i, "
    "past_b = tokens already in the cache.",
    "GQA: query head h reads KV head floor(h / (H/G)) (contiguous groups).",
    "Attention scale 1/sqrt(d), causal mask keeps keys with position <= "
    "query position, softmax with max subtraction.",
    "Biases: q, k, v only (when attention_bias); never on o, gate, up, down.",
    "SwiGLU: silu(h Wg^T) * (h Wu^T), silu(z) = z / (1 + exp(-z)); with "
    "hidden_act gelu_tanh the gate takes gelu_new, 0.5 z (1 + tanh(sqrt(2/pi) "
    "(z + 0.044715 z^3))), the GELU of the GPT-2 listing.",
    "LM head: logits = rmsnorm(x) Whead^T with Whead = embedding when tied.",
    "Greedy next token: argmax of the logits, lowest index on ties.",
    "KV cache: keys stored after RoPE; the paged overlay maps position p of "
    "sequence b to block_table[b][p // block_size], offset p % block_size.",
    "RoPE frequency scaling (Llama-3.1-family checkpoints; off unless "
    "rope_factor > 0): with wavelength w_j = 2 pi / f_j and the original "
    "context C, frequencies with w_j < C / high_freq_factor stay, those with "
    "w_j > C / low_freq_factor are divided by the factor, and in between "
    "f_j is blended linearly in t = (C / w_j - low) / (high - low): "
    "(1 - t) f_j / factor + t f_j.",
    "qk-norm (Qwen3-family layers, off unless configured): after the q and "
    "k projections (and biases), each head's d values go through the same "
    "RMSNorm as the hidden state, with gains q_norm / k_norm of length d, "
    "before RoPE.",
    "Mixture of experts (the MoE built-ins: MoE.softmax_topk_router and "
    "grouped experts; off unless n_experts > 0): layers from first_dense on "
    "replace the MLP by p = softmax(h Wr^T) over the E experts, the top_k "
    "experts by p (lowest index on ties), weights p of those (divided by "
    "their sum when norm_topk), y = sum_j w_j * swiglu-MLP_e_j(h), plus the "
    "shared experts' SwiGLU MLP of width n_shared * F_e when n_shared > 0 "
    "(DeepSeek-MoE layout; HF names mlp.gate, mlp.experts.{e}.*, "
    "mlp.shared_experts.*).",
    "Sliding window (the `window=` argument of causal_mask_for_input in the "
    "appendix GPT-2 listing): with window W > 0 a query at position p sees "
    "the keys at positions t with p - W < t <= p (itself and the W - 1 "
    "before it); W = 0 means no window.",
]


@dataclass(frozen=True)
class DecoderConfig:
    """HF config.json equivalents read through `Config.dim @@key` (appendix
    GPT-2 causal_lm listing reads n_embd, n_layer, n_head, vocab_size the same
    way)."""

    L: int  # num_hidden_layers
    D: int  # hidden_size
    H: int  # num_attention_heads
    G: int  # num_key_value_heads
    d: int  # head_dim
    F: int  # intermediate_size
    V: int  # vocab_size
    tie: bool  # tie_word_embeddings
    bias: bool  # attention_bias (q, k, v)
    theta: float  # rope_theta
    eps: float  # rms_norm_eps
    window: int = 0  # sliding_window (0: none)
    # rope_scaling of Llama-3.1-family configs (rope_factor 0: none)
    rope_factor: float = 0.0
    rope_low: float = 1.0  # low_freq_factor
    rope_high: float = 4.0  # high_freq_factor
    rope_orig: int = 8192  # original_max_position_embeddings
    act: str = "silu"  # hidden_act of the gated MLP: "silu" or "gelu_tanh"
    qk_norm: bool = False  # per-head RMSNorm of q and k before RoPE (Qwen3-family layers)
    # mixture of experts (n_experts 0: every layer has the dense MLP)
    n_experts: int = 0  # E routed experts
    top_k: int = 0  # experts per token
    moe_F: int = 0  # intermediate size of one expert
    n_shared: int = 0  # shared experts (one dense MLP of width n_shared * moe_F)
    first_dense: int = 0  # leading layers that keep the dense MLP (width F)
    norm_topk: bool = False  # divide the top-k weights by their sum

    @staticmethod
    def from_dict(c: dict) -> "DecoderConfig":
        return DecoderConfig(L=int(c["L"]), D=int(c["D"]), H=int(c["H"]), G=int(c["G"]),
                             d=int(c["d"]), F=int(c["F"]), V=int(c["V"]), tie=bool(c["tie"]),
                             bias=bool(c["bias"]), theta=float(c["theta"]), eps=float(c["eps"]),
                             window=int(c.get("window", 0)), rope_factor=float(c.get("rope_factor", 0.0)),
                             rope_low=float(c.get("rope_low", 1.0)), rope_high=float(c.get("rope_high", 4.0)),
                             rope_orig=int(c.get("rope_orig", 8192)), act=str(c.get("act", "silu")),
                             qk_norm=bool(c.get("qk_norm", False)), n_experts=int(c.get("n_experts", 0)),
                             top_k=int(c.get("top_k", 0)), moe_F=int(c.get("moe_F", 0)),
                             n_shared=int(c.get("n_shared", 0)), first_dense=int(c.get("first_dense", 0)),
                             norm_topk=bool(c.get("norm_topk", False)))

    def is_moe_layer(self, l: int) -> bool:
        return self.n_experts > 0 and l >= self.first_dense

    def rope_scaling(self):
        """(factor, low_freq_factor, high_freq_factor, original context), or None."""
        return (self.rope_factor, self.rope_low, self.rope_high, self.rope_orig) if self.rope_factor > 0 else None


# ---------------------------------------------------------------------------
# Elementary operations
# ---------------------------------------------------------------------------

def rmsnorm(x, g, eps):
    """NN.rmsnorm (Sec. Built-In Libraries, core built-ins listing; the
    pre-norm block of Sec. The Axon Language): scale each vector along the
    last axis to unit root-mean-square, then multiply by the gain g."""
    x = np.asarray(x, dtype=np.float64)
    ms = np.mean(x * x, axis=-1, keepdims=True)
    return x / np.sqrt(ms + eps) * np.asarray(g, dtype=np.float64)


def linear(x, W, b=None):
    """NN.linear (Sec. Built-In Libraries; compiler running example): y = x W^T
    (+ b), W stored `[out, in]` as in HF checkpoints."""
    y = np.asarray(x, dtype=np.float64) @ np.asarray(W, dtype=np.float64).T
    if b is not None:
        y = y + np.asarray(b, dtype=np.float64)
    return y


def rope_inv_freq(d, theta, scaling=None):
    """Positions (Sec. Built-In Libraries, positions and cache management):
    rotary inverse frequencies theta^(-2j/d), j = 0 .. d/2-1.

    scaling = (factor, low_freq_factor, high_freq_factor, original context C)
    applies the frequency-dependent stretch of Llama-3.1-family checkpoints
    (one of the families the paper's benchmarks cover, Sec. Sub-4B Models):
    each frequency's wavelength 2 pi / f is compared with C / high and
    C / low; short wavelengths keep f, long ones take f / factor, and the
    band between blends the two linearly in C / wavelength."""
    j = np.arange(d // 2, dtype=np.float64)
    f = np.power(float(theta), -2.0 * j / d)
    if scaling is None:
        return f
    factor, low, high, C = (float(v) for v in scaling)
    wavelen = 2.0 * math.pi / f
    out = np.empty_like(f)
    for i in range(f.shape[0]):
        if wavelen[i] < C / high:  # high frequency: unchanged
            out[i] = f[i]
        elif wavelen[i] > C / low:  # low frequency: stretched by the factor
            out[i] = f[i] / factor
        else:  # between: linear blend in C / wavelength
            t = (C / wavelen[i] - low) / (high - low)
            out[i] = (1.0 - t) * f[i] / factor + t * f[i]
    return out


def rope(x, pos, theta, scaling=None):
    """Rotary embedding applied by `rope_apply` (Table 6 call counts) with the
    rotate-half pairing: for j < d/2,
        out_j       = x_j cos(p f_j) - x_{j+d/2} sin(p f_j)
        out_{j+d/2} = x_{j+d/2} cos(p f_j) + x_j sin(p f_j).
    x: [..., d]; pos broadcasts against x[..., 0]."""
    x = np.asarray(x, dtype=np.float64)
    d = x.shape[-1]
    f = rope_inv_freq(d, theta, scaling)
    ang = np.asarray(pos, dtype=np.float64)[..., None] * f
    c, s = np.cos(ang), np.sin(ang)
    x1, x2 = x[..., : d // 2], x[..., d // 2:]
    return np.concatenate([x1 * c - x2 * s, x2 * c + x1 * s], axis=-1)


def silu(z):
    """Activations.silu (Sec. Built-In Libraries, activations): z / (1 + e^-z)."""
    z = np.asarray(z, dtype=np.float64)
    with np.errstate(over="ignore"):
        return z / (1.0 + np.exp(-z))


def gelu_tanh(z):
    """Activations.gelu_new (appendix GPT-2 listing; Sec. Built-In Libraries,
    activations), the tanh form of GELU:
    0.5 z (1 + tanh(sqrt(2/pi) (z + 0.044715 z^3)))."""
    z = np.asarray(z, dtype=np.float64)
    return 0.5 * z * (1.0 + np.tanh(math.sqrt(2.0 / math.pi) * (z + 0.044715 * z ** 3)))


def swiglu(gate, up, act="silu"):
    """Act.swiglu between NN.linear@up and NN.linear@down (appendix, function
    application listing): silu(gate) * up; with act="gelu_tanh" the gate
    goes through gelu_new instead (the gated-GELU MLP)."""
    a = gelu_tanh(gate) if act == "gelu_tanh" else silu(gate)
    return a * np.asarray(up, dtype=np.float64)


def topk_lowest(p, k):
    """Indices of the k largest entries along the last axis, largest first;
    among equal entries the lower index comes first."""
    p = np.asarray(p)
    return np.argsort(-p, axis=-1, kind="stable")[..., :k]


def moe_route(h, Wr, top_k, norm_topk, forced=None):
    """MoE.softmax_topk_router (Sec. Built-In Libraries, specialised
    modules listing): router probabilities p = softmax(h Wr^T) over the
    experts, the top_k experts by p and their weights (divided by their sum
    when norm_topk). h: [T, D]; Wr: [E, D]. With `forced` [T, k] the given
    experts are taken instead of the top_k (teacher-forced routing).
    Returns (experts [T, k], weights [T, k], p [T, E])."""
    p = softmax(linear(h, Wr), axis=-1)
    idx = topk_lowest(p, top_k) if forced is None else np.asarray(forced, dtype=np.int64)
    w = np.take_along_axis(p, idx, axis=-1)
    if norm_topk:
        w = w / np.sum(w, axis=-1, keepdims=True)
    return idx, w, p


def softmax(s, axis=-1):
    """Tensor.softmax (Sec. Built-In Libraries, tensor and math primitives),
    with the row maximum subtracted first; -inf entries get weight 0."""
    s = np.asarray(s, dtype=np.float64)
    m = np.max(s, axis=axis, keepdims=True)
    e = np.exp(s - m)
    return e / np.sum(e, axis=axis, keepdims=True)


def attention_one_query(q, K, V, H, G):
    """Grouped-query scaled dot-product attention for one query position
    (Sec. Built-In Libraries, attention and masking; scale from `scale_heads`).
    q: [H, d]; K, V: [T, G, d] holding exactly the visible keys.
    Returns o: [H, d]."""
    q = np.asarray(q, dtype=np.float64)
    d = q.shape[-1]
    o = np.empty_like(q)
    per = H // G
    for h in range(H):
        g = h // per
        s = (K[:, g, :] @ q[h]) / math.sqrt(d)
        o[h] = softmax(s) @ V[:, g, :]
    return o


def causal_attention(q, K, V, q_pos, H, G, window=0):
    """Masking.causal_mask + Attention.attention for S queries of one sequence
    (Sec. Built-In Libraries, attention and masking; the `window=` argument
    of causal_mask_for_input, appendix GPT-2 listing).
    q: [S, H, d] at positions q_pos [S]; K, V: [T, G, d] at positions 0..T-1.
    Key t is visible to query i iff t <= q_pos[i] and, with a window W > 0,
    t > q_pos[i] - W. Returns o: [S, H, d]."""
    q = np.asarray(q, dtype=np.float64)
    S, _, d = q.shape
    T = K.shape[0]
    t = np.arange(T)[None, :]
    p = np.asarray(q_pos)[:, None]
    keep = t <= p  # [S, T]
    if window > 0:
        keep = keep & (t > p - window)
    o = np.empty_like(q)
    per = H // G
    for h in range(H):
        g = h // per
        s = (q[:, h, :] @ K[:, g, :].T) / math.sqrt(d)  # [S, T]
        s = np.where(keep, s, -np.inf)
        o[:, h, :] = softmax(s, axis=-1) @ V[:, g, :]
    return o


def argmax_lowest(logits):
    """Greedy selection in `generate()` (Sec. Results, Measures): the index of
    the largest logit, the lowest such index on ties (np.argmax's rule)."""
    return np.argmax(np.asarray(logits), axis=-1).astype(np.int64)


# ---------------------------------------------------------------------------
# KV caches (Sec. Built-In Libraries: dynamic vs static `Cache` overlays with
# one interface; the paged manager is vLLM's PagedAttention, Sec. Related Work)
# ---------------------------------------------------------------------------

class ContiguousKV:
    """Static-overlay cache: per layer K, V of shape [B, Tmax, G, d], float64."""

    def __init__(self, L, B, Tmax, G, d):
        self.K = [np.zeros((B, Tmax, G, d)) for _ in range(L)]
        self.V = [np.zeros((B, Tmax, G, d)) for _ in range(L)]

    def write(self, l, b, pos, k, v):
        """Cache.update: store k, v [S, G, d] at positions pos [S]."""
        self.K[l][b, pos] = k
        self.V[l][b, pos] = v

    def read(self, l, b, T):
        """Cache.read: keys and values at positions 0 .. T-1."""
        return self.K[l][b, :T], self.V[l][b, :T]


def slot_of(block_table, b, p, block_size):
    """Paged slot of position p of sequence b: (block, offset) with
    block = block_table[b][p // block_size] and offset = p % block_size."""
    return int(block_table[b][p // block_size]), int(p % block_size)


class SeqSlot:
    """One sequence's view of a batched cache: sequence slot `b` of `cache`
    as if it were slot 0 (Cache.update / Cache.read of that sequence)."""

    def __init__(self, cache, b):
        self.cache = cache
        self.b = int(b)

    def write(self, l, b, pos, k, v):
        self.cache.write(l, self.b, pos, k, v)

    def read(self, l, b, T):
        return self.cache.read(l, self.b, T)


class PagedKV:
    """Paged cache: per layer a pool [num_blocks, block_size, G, d] and an
    integer block table [B, max_blocks] naming the pool block of each
    sequence's logical block."""

    def __init__(self, L, num_blocks, block_size, G, d, block_table):
        self.bs = int(block_size)
        self.bt = np.asarray(block_table, dtype=np.int64)
        self.K = [np.zeros((num_blocks, block_size, G, d)) for _ in range(L)]
        self.V = [np.zeros((num_blocks, block_size, G, d)) for _ in range(L)]

    def write(self, l, b, pos, k, v):
        for i, p in enumerate(np.asarray(pos).tolist()):
            blk, off = slot_of(self.bt, b, p, self.bs)
            self.K[l][blk, off] = k[i]
            self.V[l][blk, off] = v[i]

    def read(self, l, b, T):
        pos = np.arange(T)
        blk = self.bt[b][pos // self.bs]
        off = pos % self.bs
        return self.K[l][blk, off], self.V[l][blk, off]


# ---------------------------------------------------------------------------
# The decoder
# ---------------------------------------------------------------------------

class Oracle:
    """Decoder forward over HF-named weights (appendix GPT-2 causal_lm listing
    for the skeleton; Llama naming `model.layers.{i}.self_attn.q_proj.weight`
    as in the `_param(...)` lookups of the Python-overhead appendix).

    weights: name -> array (float32 holding exact bf16 values, or float64),
    or any mapping whose values numpy can widen.
    keep_f64: convert every matrix to float64 once (faster, 8 bytes/param);
    otherwise the mapping is kept as given and each use widens its matrix
    on the fly (for models whose float64 copy would not fit in memory).
    """

    def __init__(self, cfg: DecoderConfig, weights, keep_f64: bool = True):
        self.cfg = cfg
        self.keep_f64 = keep_f64
        if keep_f64:
            self.W = {k: np.asarray(v, dtype=np.float64) for k, v in weights.items()}
        else:
            self.W = weights
        # MoE: per-layer expert choices to use instead of the router's top-k
        # ({layer: [tokens, k]} for the rows of the next forward), and the
        # routing each MoE layer took in the last forward
        self.forced_routing = None
        self.last_routing = {}

    def _w(self, name):
        return self.W[name] if self.keep_f64 else np.asarray(self.W[name], dtype=np.float64)

    def new_contiguous_cache(self, B, Tmax):
        c = self.cfg
        return ContiguousKV(c.L, B, Tmax, c.G, c.d)

    def new_paged_cache(self, num_blocks, block_size, block_table):
        c = self.cfg
        return PagedKV(c.L, num_blocks, block_size, c.G, c.d, block_table)

    def forward(self, ids, cache, past_lens, last_hidden_only=False, rows=None):
        """One pass over new tokens ids [B, S] whose sequence b already holds
        past_lens[b] cached tokens. Writes their K, V into the cache
        (Cache.update / Cache.append) and returns logits [B, S, V]; with
        `rows` (indices into the S new tokens) only those positions go
        through the final norm and LM head: logits [B, len(rows), V]."""
        c = self.cfg
        ids = np.asarray(ids, dtype=np.int64)
        B, S = ids.shape
        past = np.asarray(past_lens, dtype=np.int64).reshape(B)
        pos = past[:, None] + np.arange(S)[None, :]  # Positions.position_ids

        x = self._w("model.embed_tokens.weight")[ids].astype(np.float64)  # NN.embedding
        for l in range(c.L):
            p = f"model.layers.{l}."
            h = rmsnorm(x, self._w(p + "input_layernorm.weight"), c.eps)
            bq = self._w(p + "self_attn.q_proj.bias") if c.bias else None
            bk = self._w(p + "self_attn.k_proj.bias") if c.bias else None
            bv = self._w(p + "self_attn.v_proj.bias") if c.bias else None
            q = linear(h, self._w(p + "self_attn.q_proj.weight"), bq).reshape(B, S, c.H, c.d)
            k = linear(h, self._w(p + "self_attn.k_proj.weight"), bk).reshape(B, S, c.G, c.d)
            v = linear(h, self._w(p + "self_attn.v_proj.weight"), bv).reshape(B, S, c.G, c.d)
            if c.qk_norm:  # NN.rmsnorm over each head's d values, gains q_norm / k_norm
                q = rmsnorm(q, self._w(p + "self_attn.q_norm.weight"), c.eps)
                k = rmsnorm(k, self._w(p + "self_attn.k_norm.weight"), c.eps)
            q = rope(q, pos[:, :, None], c.theta, c.rope_scaling())
            k = rope(k, pos[:, :, None], c.theta, c.rope_scaling())
            o = np.empty((B, S, c.H, c.d))
            for b in range(B):
                cache.write(l, b, pos[b], k[b], v[b])
                Kb, Vb = cache.read(l, b, int(pos[b, -1]) + 1)
                o[b] = causal_attention(q[b], Kb, Vb, pos[b], c.H, c.G, c.window)
            x = x + linear(o.reshape(B, S, c.H * c.d), self._w(p + "self_attn.o_proj.weight"))
            h2 = rmsnorm(x, self._w(p + "post_attention_layernorm.weight"), c.eps)
            if c.is_moe_layer(l):
                forced = None if self.forced_routing is None else self.forced_routing[l]
                x = x + self.moe_mlp(h2.reshape(B * S, c.D), p, forced).reshape(B, S, c.D)
            else:
                u = swiglu(linear(h2, self._w(p + "mlp.gate_proj.weight")),
                           linear(h2, self._w(p + "mlp.up_proj.weight")), c.act)
                x = x + linear(u, self._w(p + "mlp.down_proj.weight"))
        if last_hidden_only:
            x = x[:, -1:, :]
        elif rows is not None:
            x = x[:, np.asarray(rows, dtype=np.int64), :]
        head = self._w("model.embed_tokens.weight") if c.tie else self._w("lm_head.weight")
        return linear(rmsnorm(x, self._w("model.norm.weight"), c.eps), head)

    def moe_mlp(self, h, p, forced=None):
        """Mixture-of-experts MLP of one layer for rows h [T, D]: each token
        goes through its routed experts one at a time (the per-expert loop
        the paper's compiler rewrites into stacked experts), weighted by its
        router weights, plus the shared experts. Records the routing in
        self.last_routing[p]."""
        c = self.cfg
        idx, w, prob = moe_route(h, self._w(p + "mlp.gate.weight"), c.top_k, c.norm_topk, forced)
        self.last_routing[p] = (idx, w, prob)
        y = np.zeros_like(h)
        for t in range(h.shape[0]):
            for j in range(idx.shape[1]):
                e = f"{p}mlp.experts.{int(idx[t, j])}."
                u = swiglu(linear(h[t], self._w(e + "gate_proj.weight")), linear(h[t], self._w(e + "up_proj.weight")),
                           c.act)
                y[t] += w[t, j] * linear(u, self._w(e + "down_proj.weight"))
        if c.n_shared:
            s = p + "mlp.shared_experts."
            u = swiglu(linear(h, self._w(s + "gate_proj.weight")), linear(h, self._w(s + "up_proj.weight")), c.act)
            y = y + linear(u, self._w(s + "down_proj.weight"))
        return y

    def prefill(self, ids, cache, last_only=False, rows=None):
        """Prompt pass from an empty cache; logits for every position, for
        the last one only, or for the positions listed in `rows`."""
        B = np.asarray(ids).shape[0]
        return self.forward(ids, cache, np.zeros(B, dtype=np.int64), last_hidden_only=last_only, rows=rows)

    def decode_step(self, tokens, cache, context_lens):
        """One KV-cached decode step: token b enters at position
        context_lens[b]. Returns logits [B, V]."""
        tokens = np.asarray(tokens, dtype=np.int64).reshape(-1, 1)
        return self.forward(tokens, cache, context_lens)[:, 0, :]

    def forward_varlen(self, chunks, cache, past_lens, last_only=True):
        """Several sequences each append one chunk of new tokens of its own
        length after past_lens[b] cached tokens -- a prompt, a further piece
        of one, or a single decode token (Positions.position_ids with
        past_length; Cache.update): sequence b's chunk runs through forward()
        on that sequence's cache slot. Returns, per sequence, the logits of
        the chunk's last token [V] (last_only) or of all its tokens [S_b, V]."""
        out = []
        for b, ch in enumerate(chunks):
            ids = np.asarray(ch, dtype=np.int64).reshape(1, -1)
            lg = self.forward(ids, SeqSlot(cache, b), [int(past_lens[b])], last_hidden_only=last_only)[0]
            out.append(lg[-1] if last_only else lg)
        return out

    def generate(self, prompt, n_new, cache, forced=None):
        """Greedy generation: prefill, then n_new - 1 decode steps feeding
        back the argmax (or, teacher-forced, the given tokens forced[:, t]).
        Returns (tokens [B, n_new], logits [B, n_new, V])."""
        prompt = np.asarray(prompt, dtype=np.int64)
        B, S = prompt.shape
        logits = [self.prefill(prompt, cache, last_only=True)[:, -1, :]]
        toks = [argmax_lowest(logits[-1])]
        lens = np.full(B, S, dtype=np.int64)
        for t in range(1, n_new):
            feed = toks[-1] if forced is None else np.asarray(forced)[:, t - 1]
            logits.append(self.decode_step(feed, cache, lens))
            toks.append(argmax_lowest(logits[-1]))
            lens = lens + 1
        return np.stack(toks, axis=1), np.stack(logits, axis=1)
