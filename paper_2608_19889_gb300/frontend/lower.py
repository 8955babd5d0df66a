"""GB300 backend of the Axon-subset front end: lowering a decoder's Graph
IR onto this library's fused kernels (Sec. "The Axon Compiler", Phase 2(c)
backend-specific rewriting and Phase 3 lowering).

The pattern the kernels implement is the pre-norm decoder layer of the
paper's language section and causal-LM listing:

    h1 = rmsnorm(x);  q, k, v = linear(h1) (+ bias), heads, [per-head rmsnorm],
    rotary positions on q and k, cache update, causal GQA attention,
    merge heads, linear -> a;  x1 = x + a
    h2 = rmsnorm(x1); m = linear_down(act(linear_gate(h2)) * linear_up(h2))
    x2 = x1 + m

inside one ``for`` loop over the layers that carries the hidden state (and
the cache), after an embedding and before a final rmsnorm and LM head
(tied when the head reads the embedding's path).

Mixture-of-experts layers replace m by

    w, idx = softmax_topk_router(h2);  m = stacked_experts(h2, w, idx) [+ shared(h2)]

where the stacked-experts node is what the Phase 2(b) rewrite (rewrite.py)
makes of a loop over the experts, and ``shared`` is a gated MLP (the shared
experts, one MLP whose width is a multiple of an expert's). Such a model is
either one loop of MoE layers or a loop of leading dense layers followed by
a loop of MoE layers that continues the first one's index range and carries
its values (DeepSeek-MoE: the first layer dense). The matcher walks the
loop body backwards from its hidden-state output and claims every node it
recognises; any node left unclaimed, and any operation outside the
supported set, is a LoweringError naming it -- there is no fallback.

The result is the model shape this library's ``make_config`` takes and a
map from the library's checkpoint names (HF Llama naming) to the module's
own parameter paths, so a checkpoint stored under the module's names
loads through ``axon_model_create``.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import Dict, Optional

from . import graph as gr
from .rewrite import ACTIVATIONS as _ACTS, SWIGLU as _SWIGLU, stack_experts

# Operations allowed outside the layer loop and around the cache: they
# carry positions, masks and cache bookkeeping, which the library keeps on
# its own (positions from the context lengths, the causal mask inside the
# attention kernels, the paged or contiguous cache).
_PLUMBING = {
    "Cache.past_length", "Cache.prepare", "Cache.read", "Cache.index", "Cache.append", "Cache.finish",
    "Positions.position_ids", "Masking.causal_mask_for_input", "Masking.causal_mask", "Masking.mask_for_input",
    "Masking.mask_length_for_input", "input",
}
# masks the attention kernels implement: causal, optionally windowed
_CAUSAL_MASKS = ("Masking.causal_mask_for_input", "Masking.causal_mask")
_ROPE_SCALING = ("factor", "low_freq_factor", "high_freq_factor", "original_max_position")
# keyword arguments the kernels implement, per operation; any other keyword
# would change the function and is refused rather than dropped
_KWARGS = {
    "NN.embedding": {"dim"}, "NN.linear": {"dim", "bias", "transpose"}, "NN.rmsnorm": {"eps"},
    "Attention.reshape_heads": {"heads"}, "Attention.merge_heads": set(), "Attention.attention": set(),
    "Positions.rope": {"theta", *_ROPE_SCALING}, "Positions.position_ids": {"past_length"},
    "Masking.causal_mask_for_input": {"window", "padding_mask"}, "Masking.causal_mask": {"window", "padding_mask"},
    "MoE.softmax_topk_router": {"top_k", "normalize", "dim"}, "MoE.expert_weight": set(),
    "Tensor.zeros_like": set(), "add": set(), "mul": set(), "Attention.split_qkv": {"heads", "kv_heads"},
    **{a: set() for a in _ACTS}, **{a: set() for a in _SWIGLU},
}


def _check_kwargs(nodes):
    for n in nodes:
        if n.op == "MoE.stacked_experts":  # the keywords of the operations the rewrite replaced
            for op, keys in n.attrs.get("kwargs", {}).items():
                extra = sorted(set(keys) - _KWARGS.get(op, set()))
                if extra:
                    raise LoweringError(f"{op} in the experts: keyword argument(s) {extra} are not implemented "
                                        "by the kernels")
            continue
        allowed = _KWARGS.get(n.op)
        if allowed is None:
            continue
        extra = sorted(set(n.attrs) - allowed)
        if extra:
            raise LoweringError(f"{n.op}{' @@' + n.path if n.path else ''}: keyword argument(s) {extra} "
                                "are not implemented by the kernels")
# limits of the mixture-of-experts kernels (the config's documented range)
_MAX_EXPERTS, _MAX_TOPK = 256, 8


class LoweringError(ValueError):
    pass


@dataclass
class LoweredDecoder:
    """shape: the model shape for make_config (L, D, H, G, d, F, V, tie,
    bias, theta, eps, window, act, qk_norm, rope scaling; for MoE decoders
    n_experts, top_k, moe_F, n_shared, first_dense, norm_topk); names:
    library checkpoint name -> module parameter path (per layer and expert,
    already instantiated)."""
    shape: dict
    names: Dict[str, str] = field(default_factory=dict)
    # role -> module path pattern ({var} per layer, {e} per expert); the roles
    # of a second (mixture-of-experts) layer loop under "moe_layers."
    paths: Dict[str, str] = field(default_factory=dict)
    # library name -> (first row, end row) of the module tensor it is cut
    # from: q/k/v of a fused projection split by Attention.split_qkv, gate
    # and up of a fused projection under swiglu
    rows: Dict[str, tuple] = field(default_factory=dict)

    def module_weights(self, library_named: dict) -> dict:
        """Re-key a library-named checkpoint under the module's own paths
        (row slices of one module tensor concatenated in row order)."""
        out, parts = {}, {}
        for k, v in library_named.items():
            if k in self.rows:
                parts.setdefault(self.names[k], []).append((self.rows[k][0], v))
            else:
                out[self.names[k]] = v
        for mod, ps in parts.items():
            ts = [t for _, t in sorted(ps, key=lambda x: x[0])]
            out[mod] = _concat_rows(ts)
        return out

    def library_weights(self, module_named: dict) -> dict:
        """Re-key a checkpoint stored under the module's paths to the names
        axon_model_create expects (cutting fused tensors by rows); every
        expected tensor must be present."""
        out = {}
        for lib, mod in self.names.items():
            if mod not in module_named:
                raise LoweringError(f"checkpoint has no tensor {mod!r} (needed as {lib})")
            t = module_named[mod]
            if lib in self.rows:
                a, b = self.rows[lib]
                if t.shape[0] < b:
                    raise LoweringError(f"{mod}: {t.shape[0]} rows, {lib} needs rows {a}..{b}")
                t = t[a:b]
            out[lib] = t
        return out


def _concat_rows(ts):
    if hasattr(ts[0], "detach"):  # torch tensors
        import torch
        return torch.cat(ts, 0)
    import numpy as np
    return np.concatenate(ts, 0)


class _Match:
    def __init__(self, body: gr.Graph, outer: gr.Graph):
        self.body = body
        self.outer = outer
        self.byid = {n.id: n for n in body.nodes}
        self.outer_byid = {n.id: n for n in outer.nodes}
        self.claimed = set()

    def node(self, ref, ops=None, what=""):
        if not isinstance(ref, gr.Ref) or ref.node not in self.byid:
            raise LoweringError(f"{what}: expected a value computed in the layer body")
        n = self.byid[ref.node]
        if ops is not None and n.op not in ops:
            raise LoweringError(f"{what}: expected {sorted(ops)}, found {n.op}"
                                f"{' @@' + n.path if n.path else ''}")
        self.claimed.add(n.id)
        return n

    def through_cache(self, ref, what):
        """k or v as they come out of Cache.update: the value that went in."""
        n = self.node(ref, what=what)
        if n.op == "Cache.update":
            if ref.index not in (0, 1) or len(n.inputs) < 3:
                raise LoweringError(f"{what}: unexpected Cache.update output")
            return n.inputs[1 + ref.index]
        self.claimed.discard(n.id)
        return ref


def _bool(v):
    return bool(v) if v is not None else False


@dataclass
class _Layer:
    """What the body of one layer loop lowered to."""
    loop: gr.Node
    params: dict  # H, G, d, bias, theta, act, qk_norm, rope scaling, window: equal across loops
    eps: set
    paths: dict  # role -> parameter path pattern with the loop's {var}
    mlp: str  # "dense" or "moe"
    F: int = 0  # dense MLP width
    moe: dict = field(default_factory=dict)  # E, top_k, Fe, Fs, norm_topk
    rows: dict = field(default_factory=dict)  # role -> row range of a fused projection


def _gated_mlp(m: _Match, down_ref, what: str):
    """down(act(gate(h)) * up(h)), or down(swiglu(gate_up(h))) with gate and
    up the two halves of one projection: (gate, up, down, activation, h,
    fused)."""
    down = m.node(down_ref, {"NN.linear"}, f"{what} output")
    src = m.byid.get(down.inputs[0].node) if isinstance(down.inputs[0], gr.Ref) else None
    if src is not None and src.op in _SWIGLU:
        sw = m.node(down.inputs[0])
        fused = m.node(sw.inputs[0], {"NN.linear"}, f"{what} fused gate/up projection")
        return fused, fused, down, "silu", fused.inputs[0], True
    mul = m.node(down.inputs[0], {"mul"}, f"{what} product")
    pa, pb = (m.byid.get(r.node) if isinstance(r, gr.Ref) else None for r in mul.inputs)
    if pa is not None and pa.op in _ACTS:
        act_n, up = m.node(mul.inputs[0]), m.node(mul.inputs[1], {"NN.linear"}, f"{what} up projection")
    elif pb is not None and pb.op in _ACTS:
        act_n, up = m.node(mul.inputs[1]), m.node(mul.inputs[0], {"NN.linear"}, f"{what} up projection")
    else:
        raise LoweringError(f"the {what} must multiply an activated gate projection with an up projection")
    gate = m.node(act_n.inputs[0], {"NN.linear"}, f"{what} gate projection")
    if gate.inputs[0] != up.inputs[0]:
        raise LoweringError("gate and up projections must read the same normalised input")
    return gate, up, down, _ACTS[act_n.op], gate.inputs[0], False


def _mlp_width(gate, up, fused, what):
    """Width F of a gated MLP (half the fused projection's width)."""
    F = int(gate.attrs.get("dim", 0) or 0)
    if fused:
        if F <= 0 or F % 2:
            raise LoweringError(f"{what}: the fused gate/up projection's width must be even (two halves)")
        return F // 2
    if int(up.attrs.get("dim", 0) or 0) != F:
        raise LoweringError(f"{what}: gate and up projection widths differ")
    return F


def _moe_mlp(m: _Match, mlp_ref):
    """The MoE pattern at the MLP output, or None when the output is not a
    stacked-experts sum: (stacked node, router node, shared MLP parts or
    None, h)."""
    n = m.byid.get(mlp_ref.node) if isinstance(mlp_ref, gr.Ref) else None
    if n is None:
        return None
    stacked, shared_ref = None, None
    if n.op == "MoE.stacked_experts":
        stacked = n
    elif n.op == "add":
        for a, b in (tuple(n.inputs), tuple(n.inputs[::-1])):
            s = m.byid.get(a.node) if isinstance(a, gr.Ref) else None
            if s is not None and s.op == "MoE.stacked_experts":
                stacked, shared_ref = s, b
                break
        if stacked is None:
            return None
        m.claimed.add(n.id)
    else:
        return None
    m.claimed.add(stacked.id)
    init, h, w, idx = stacked.inputs
    init_n = m.byid.get(init.node) if isinstance(init, gr.Ref) else None
    if init_n is not None and init_n.op == "Tensor.zeros_like":
        m.claimed.add(init_n.id)
    elif shared_ref is None:
        shared_ref = init  # the experts' sum starts from the shared experts' output
    else:
        raise LoweringError("the experts' sum must start from zeros or from the shared experts' output")
    if not (isinstance(w, gr.Ref) and isinstance(idx, gr.Ref) and w.node == idx.node
            and (w.index, idx.index) == (0, 1)):
        raise LoweringError("expert weights and indices must be the two outputs of one MoE.softmax_topk_router")
    router = m.node(w, {"MoE.softmax_topk_router"}, "router")
    if router.inputs[0] != h:
        raise LoweringError("the router and the experts must read the same normalised input")
    shared = None
    if shared_ref is not None:
        shared = _gated_mlp(m, shared_ref, "shared experts")
        if shared[4] != h:
            raise LoweringError("the shared experts must read the routed experts' input")
    return stacked, router, shared, h


def _match_layer(loop: gr.Node, g: gr.Graph, cfg: dict, D: int) -> _Layer:
    """Match one layer loop's body, backwards from its hidden-state output."""
    body = loop.body
    inner = [n for n in body.nodes if n.op == "loop"]
    if inner:
        raise LoweringError(f"a loop over {inner[0].attrs.get('scope') or inner[0].attrs.get('var')} inside the "
                            "layer is not a router-weighted sum over experts (the stacked-experts rewrite does "
                            "not apply), and the kernels run no other loop")
    m = _Match(body, g)
    x_in = body.inputs[0]
    out_x = body.outputs[0]
    add2 = m.node(out_x, {"add"}, "layer output")
    # one operand is x1 = x + a, the other the MLP output
    a0, a1 = add2.inputs
    n0 = m.byid.get(a0.node) if isinstance(a0, gr.Ref) else None
    if n0 is not None and n0.op == "add" and x_in in n0.inputs:
        x1_ref, mlp_ref = a0, a1
    else:
        x1_ref, mlp_ref = a1, a0
    add1 = m.node(x1_ref, {"add"}, "attention residual")
    if x_in not in add1.inputs:
        raise LoweringError("the attention residual must add the layer input (pre-norm block)")
    attn_out = add1.inputs[1] if add1.inputs[0] == x_in else add1.inputs[0]

    # MLP: down(act(gate(h2)) * up(h2)), or the mixture of experts
    moe = _moe_mlp(m, mlp_ref)
    if moe is None:
        gate, up, down, act, h2, mlp_fused = _gated_mlp(m, mlp_ref, "MLP")
    else:
        stacked, router, shared, h2 = moe
        act = "silu" if stacked.attrs.get("fused") else _ACTS.get(stacked.attrs.get("act"))
        if act is None:
            raise LoweringError(f"expert activation {stacked.attrs.get('act')} has no kernel")
        if shared is not None and shared[3] != act:
            raise LoweringError("the shared and the routed experts must use one activation")
    norm2 = m.node(h2, {"NN.rmsnorm"}, "post-attention norm")
    if norm2.inputs[0] != x1_ref:
        raise LoweringError("the post-attention norm must read x + attention")

    # attention: o(merge(attention(q, k, v)))
    o_proj = m.node(attn_out, {"NN.linear"}, "attention output projection")
    merge = m.node(o_proj.inputs[0], {"Attention.merge_heads"}, "merged heads")
    att = m.node(merge.inputs[0], {"Attention.attention"}, "attention")
    q_ref, k_ref, v_ref = att.inputs[0], m.through_cache(att.inputs[1], "keys"), m.through_cache(att.inputs[2],
                                                                                                  "values")
    for r in att.inputs[1:3]:
        n = m.byid.get(r.node) if isinstance(r, gr.Ref) else None
        if n is not None and n.op == "Cache.update":
            m.claimed.add(n.id)
    # the mask: built before the loop from the ids, or in the layer from q
    # and k; the kernels attend causally, so nothing else is accepted
    mask_ref = att.inputs[3] if len(att.inputs) > 3 else None
    mask = None
    if isinstance(mask_ref, gr.Ref):
        mask = m.byid.get(mask_ref.node) or m.outer_byid.get(mask_ref.node)
    if mask is None or mask.op not in _CAUSAL_MASKS:
        raise LoweringError("attention must take a causal mask (Masking.causal_mask_for_input or "
                            "Masking.causal_mask): the kernels attend causally"
                            + (f", found {mask.op}" if mask is not None else ", found none"))
    if mask.attrs.get("padding_mask") is not None:
        raise LoweringError("padding masks: the kernels take per-sequence lengths instead")
    window = int(mask.attrs.get("window", 0) or 0)
    rope_scaling = {}

    heads_ops = {"Attention.reshape_heads", "Attention.split_qkv"}
    splits = []  # the split_qkv node behind q, k and v (fused projection)

    def heads_of(ref, what, index):
        """The projection behind reshape_heads, or behind output `index` of
        split_qkv (q 0, k 1, v 2): (linear, heads)."""
        inner = m.node(ref, heads_ops, f"{what} heads")
        if inner.op == "Attention.split_qkv":
            if ref.index != index:
                raise LoweringError(f"{what}: Attention.split_qkv gives q, k, v in that order")
            splits.append(inner)
            n = int(inner.attrs.get("heads" if index == 0 else "kv_heads", 0) or 0)
        else:
            n = int(inner.attrs.get("heads", 0) or 0)
        return m.node(inner.inputs[0], {"NN.linear"}, f"{what} projection"), n

    def qk_chain(ref, what, index):
        """rope([rmsnorm](heads(linear(h1)))): (linear, heads, norm or None, rope node)."""
        rope = m.node(ref, {"Positions.rope"}, f"{what} rotary positions")
        qn = None
        src = m.byid.get(rope.inputs[0].node) if isinstance(rope.inputs[0], gr.Ref) else None
        inner_ref = rope.inputs[0]
        if src is not None and src.op == "NN.rmsnorm":
            qn = m.node(inner_ref)
            inner_ref = qn.inputs[0]
        lin, n = heads_of(inner_ref, what, index)
        return lin, n, qn, rope

    q_lin, H, q_norm, q_rope = qk_chain(q_ref, "query", 0)
    k_lin, G, k_norm, k_rope = qk_chain(k_ref, "key", 1)
    v_lin, Gv = heads_of(v_ref, "value", 2)
    if Gv != G:
        raise LoweringError("keys and values must have the same number of heads")
    if splits and (len(splits) != 3 or len({n.id for n in splits}) != 1):
        raise LoweringError("q, k and v must all come from one Attention.split_qkv, or none")
    if not (q_lin.inputs[0] == k_lin.inputs[0] == v_lin.inputs[0]):
        raise LoweringError("q, k and v must project the same normalised input")
    norm1 = m.node(q_lin.inputs[0], {"NN.rmsnorm"}, "input norm")
    if norm1.inputs[0] != x_in:
        raise LoweringError("the input norm must read the layer input")
    if (q_norm is None) != (k_norm is None):
        raise LoweringError("qk-norm must apply to both q and k")
    scalings = [tuple((key, r.attrs[key]) for key in _ROPE_SCALING if key in r.attrs) for r in (q_rope, k_rope)]
    if scalings[0] != scalings[1]:
        raise LoweringError("q and k must use one rotary frequency scaling")
    rope_scaling.update(scalings[0])
    thetas = {float(r.attrs.get("theta", cfg.get("rope_theta", 10000.0))) for r in (q_rope, k_rope)}
    if len(thetas) != 1:
        raise LoweringError("q and k must use one rotary base")
    # rotary positions: the new tokens' positions after the cached ones
    for r in (q_rope, k_rope):
        pos = r.inputs[1] if len(r.inputs) > 1 else None
        pn = (m.byid.get(pos.node) or m.outer_byid.get(pos.node)) if isinstance(pos, gr.Ref) else None
        past = pn.attrs.get("past_length") if pn is not None and pn.op == "Positions.position_ids" else None
        pl = (m.byid.get(past.node) or m.outer_byid.get(past.node)) if isinstance(past, gr.Ref) else None
        if pl is None or pl.op != "Cache.past_length":
            raise LoweringError("rotary positions must be Positions.position_ids offset by the cache's past "
                                "length (past_length=Cache.past_length ...): the kernels place token i of a "
                                "sequence at its cached length + i")

    # claimed plumbing inside the body (cache index/append, inputs)
    for n in body.nodes:
        if n.op in _PLUMBING or n.op == "Cache.update":
            m.claimed.add(n.id)
    left = [n for n in body.nodes if n.id not in m.claimed]
    if left:
        raise LoweringError("layer operations with no GB300 kernel: " +
                            ", ".join(f"{n.op}{' @@' + n.path if n.path else ''}" for n in left))
    _check_kwargs(body.nodes)

    biases = {_bool(n.attrs.get("bias")) for n in (q_lin, k_lin, v_lin)}
    if len(biases) != 1:
        raise LoweringError("q, k and v must all have biases or none")
    plain = [o_proj] + ([gate, up, down] if moe is None else [router] + (list(shared[:3]) if shared else []))
    for n in plain:
        if _bool(n.attrs.get("bias")) or _bool(n.attrs.get("transpose")):
            raise LoweringError(f"{n.path}: the kernels take [out, in] matrices without bias here")
    for n in (q_lin, k_lin, v_lin):
        if _bool(n.attrs.get("transpose")):
            raise LoweringError(f"{n.path}: the kernels take [out, in] matrices here")
    rows = {}
    if splits:  # one fused projection [(H + 2G) d, D]: q, k, v rows in that order
        qkv = int(q_lin.attrs.get("dim", 0) or 0)
        if not D or not H or not G or not qkv or qkv % (H + 2 * G):
            raise LoweringError("the fused q/k/v projection's width must be (heads + 2 kv_heads) * head_dim")
        d = qkv // (H + 2 * G)
        rows.update(q=(0, H * d), k=(H * d, (H + G) * d), v=((H + G) * d, (H + 2 * G) * d))
    else:
        qdim = int(q_lin.attrs.get("dim", 0))
        if not D or not qdim or not H or not G or qdim % H:
            raise LoweringError("hidden size, head counts and projection widths must be known")
        d = qdim // H
        if int(k_lin.attrs.get("dim", 0)) != G * d or int(v_lin.attrs.get("dim", 0)) != G * d:
            raise LoweringError("k and v widths must be kv_heads * head_dim")
    if int(o_proj.attrs.get("dim", D)) != D:
        raise LoweringError("MLP and output projection widths disagree with the hidden size")
    params = dict(H=H, G=G, d=d, bias=biases.pop(), theta=thetas.pop(), act=act, qk_norm=q_norm is not None,
                  rope_scaling=tuple(sorted(rope_scaling.items())), window=window)
    norms = (norm1, norm2) + ((q_norm, k_norm) if q_norm is not None else ())
    eps = {float(n.attrs.get("eps", cfg.get("rms_norm_eps", 1e-6))) for n in norms}
    paths = {"input_norm": norm1.path, "post_norm": norm2.path, "q": q_lin.path, "k": k_lin.path,
             "v": v_lin.path, "o": o_proj.path}
    if q_norm is not None:
        paths.update(q_norm=q_norm.path, k_norm=k_norm.path)
    layer = _Layer(loop, params, eps, paths, "dense" if moe is None else "moe")
    layer.rows = rows
    if moe is None:
        F = _mlp_width(gate, up, mlp_fused, "MLP")
        if int(down.attrs.get("dim", 0)) != D:
            raise LoweringError("MLP and output projection widths disagree with the hidden size")
        layer.F = F
        paths.update(gate=gate.path, up=up.path, down=down.path)
        if mlp_fused:
            rows.update(gate=(0, F), up=(F, 2 * F))
    else:
        layer.moe = _moe_params(stacked, router, shared, D)
        paths.update(router=router.path, expert_gate=stacked.attrs["gate"], expert_up=stacked.attrs["up"],
                     expert_down=stacked.attrs["down"])
        Fe, Fs = layer.moe["Fe"], layer.moe["Fs"]
        if stacked.attrs.get("fused"):
            rows.update(expert_gate=(0, Fe), expert_up=(Fe, 2 * Fe))
        if shared is not None:
            paths.update(shared_gate=shared[0].path, shared_up=shared[1].path, shared_down=shared[2].path)
            if shared[5]:
                rows.update(shared_gate=(0, Fs), shared_up=(Fs, 2 * Fs))
    var = "{" + loop.attrs["var"] + "}"
    for role, p in paths.items():
        if not p:
            raise LoweringError(f"{role}: parameterised operation without a path")
        if var not in p:
            raise LoweringError(f"{role}: the layer's parameter path {p!r} does not vary with the layer")
    return layer


def _moe_params(stacked: gr.Node, router: gr.Node, shared, D: int) -> dict:
    """Sizes of a matched MoE MLP, within the kernels' limits."""
    a = stacked.attrs
    if a.get("bias"):
        raise LoweringError("expert projections: the kernels take [out, in] matrices without bias here")
    E, Fe = int(a.get("experts", 0)), int(a.get("dim") or 0)
    if not 1 <= E <= _MAX_EXPERTS:
        raise LoweringError(f"{E} experts: the kernels take 1 to {_MAX_EXPERTS}")
    if Fe <= 0 or int(a.get("up_dim") or 0) != Fe or int(a.get("down_dim") or 0) != D:
        raise LoweringError("expert widths must be known and the down projection must return the hidden size")
    if "{" + str(a.get("var")) + "}" not in str(a.get("gate")):
        raise LoweringError("expert parameters must vary with the expert")
    top_k = router.attrs.get("top_k")
    if not isinstance(top_k, int) or not 1 <= top_k <= min(_MAX_TOPK, E):
        raise LoweringError(f"router top_k {top_k!r}: the kernels take 1 to min({_MAX_TOPK}, experts)")
    if router.attrs.get("dim") not in (None, E):
        raise LoweringError("the router's width must be the number of experts")
    Fs = 0
    if shared is not None:
        Fs = _mlp_width(shared[0], shared[1], shared[5], "shared experts")
        if int(shared[2].attrs.get("dim", 0)) != D:
            raise LoweringError("shared experts' widths disagree with each other or with the hidden size")
        if Fs <= 0 or Fs % Fe:
            raise LoweringError("the shared experts' width must be a multiple of one expert's width")
    return dict(E=E, top_k=top_k, Fe=Fe, Fs=Fs, norm_topk=_bool(router.attrs.get("normalize")),
                evar="{" + str(a["var"]) + "}")


def lower_decoder(g: gr.Graph, config: Optional[dict] = None) -> LoweredDecoder:
    """Match the Graph IR of a causal-LM entry definition onto the fused
    decoder kernels, after the stacked-experts rewrite. `config`: the values
    the module read through Config (for defaults of epsilon and rotary
    base); `g.config_reads` is used when absent."""
    cfg = dict(getattr(g, "config_reads", {}) or {})
    cfg.update(config or {})
    stack_experts(g)
    loops = [n for n in g.nodes if n.op == "loop"]
    if not 1 <= len(loops) <= 2:
        raise LoweringError(f"expected one layer loop (or a dense one, then a mixture-of-experts one), "
                            f"found {len(loops)}")
    if loops[0].attrs["start"] != 0:
        raise LoweringError("the layer loop must start at 0")
    if any(lp.attrs.get("step", 1) != 1 for lp in loops):
        raise LoweringError("a layer loop must advance one layer per iteration (step=1)")
    if len(loops) == 2:
        a, b = loops
        if b.attrs["start"] != a.attrs["stop"]:
            raise LoweringError("the second layer loop must continue the first one's index range")
        if len(b.inputs) != a.n_out or any(not (isinstance(r, gr.Ref) and r.node == a.id and r.index == i)
                                           for i, r in enumerate(b.inputs)):
            raise LoweringError("the second layer loop must carry the values the first one yields")
    last = loops[-1]
    L = last.attrs["stop"]

    # ---- outside the loops: embedding -> loop(s) -> final norm -> head
    outer = {n.id: n for n in g.nodes}
    emb = [n for n in g.nodes if n.op == "NN.embedding"]
    if len(emb) != 1 or not emb[0].path:
        raise LoweringError("expected one NN.embedding with a parameter path")
    emb = emb[0]
    first = loops[0]
    if not first.inputs or not isinstance(first.inputs[0], gr.Ref) or first.inputs[0].node != emb.id:
        raise LoweringError("the layer loop must carry the embedding output as its first value")
    heads_out = [n for n in g.nodes if n.op == "NN.linear"]
    if len(heads_out) != 1:
        raise LoweringError(f"expected one NN.linear (the LM head) outside the layer loop, found {len(heads_out)}")
    head = heads_out[0]
    fnorm = outer.get(head.inputs[0].node) if isinstance(head.inputs[0], gr.Ref) else None
    if fnorm is None or fnorm.op != "NN.rmsnorm" or not fnorm.path:
        raise LoweringError("the LM head must read an NN.rmsnorm of the final hidden state")
    if not (isinstance(fnorm.inputs[0], gr.Ref) and fnorm.inputs[0].node == last.id and fnorm.inputs[0].index == 0):
        raise LoweringError("the final norm must read the layer loop's hidden state")
    if not any(isinstance(o, gr.Ref) and o.node == head.id for o in g.outputs):
        raise LoweringError("the entry definition must return the LM head's logits")
    for n in g.nodes:
        if n.op in ("NN.embedding", "NN.linear", "NN.rmsnorm", "loop"):
            continue
        if n.op not in _PLUMBING:
            raise LoweringError(f"operation {n.op} outside the layer loop has no GB300 kernel")
    _check_kwargs(g.nodes)
    tie = head.path == emb.path
    if head.attrs.get("bias") or head.attrs.get("transpose"):
        raise LoweringError("the LM head takes neither a bias nor a transposed matrix here")

    # ---- the layer bodies
    D = int(emb.attrs.get("dim", 0))
    layers = [_match_layer(lp, g, cfg, D) for lp in loops]
    if len(layers) == 2 and [ly.mlp for ly in layers] != ["dense", "moe"]:
        raise LoweringError("two layer loops must be the leading dense layers, then the mixture-of-experts ones")
    p0 = layers[0].params
    for ly in layers[1:]:
        for key, v in ly.params.items():
            if p0[key] != v:
                raise LoweringError(f"the dense and the mixture-of-experts layers disagree on {key}")
    epss = set().union(*(ly.eps for ly in layers))
    epss.add(float(fnorm.attrs.get("eps", cfg.get("rms_norm_eps", 1e-6))))
    if len(epss) != 1:
        raise LoweringError("every RMSNorm must use one epsilon")
    V = int(head.attrs.get("dim", 0)) or int(cfg.get("vocab_size", 0))
    moe = layers[-1].moe if layers[-1].mlp == "moe" else None
    F = layers[0].F if layers[0].mlp == "dense" else (moe["Fs"] or moe["Fe"])
    shape = dict(L=L, D=D, H=p0["H"], G=p0["G"], d=p0["d"], F=F, V=V, tie=tie, bias=p0["bias"],
                 theta=p0["theta"], eps=epss.pop(), window=p0["window"], act=p0["act"], qk_norm=p0["qk_norm"])
    rope_scaling = dict(p0["rope_scaling"])
    if rope_scaling:
        shape.update(rope_factor=float(rope_scaling.get("factor", 0.0)),
                     rope_low=float(rope_scaling.get("low_freq_factor", 1.0)),
                     rope_high=float(rope_scaling.get("high_freq_factor", 4.0)),
                     rope_orig=int(rope_scaling.get("original_max_position", 8192)))
    if moe is not None:
        shape.update(n_experts=moe["E"], top_k=moe["top_k"], moe_F=moe["Fe"], n_shared=moe["Fs"] // moe["Fe"],
                     first_dense=first.attrs["stop"] if len(layers) == 2 else 0, norm_topk=moe["norm_topk"])

    # ---- library checkpoint name -> module parameter path
    names = {"model.embed_tokens.weight": emb.path + ".weight", "model.norm.weight": fnorm.path + ".weight"}
    if not tie:
        names["lm_head.weight"] = head.path + ".weight"
    attn = [("input_layernorm.weight", "input_norm"), ("post_attention_layernorm.weight", "post_norm"),
            ("self_attn.q_proj.weight", "q"), ("self_attn.k_proj.weight", "k"),
            ("self_attn.v_proj.weight", "v"), ("self_attn.o_proj.weight", "o")]
    if shape["bias"]:
        attn += [("self_attn.q_proj.bias", "q"), ("self_attn.k_proj.bias", "k"), ("self_attn.v_proj.bias", "v")]
    if shape["qk_norm"]:
        attn += [("self_attn.q_norm.weight", "q_norm"), ("self_attn.k_norm.weight", "k_norm")]
    dense = [("mlp.gate_proj.weight", "gate"), ("mlp.up_proj.weight", "up"), ("mlp.down_proj.weight", "down")]
    shared = [("mlp.shared_experts.gate_proj.weight", "shared_gate"), ("mlp.shared_experts.up_proj.weight", "shared_up"),
              ("mlp.shared_experts.down_proj.weight", "shared_down")]
    expert = [("gate_proj.weight", "expert_gate"), ("up_proj.weight", "expert_up"), ("down_proj.weight", "expert_down")]
    paths = {"embed": emb.path, "final_norm": fnorm.path, "head": head.path}
    rows = {}
    for k, ly in enumerate(layers):
        var = "{" + ly.loop.attrs["var"] + "}"
        per_layer = attn + (dense if ly.mlp == "dense" else [("mlp.gate.weight", "router")] +
                            (shared if ly.moe["Fs"] else []))
        paths.update({(role if k == 0 else f"moe_layers.{role}"): p for role, p in ly.paths.items()})
        for l in range(ly.loop.attrs["start"], ly.loop.attrs["stop"]):
            for lib, role in per_layer:
                leaf = lib.rsplit(".", 1)[1]
                name = f"model.layers.{l}.{lib}"
                names[name] = ly.paths[role].replace(var, str(l)) + "." + leaf
                if role in ly.rows:
                    rows[name] = ly.rows[role]
            if ly.mlp == "moe":
                evar = ly.moe["evar"]
                for e in range(ly.moe["E"]):
                    for lib, role in expert:
                        name = f"model.layers.{l}.mlp.experts.{e}.{lib}"
                        names[name] = ly.paths[role].replace(var, str(l)).replace(evar, str(e)) + ".weight"
                        if role in ly.rows:
                            rows[name] = ly.rows[role]
    return LoweredDecoder(shape, names, paths, rows)
