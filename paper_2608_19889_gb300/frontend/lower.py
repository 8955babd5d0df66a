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
(tied when the head reads the embedding's path). The matcher walks the
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
from typing import Dict, List, Optional

from . import graph as gr

# Operations allowed outside the layer loop and around the cache: they
# carry positions, masks and cache bookkeeping, which the library keeps on
# its own (positions from the context lengths, the causal mask inside the
# attention kernels, the paged or contiguous cache).
_PLUMBING = {
    "Cache.past_length", "Cache.prepare", "Cache.read", "Cache.index", "Cache.append", "Cache.finish",
    "Positions.position_ids", "Masking.causal_mask_for_input", "Masking.mask_for_input",
    "Masking.mask_length_for_input", "input",
}
_ACTS = {"Act.silu": "silu", "Activations.silu": "silu", "Act.gelu_tanh": "gelu_tanh",
         "Activations.gelu_new": "gelu_tanh", "Act.gelu_new": "gelu_tanh", "Activations.gelu_tanh": "gelu_tanh"}


class LoweringError(ValueError):
    pass


@dataclass
class LoweredDecoder:
    """shape: the model shape for make_config (L, D, H, G, d, F, V, tie,
    bias, theta, eps, window, act, qk_norm, rope scaling); names: library
    checkpoint name -> module parameter path (per layer, already
    instantiated)."""
    shape: dict
    names: Dict[str, str] = field(default_factory=dict)
    paths: Dict[str, str] = field(default_factory=dict)  # role -> module path pattern ({i} per layer)

    def module_weights(self, library_named: dict) -> dict:
        """Re-key a library-named checkpoint under the module's own paths."""
        return {self.names[k]: v for k, v in library_named.items()}

    def library_weights(self, module_named: dict) -> dict:
        """Re-key a checkpoint stored under the module's paths to the names
        axon_model_create expects; every expected tensor must be present."""
        out = {}
        for lib, mod in self.names.items():
            if mod not in module_named:
                raise LoweringError(f"checkpoint has no tensor {mod!r} (needed as {lib})")
            out[lib] = module_named[mod]
        return out


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


def lower_decoder(g: gr.Graph, config: Optional[dict] = None) -> LoweredDecoder:
    """Match the Graph IR of a causal-LM entry definition onto the fused
    decoder kernels. `config`: the values the module read through Config
    (for defaults of epsilon and rotary base); `g.config_reads` is used when
    absent."""
    cfg = dict(getattr(g, "config_reads", {}) or {})
    cfg.update(config or {})
    loops = [n for n in g.nodes if n.op == "loop"]
    if len(loops) != 1:
        raise LoweringError(f"expected one layer loop, found {len(loops)}")
    loop = loops[0]
    body = loop.body
    L = loop.attrs["stop"] - loop.attrs["start"]
    if loop.attrs["start"] != 0:
        raise LoweringError("the layer loop must start at 0")

    # ---- outside the loop: embedding -> loop -> final norm -> head
    outer = {n.id: n for n in g.nodes}
    emb = [n for n in g.nodes if n.op == "NN.embedding"]
    if len(emb) != 1 or not emb[0].path:
        raise LoweringError("expected one NN.embedding with a parameter path")
    emb = emb[0]
    if not loop.inputs or not isinstance(loop.inputs[0], gr.Ref) or loop.inputs[0].node != emb.id:
        raise LoweringError("the layer loop must carry the embedding output as its first value")
    heads_out = [n for n in g.nodes if n.op == "NN.linear"]
    if len(heads_out) != 1:
        raise LoweringError(f"expected one NN.linear (the LM head) outside the layer loop, found {len(heads_out)}")
    head = heads_out[0]
    fnorm = outer.get(head.inputs[0].node) if isinstance(head.inputs[0], gr.Ref) else None
    if fnorm is None or fnorm.op != "NN.rmsnorm" or not fnorm.path:
        raise LoweringError("the LM head must read an NN.rmsnorm of the final hidden state")
    if not (isinstance(fnorm.inputs[0], gr.Ref) and fnorm.inputs[0].node == loop.id and fnorm.inputs[0].index == 0):
        raise LoweringError("the final norm must read the layer loop's hidden state")
    if not any(isinstance(o, gr.Ref) and o.node == head.id for o in g.outputs):
        raise LoweringError("the entry definition must return the LM head's logits")
    window = 0
    for n in g.nodes:
        if n.op in ("NN.embedding", "NN.linear", "NN.rmsnorm", "loop"):
            continue
        if n.op not in _PLUMBING:
            raise LoweringError(f"operation {n.op} outside the layer loop has no GB300 kernel")
        if n.op == "Masking.causal_mask_for_input":
            window = int(n.attrs.get("window", 0) or 0)
    tie = head.path == emb.path
    if head.attrs.get("bias") or head.attrs.get("transpose"):
        raise LoweringError("the LM head takes neither a bias nor a transposed matrix here")

    # ---- the layer body, backwards from the hidden-state output
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

    # MLP: down(act(gate(h2)) * up(h2))
    down = m.node(mlp_ref, {"NN.linear"}, "MLP output")
    mul = m.node(down.inputs[0], {"mul"}, "MLP product")
    pa, pb = (m.byid.get(r.node) if isinstance(r, gr.Ref) else None for r in mul.inputs)
    if pa is not None and pa.op in _ACTS:
        act_n, up = m.node(mul.inputs[0]), m.node(mul.inputs[1], {"NN.linear"}, "MLP up projection")
    elif pb is not None and pb.op in _ACTS:
        act_n, up = m.node(mul.inputs[1]), m.node(mul.inputs[0], {"NN.linear"}, "MLP up projection")
    else:
        raise LoweringError("the MLP must multiply an activated gate projection with an up projection")
    act = _ACTS[act_n.op]
    gate = m.node(act_n.inputs[0], {"NN.linear"}, "MLP gate projection")
    if gate.inputs[0] != up.inputs[0]:
        raise LoweringError("gate and up projections must read the same normalised input")
    norm2 = m.node(gate.inputs[0], {"NN.rmsnorm"}, "post-attention norm")
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
    rope_scaling = {}

    def qk_chain(ref, what):
        """rope([rmsnorm](reshape_heads(linear(h1)))): (linear, heads, norm or None, rope node)."""
        rope = m.node(ref, {"Positions.rope"}, f"{what} rotary positions")
        inner = m.node(rope.inputs[0], {"Attention.reshape_heads", "NN.rmsnorm"}, f"{what} heads")
        qn = None
        if inner.op == "NN.rmsnorm":
            qn = inner
            inner = m.node(inner.inputs[0], {"Attention.reshape_heads"}, f"{what} heads")
        lin = m.node(inner.inputs[0], {"NN.linear"}, f"{what} projection")
        return lin, int(inner.attrs.get("heads", 0)), qn, rope

    q_lin, H, q_norm, q_rope = qk_chain(q_ref, "query")
    k_lin, G, k_norm, k_rope = qk_chain(k_ref, "key")
    v_heads = m.node(v_ref, {"Attention.reshape_heads"}, "value heads")
    v_lin = m.node(v_heads.inputs[0], {"NN.linear"}, "value projection")
    if int(v_heads.attrs.get("heads", 0)) != G:
        raise LoweringError("keys and values must have the same number of heads")
    if not (q_lin.inputs[0] == k_lin.inputs[0] == v_lin.inputs[0]):
        raise LoweringError("q, k and v must project the same normalised input")
    norm1 = m.node(q_lin.inputs[0], {"NN.rmsnorm"}, "input norm")
    if norm1.inputs[0] != x_in:
        raise LoweringError("the input norm must read the layer input")
    if (q_norm is None) != (k_norm is None):
        raise LoweringError("qk-norm must apply to both q and k")
    for r in (q_rope, k_rope):
        for key in ("factor", "low_freq_factor", "high_freq_factor", "original_max_position"):
            if key in r.attrs:
                rope_scaling[key] = r.attrs[key]
    thetas = {float(r.attrs.get("theta", cfg.get("rope_theta", 10000.0))) for r in (q_rope, k_rope)}
    if len(thetas) != 1:
        raise LoweringError("q and k must use one rotary base")

    # claimed plumbing inside the body (cache index/append, inputs)
    for n in body.nodes:
        if n.op in _PLUMBING or n.op == "Cache.update":
            m.claimed.add(n.id)
    left = [n for n in body.nodes if n.id not in m.claimed]
    if left:
        raise LoweringError("layer operations with no GB300 kernel: " +
                            ", ".join(f"{n.op}{' @@' + n.path if n.path else ''}" for n in left))

    biases = {_bool(n.attrs.get("bias")) for n in (q_lin, k_lin, v_lin)}
    if len(biases) != 1:
        raise LoweringError("q, k and v must all have biases or none")
    for n in (o_proj, gate, up, down):
        if _bool(n.attrs.get("bias")) or _bool(n.attrs.get("transpose")):
            raise LoweringError(f"{n.path}: the kernels take [out, in] matrices without bias here")
    for n in (q_lin, k_lin, v_lin):
        if _bool(n.attrs.get("transpose")):
            raise LoweringError(f"{n.path}: the kernels take [out, in] matrices here")
    D = int(emb.attrs.get("dim", 0))
    qdim = int(q_lin.attrs.get("dim", 0))
    if not D or not qdim or not H or not G or qdim % H:
        raise LoweringError("hidden size, head counts and projection widths must be known")
    d = qdim // H
    F = int(gate.attrs.get("dim", 0))
    V = int(head.attrs.get("dim", 0)) or int(cfg.get("vocab_size", 0))
    if int(k_lin.attrs.get("dim", 0)) != G * d or int(v_lin.attrs.get("dim", 0)) != G * d:
        raise LoweringError("k and v widths must be kv_heads * head_dim")
    if int(up.attrs.get("dim", 0)) != F or int(down.attrs.get("dim", 0)) != D or int(o_proj.attrs.get("dim", D)) != D:
        raise LoweringError("MLP and output projection widths disagree with the hidden size")
    epss = {float(n.attrs.get("eps", cfg.get("rms_norm_eps", 1e-6))) for n in (norm1, norm2, fnorm)}
    if len(epss) != 1:
        raise LoweringError("every RMSNorm must use one epsilon")
    shape = dict(L=L, D=D, H=H, G=G, d=d, F=F, V=V, tie=tie, bias=biases.pop(), theta=thetas.pop(),
                 eps=epss.pop(), window=window, act=act, qk_norm=q_norm is not None)
    if rope_scaling:
        shape.update(rope_factor=float(rope_scaling.get("factor", 0.0)),
                     rope_low=float(rope_scaling.get("low_freq_factor", 1.0)),
                     rope_high=float(rope_scaling.get("high_freq_factor", 4.0)),
                     rope_orig=int(rope_scaling.get("original_max_position", 8192)))

    paths = {"embed": emb.path, "final_norm": fnorm.path, "head": head.path, "input_norm": norm1.path,
             "post_norm": norm2.path, "q": q_lin.path, "k": k_lin.path, "v": v_lin.path, "o": o_proj.path,
             "gate": gate.path, "up": up.path, "down": down.path}
    if q_norm is not None:
        paths.update(q_norm=q_norm.path, k_norm=k_norm.path)
    for role, p in paths.items():
        if not p:
            raise LoweringError(f"{role}: parameterised operation without a path")
    var = "{" + loop.attrs["var"] + "}"
    names = {"model.embed_tokens.weight": emb.path + ".weight", "model.norm.weight": fnorm.path + ".weight"}
    if not tie:
        names["lm_head.weight"] = head.path + ".weight"
    per_layer = [("input_layernorm.weight", "input_norm", "weight"),
                 ("post_attention_layernorm.weight", "post_norm", "weight"),
                 ("self_attn.q_proj.weight", "q", "weight"), ("self_attn.k_proj.weight", "k", "weight"),
                 ("self_attn.v_proj.weight", "v", "weight"), ("self_attn.o_proj.weight", "o", "weight"),
                 ("mlp.gate_proj.weight", "gate", "weight"), ("mlp.up_proj.weight", "up", "weight"),
                 ("mlp.down_proj.weight", "down", "weight")]
    if shape["bias"]:
        per_layer += [("self_attn.q_proj.bias", "q", "bias"), ("self_attn.k_proj.bias", "k", "bias"),
                      ("self_attn.v_proj.bias", "v", "bias")]
    if shape["qk_norm"]:
        per_layer += [("self_attn.q_norm.weight", "q_norm", "weight"), ("self_attn.k_norm.weight", "k_norm", "weight")]
    for role in ("input_norm", "post_norm", "q", "k", "v", "o", "gate", "up", "down"):
        if var not in paths[role]:
            raise LoweringError(f"{role}: the layer's parameter path {paths[role]!r} does not vary with the layer")
    for l in range(L):
        for lib, role, leaf in per_layer:
            names[f"model.layers.{l}.{lib}"] = paths[role].replace(var, str(l)) + "." + leaf
    return LoweredDecoder(shape, names, paths)
