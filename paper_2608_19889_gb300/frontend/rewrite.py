"""Generic graph rewriting (Sec. "The Axon Compiler", Phase 2(b)): loops
that iterate over the experts of a mixture-of-experts MLP become one
stacked-experts operation.

A module states the MoE MLP the way its mathematics reads: a loop over the
E experts that carries an accumulator and adds, for expert e, the expert's
gated MLP of the layer's normalised input scaled by the router weight that
expert e received (zero for the tokens that did not route to it):

    y <- Tensor.zeros_like h
    y <- for@experts e <- [0..E) carry (y) do
      y <- y + MoE.expert_weight w idx e * ffn h     -- ffn: down(act(gate h) * up h)
      yield y

Written that way, every expert would run on every token. The rewrite
recognises the pattern from the operations' provenance -- the loop variable
feeds only the expert-weight selection and the parameter paths, the
accumulator is only added to -- and replaces the loop node by

    MoE.stacked_experts(init, h, w, idx)   attrs: experts E, dim (expert
        width), act, var, gate / up / down path patterns with {var}, fused
        (gate and up as the two halves of one projection under swiglu), and
        the replaced operations' keyword names (kwargs)

whose value is init + sum_e expert_weight(w, idx, e) * ffn_e(h): the
experts' matrices stacked along a leading expert axis, each token computed
by its routed experts only (the grouped expert GEMMs of the kernels). The
replacement keeps the loop node's id, so every use of the loop's value
reads the new node unchanged. Loops of any other shape are left alone.
"""
from __future__ import annotations

from typing import Optional

from . import graph as gr

# gate activations of the gated MLP the kernels implement (op -> kernel name)
ACTIVATIONS = {"Act.silu": "silu", "Activations.silu": "silu", "Act.gelu_tanh": "gelu_tanh",
               "Activations.gelu_new": "gelu_tanh", "Act.gelu_new": "gelu_tanh", "Activations.gelu_tanh": "gelu_tanh"}
# swiglu of one fused projection z of width 2F: silu(z[:F]) * z[F:] (gate
# half first), the MLP idiom `linear@up |> swiglu |> linear@down`
SWIGLU = {"Act.swiglu", "Activations.swiglu"}


def _other(pair, ref):
    """The input of a two-input node that is not `ref` (None if neither is)."""
    a, b = pair
    if a == ref:
        return b
    if b == ref:
        return a
    return None


def _expert_loop(loop: gr.Node) -> Optional[gr.Node]:
    """The stacked-experts node equivalent to `loop`, or None when the loop
    is not a sum over experts."""
    body = loop.body
    if body is None or loop.n_out != 1 or len(body.inputs) != 1 or len(body.outputs) != 1:
        return None
    if loop.attrs.get("start") != 0 or loop.attrs.get("stop", 0) <= 0 or loop.attrs.get("step", 1) != 1:
        return None  # not every expert once
    var = loop.attrs.get("var")
    byid = {n.id: n for n in body.nodes}

    def inner(ref, ops):
        if not isinstance(ref, gr.Ref) or ref.node not in byid:
            return None
        n = byid[ref.node]
        return n if n.op in ops else None

    y_in = body.inputs[0]
    acc = inner(body.outputs[0], {"add"})
    if acc is None or len(acc.inputs) != 2:
        return None
    term_ref = _other(acc.inputs, y_in)
    term = inner(term_ref, {"mul"})
    if term is None:
        return None
    # weight * ffn, in either order
    sel = inner(term.inputs[0], {"MoE.expert_weight"})
    ffn_ref = term.inputs[1]
    if sel is None:
        sel = inner(term.inputs[1], {"MoE.expert_weight"})
        ffn_ref = term.inputs[0]
    if sel is None or len(sel.inputs) != 3:
        return None
    w, idx, e = sel.inputs
    if not (isinstance(e, gr.LoopVar) and e.name == var):
        return None
    if any(isinstance(r, gr.Ref) and r.node in byid for r in (w, idx)):
        return None  # the routing must come from outside the loop
    down = inner(ffn_ref, {"NN.linear"})
    if down is None:
        return None
    sw = inner(down.inputs[0], SWIGLU)
    if sw is not None:  # one fused gate/up projection
        act = prod = sw
        gate = up = inner(sw.inputs[0], {"NN.linear"})
        if gate is None:
            return None
    else:
        prod = inner(down.inputs[0], {"mul"})
        if prod is None:
            return None
        a, b = (inner(r, set(ACTIVATIONS)) for r in prod.inputs)
        act, up_ref = (a, prod.inputs[1]) if a is not None else (b, prod.inputs[0])
        if act is None:
            return None
        gate = inner(act.inputs[0], {"NN.linear"})
        up = inner(up_ref, {"NN.linear"})
        if gate is None or up is None or gate.inputs[0] != up.inputs[0]:
            return None
    h = gate.inputs[0]
    if not isinstance(h, gr.Ref) or h.node in byid:
        return None  # the experts read a value computed before the loop
    token = "{" + str(var) + "}"
    if not all(n.path and token in n.path for n in (gate, up, down)):
        return None  # parameters that do not vary with the expert
    used = {y_in.node, acc.id, term.id, sel.id, down.id, prod.id, act.id, gate.id, up.id}
    if set(byid) != used:
        return None  # anything else in the body: not a plain sum over experts
    fused = sw is not None
    dim = gate.attrs.get("dim")
    if fused:
        dim = dim // 2 if isinstance(dim, int) and dim % 2 == 0 else None
    attrs = {"experts": loop.attrs["stop"], "var": var, "dim": dim, "act": act.op, "fused": fused,
             "gate": gate.path, "up": up.path, "down": down.path, "down_dim": down.attrs.get("dim"),
             "up_dim": dim if fused else up.attrs.get("dim"),
             "bias": any(bool(n.attrs.get("bias")) or bool(n.attrs.get("transpose")) for n in (gate, up, down)),
             # the replaced operations' own keyword arguments, for the backend to vet
             "kwargs": {"NN.linear": sorted(set(gate.attrs) | set(up.attrs) | set(down.attrs)),
                        act.op: sorted(act.attrs), "MoE.expert_weight": sorted(sel.attrs)}}
    return gr.Node(loop.id, "MoE.stacked_experts", [loop.inputs[0], h, w, idx], attrs, None, 1, None)


def stack_experts(g: gr.Graph) -> int:
    """Rewrite, in place and inside loop bodies too, every loop over experts
    of `g` into a MoE.stacked_experts node. Returns how many were replaced;
    a second call finds none."""
    count = 0
    for n in g.nodes:
        if n.body is not None:
            count += stack_experts(n.body)
    for i, n in enumerate(g.nodes):
        if n.op == "loop":
            s = _expert_loop(n)
            if s is not None:
                g.nodes[i] = s
                count += 1
    return count
