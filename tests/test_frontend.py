"""CPU tests of the Axon-subset front end: lexing and parsing, Graph IR
building (definition inlining, scoped parameter paths, loops, configuration
reads), the stacked-experts rewrite, and the lowering of decoder modules
onto the library's kernels (shape and checkpoint-name map), including the
variants it accepts and the modules it must refuse. The lowering is also
checked for meaning: a module's Graph IR, evaluated directly on its own
parameter paths (graph_eval.py), gives the oracle's logits for the lowered
shape on the checkpoint re-keyed through the name map."""
import os
import re

import numpy as np
import pytest

import synth_inputs as si
from graph_eval import GraphEval
from helpers import oracle_for
from paper_2608_19889_gb300 import frontend as fe
from paper_2608_19889_gb300.frontend import rewrite as rw
from paper_2608_19889_gb300.frontend import syntax as sx

HERE = os.path.dirname(os.path.abspath(__file__))
LLAMA = open(os.path.join(HERE, "data", "llama_decoder.axon")).read()
MOE = open(os.path.join(HERE, "data", "moe_decoder.axon")).read()
CFG = dict(hidden_size=128, num_hidden_layers=2, num_attention_heads=4, num_key_value_heads=2, head_dim=32,
           intermediate_size=192, vocab_size=1000, rope_theta=10000.0, rms_norm_eps=1e-5)
# DeepSeek-MoE-like at toy width: layer 0 dense, layers 1-2 with 6 experts
# (2 per token) of width 16 and a shared MLP of 2 experts' width
MOE_CFG = dict(hidden_size=32, num_hidden_layers=3, first_k_dense_replace=1, num_attention_heads=4,
               num_key_value_heads=2, head_dim=8, intermediate_size=48, n_routed_experts=6, num_experts_per_tok=2,
               moe_intermediate_size=16, n_shared_experts=2, vocab_size=64, rope_theta=10000.0, rms_norm_eps=1e-5)


# ------------------------------------------------------------------ syntax
def test_layout_tokens_and_comments():
    toks = sx.tokenize("f x = do\n  y <- g x -- note\n  return y\nh = 1\n")
    kinds = [t.kind for t in toks]
    assert kinds.count("INDENT") == 1 and kinds.count("DEDENT") == 1
    assert "note" not in [t.text for t in toks]
    paths = [t.text for t in sx.tokenize("a <- NN.rmsnorm@ln x\nb <- @@model.embed_tokens\n") if t.kind == "PATH"]
    assert paths == ["@ln", "@@model.embed_tokens"]


def test_pipe_is_application_with_the_left_value_first():
    mod = sx.parse_module("f x = x |> g a k=2 |> h\n")
    e = mod.definitions["f"].body
    assert isinstance(e, sx.Call) and e.fn.name == "h"
    inner = e.args[0]
    assert inner.fn.name == "g" and isinstance(inner.args[0], sx.Name) and inner.args[0].name == "x"
    assert inner.args[1].name == "a" and inner.kwargs["k"].value == 2


def test_precedence_application_over_arithmetic_over_pipe():
    mod = sx.parse_module("f g u = Act.silu g * u |> NN.linear@down dim=4\n")
    e = mod.definitions["f"].body
    assert e.fn.name == "NN.linear" and e.fn.path == "down"
    mul = e.args[0]
    assert isinstance(mul, sx.BinOp) and mul.op == "*"
    assert isinstance(mul.left, sx.Call) and mul.left.fn.name == "Act.silu"


def test_statements_loops_scopes_and_ascription():
    src = ("n <- (Config.dim @@n default=3 :: Dim)\n"
           "f x = do\n"
           "  a, b <- scope@attn do\n"
           "    q <- NN.linear@q x\n"
           "    return q, q\n"
           "  y <- for@h i <- [0..n) carry (a) do\n"
           "    a <- a + b\n"
           "    yield a\n"
           "  return y\n")
    mod = sx.parse_module(src)
    name, c = mod.constants[0]
    assert name == "n" and isinstance(c, sx.Ascribe) and c.type_text == "Dim"
    body = mod.definitions["f"].body.body
    assert body[0].targets == ["a", "b"] and isinstance(body[0].expr, sx.ScopeE)
    loop = body[1].expr
    assert isinstance(loop, sx.ForE) and loop.scope == "h" and loop.carry == ["a"]
    assert loop.lo_closed and not loop.hi_closed


@pytest.mark.parametrize("bad", ["f x = (x\n", "f x = do\n  y <-\n", "f x = x |> 3\n", "f = @\n"])
def test_syntax_errors_are_reported(bad):
    with pytest.raises(fe.AxonSyntaxError):
        sx.parse_module(bad)


# ------------------------------------------------------------------- graph
def test_paths_resolve_through_scopes_definitions_and_absolute_paths():
    src = ("import NN\n"
           "proj@tok x = NN.linear@q x dim=4\n"
           "f x = do\n"
           "  a <- proj x\n"
           "  b <- proj@other x\n"
           "  c <- scope@outer do\n"
           "    return NN.rmsnorm@ln x\n"
           "  d <- NN.rmsnorm@@abs.norm x\n"
           "  return a + b + c + d\n")
    g = fe.build_graph(sx.parse_module(src), entry="f")
    paths = [n.path for n in g.nodes if n.path]
    assert paths == ["tok.q", "other.q", "outer.ln", "abs.norm"]


def test_loop_body_is_built_once_with_a_symbolic_layer_index():
    g = fe.build_graph(sx.parse_module(LLAMA), CFG)
    loops = [n for n in g.nodes if n.op == "loop"]
    assert len(loops) == 1 and loops[0].attrs["stop"] == 2
    body_paths = {n.path for n in loops[0].body.nodes if n.path}
    assert "layers.{i}.attention.wq" in body_paths and "layers.{i}.feed_forward.w2" in body_paths
    assert all("{i}" in p for p in body_paths)


def test_config_reads_use_values_then_defaults_and_fold_constants():
    src = "import NN\nD <- (Config.dim @@hidden default=8 :: Dim)\nf x = NN.linear@p x dim=(2 * D + 1)\n"
    g = fe.build_graph(sx.parse_module(src), {"hidden": 16}, entry="f")
    assert [n.attrs["dim"] for n in g.nodes if n.op == "NN.linear"] == [33]
    g2 = fe.build_graph(sx.parse_module(src), {}, entry="f")
    assert [n.attrs["dim"] for n in g2.nodes if n.op == "NN.linear"] == [17]
    with pytest.raises(fe.AxonGraphError):
        fe.build_graph(sx.parse_module("D <- Config.dim @@missing\nf x = x\n"), {}, entry="f")


def test_unknown_functions_and_bad_binds_are_errors():
    with pytest.raises(fe.AxonGraphError, match="unknown function"):
        fe.build_graph(sx.parse_module("f x = frobnicate x\n"), entry="f")
    with pytest.raises(fe.AxonGraphError, match="targets"):
        fe.build_graph(sx.parse_module("import NN\nf x = do\n  a, b <- (x, x, x)\n  return a\n"), entry="f")


# ---------------------------------------------------------------- lowering
def test_llama_module_lowers_to_the_kernels_shape_and_names():
    low = fe.compile_decoder(LLAMA, CFG)
    assert low.shape == dict(L=2, D=128, H=4, G=2, d=32, F=192, V=1000, tie=False, bias=False, theta=10000.0,
                             eps=1e-5, window=0, act="silu", qk_norm=False)
    want = {"model.embed_tokens.weight": "tok_embeddings.weight", "model.norm.weight": "norm.weight",
            "lm_head.weight": "output.weight"}
    for l in range(2):
        p = f"model.layers.{l}."
        want.update({p + "input_layernorm.weight": f"layers.{l}.attention_norm.weight",
                     p + "post_attention_layernorm.weight": f"layers.{l}.ffn_norm.weight",
                     p + "self_attn.q_proj.weight": f"layers.{l}.attention.wq.weight",
                     p + "self_attn.k_proj.weight": f"layers.{l}.attention.wk.weight",
                     p + "self_attn.v_proj.weight": f"layers.{l}.attention.wv.weight",
                     p + "self_attn.o_proj.weight": f"layers.{l}.attention.wo.weight",
                     p + "mlp.gate_proj.weight": f"layers.{l}.feed_forward.w1.weight",
                     p + "mlp.up_proj.weight": f"layers.{l}.feed_forward.w3.weight",
                     p + "mlp.down_proj.weight": f"layers.{l}.feed_forward.w2.weight"})
    assert low.names == want


def _variant(old, new, count=1):
    assert LLAMA.count(old) >= count, old
    return LLAMA.replace(old, new)


def test_variants_bias_qk_norm_gelu_tied_window_and_rope_scaling():
    src = LLAMA
    for proj in ("wq", "wk", "wv"):
        src = re.sub(rf"(NN\.linear@{proj} h dim=\([A-Z_]+ \* HEAD_DIM\))", r"\1 bias=true", src)
    src = src.replace("  q <- rope q pos theta=THETA",
                      "  q <- NN.rmsnorm@q_norm q eps=EPS\n  q <- rope q pos theta=THETA factor=8.0 "
                      "low_freq_factor=1.0 high_freq_factor=4.0 original_max_position=8192")
    src = src.replace("  k <- rope k pos theta=THETA",
                      "  k <- NN.rmsnorm@k_norm k eps=EPS\n  k <- rope k pos theta=THETA factor=8.0 "
                      "low_freq_factor=1.0 high_freq_factor=4.0 original_max_position=8192")
    src = src.replace("Act.silu g", "Act.gelu_tanh g").replace("NN.linear@output dim=VOCAB",
                                                              "NN.linear@tok_embeddings dim=VOCAB")
    low = fe.compile_decoder(src, dict(CFG, sliding_window=64))
    s = low.shape
    assert s["bias"] and s["qk_norm"] and s["act"] == "gelu_tanh" and s["tie"] and s["window"] == 64
    assert (s["rope_factor"], s["rope_low"], s["rope_high"], s["rope_orig"]) == (8.0, 1.0, 4.0, 8192)
    assert "lm_head.weight" not in low.names
    assert low.names["model.layers.1.self_attn.k_proj.bias"] == "layers.1.attention.wk.bias"
    assert low.names["model.layers.0.self_attn.q_norm.weight"] == "layers.0.attention.q_norm.weight"


@pytest.mark.parametrize("old,new,msg", [
    ("NN.rmsnorm@attention_norm x", "NN.layernorm@attention_norm x", "input norm"),
    ("NN.linear@wq h dim=(HEADS * HEAD_DIM)", "NN.linear@wq h dim=(HEADS * HEAD_DIM) bias=true", "biases"),
    ("  q <- rope q pos theta=THETA", "  q <- NN.rmsnorm@q_norm q eps=EPS\n  q <- rope q pos theta=THETA",
     "qk-norm"),
    ("Act.silu g * u", "Act.relu g * u", "activated gate"),
    ("  return x + m, new_kv", "  m <- Tensor.dropout m\n  return x + m, new_kv", "MLP output"),
    ("  x <- x + a\n  m <- NN.rmsnorm@ffn_norm x eps=EPS |> ffn@feed_forward",
     "  m <- NN.rmsnorm@ffn_norm x eps=EPS |> ffn@feed_forward\n  x <- x + a", "post-attention norm"),
    ("  past_len <- Cache.past_length past", "  past_len <- Cache.past_length past\n  z <- Tensor.noise ids",
     "outside the layer loop"),
    # no mask (bidirectional attention) or a non-causal one: the kernels attend causally
    ("attention q k v mask |>", "attention q k v |>", "causal mask"),
    ("  mask <- causal_mask_for_input ids past_len window=WINDOW",
     "  mask <- Masking.mask_for_input ids past_len", "causal mask"),
    ("attention q k v mask |>", "attention q k v (Masking.causal_mask q k padding_mask=pos) |>", "padding"),
    # positions that restart at 0 on every decode step
    ("  pos <- position_ids ids past_length=past_len", "  pos <- position_ids ids", "rotary positions"),
    ("  k <- rope k pos theta=THETA", "  k <- rope k pos theta=THETA factor=8.0", "frequency scaling"),
    # keywords that would change the function
    ("NN.rmsnorm@attention_norm x eps=EPS", "NN.rmsnorm@attention_norm x eps=EPS offset=1.0", "offset"),
    ("attention q k v mask |>", "attention q k v mask scale=0.5 |>", "scale"),
    # qk-norm with its own epsilon: the kernels use one rms_norm_eps
    ("  q <- rope q pos theta=THETA", "  q <- NN.rmsnorm@q_norm q eps=0.5\n  q <- rope q pos theta=THETA\n"
     "  k <- NN.rmsnorm@k_norm k eps=0.5", "epsilon"),
])
def test_modules_outside_the_kernels_are_refused(old, new, msg):
    with pytest.raises(fe.LoweringError, match=msg):
        fe.compile_decoder(_variant(old, new), CFG)


def test_checkpoint_renaming_both_ways_and_missing_tensors():
    low = fe.compile_decoder(LLAMA, CFG)
    lib = {k: i for i, k in enumerate(low.names)}
    mod = low.module_weights(lib)
    assert set(mod) == set(low.names.values())
    assert low.library_weights(mod) == lib
    mod.pop("layers.1.feed_forward.w3.weight")
    with pytest.raises(fe.LoweringError, match="w3"):
        low.library_weights(mod)


# ------------------------------------------------------ mixture of experts
def _moe_body(g):
    """The body graph of the mixture-of-experts layer loop."""
    return [n for n in g.nodes if n.op == "loop"][-1].body


def test_stacked_experts_rewrite_replaces_the_loop_over_experts():
    g = fe.build_graph(sx.parse_module(MOE), MOE_CFG)
    inner = [n for n in _moe_body(g).nodes if n.op == "loop"]
    assert len(inner) == 1 and inner[0].attrs["var"] == "e" and inner[0].attrs["stop"] == 6
    loop_id = inner[0].id
    assert rw.stack_experts(g) == 1
    assert rw.stack_experts(g) == 0  # nothing left to rewrite
    body = _moe_body(g)
    assert not [n for n in body.nodes if n.op == "loop"]
    st = [n for n in body.nodes if n.op == "MoE.stacked_experts"]
    assert len(st) == 1 and st[0].id == loop_id  # uses of the loop's value now read the stacked node
    a = st[0].attrs
    assert (a["experts"], a["dim"], a["act"], a["var"]) == (6, 16, "Act.silu", "e")
    assert (a["gate"], a["up"], a["down"]) == tuple(f"blocks.{{i}}.ffn.experts.{{e}}.{w}"
                                                     for w in ("w_gate", "w_up", "w_down"))
    router = [n for n in body.nodes if n.op == "MoE.softmax_topk_router"][0]
    init, h, w, idx = st[0].inputs
    assert (w, idx) == (fe.Ref(router.id, 0), fe.Ref(router.id, 1)) and router.inputs[0] == h


def test_dense_loops_are_not_rewritten():
    g = fe.build_graph(sx.parse_module(LLAMA), CFG)
    before = fe.dump(g)
    assert rw.stack_experts(g) == 0 and fe.dump(g) == before


def test_moe_module_lowers_to_the_kernels_shape_and_names():
    low = fe.compile_decoder(MOE, MOE_CFG)
    assert low.shape == dict(L=3, D=32, H=4, G=2, d=8, F=48, V=64, tie=False, bias=False, theta=10000.0, eps=1e-5,
                             window=0, act="silu", qk_norm=False, n_experts=6, top_k=2, moe_F=16, n_shared=2,
                             first_dense=1, norm_topk=False)
    # exactly the tensors the library reads for that shape, each from its module path
    assert set(low.names) == set(si.weight_shapes(low.shape))
    assert low.names["model.layers.0.mlp.down_proj.weight"] == "blocks.0.ffn.w_down.weight"
    assert low.names["model.layers.2.mlp.gate.weight"] == "blocks.2.ffn.router.weight"
    assert low.names["model.layers.1.mlp.experts.5.up_proj.weight"] == "blocks.1.ffn.experts.5.w_up.weight"
    assert low.names["model.layers.2.mlp.shared_experts.down_proj.weight"] == "blocks.2.ffn.shared.w_down.weight"
    assert low.paths["moe_layers.expert_gate"] == "blocks.{i}.ffn.experts.{e}.w_gate"


def test_llama_module_names_are_the_librarys_tensors():
    low = fe.compile_decoder(LLAMA, CFG)
    assert set(low.names) == set(si.weight_shapes(low.shape))


def test_moe_config_variants():
    low = fe.compile_decoder(MOE, dict(MOE_CFG, norm_topk_prob=True, first_k_dense_replace=0, n_shared_experts=1))
    s = low.shape
    assert s["norm_topk"] and s["first_dense"] == 0 and s["n_shared"] == 1
    assert set(low.names) == set(si.weight_shapes(s))
    assert not any(".mlp.gate_proj." in k for k in low.names)  # no dense layer left


def _moe_variant(old, new):
    assert MOE.count(old) >= 1, old
    return MOE.replace(old, new)


@pytest.mark.parametrize("src,cfg,msg", [
    (None, dict(num_experts_per_tok=9), "top_k"),
    (None, dict(n_routed_experts=300, num_experts_per_tok=2), "experts"),
    (("s <- gated@shared h (SHARED * EXPERT_FFN)", "s <- gated@shared h (SHARED * EXPERT_FFN + 8)"), {}, "multiple"),
    # no router weight on the expert term: not a mixture, every expert on every token
    (("y <- y + MoE.expert_weight w idx e * gated h EXPERT_FFN", "y <- y + gated h EXPERT_FFN"), {},
     "sum over experts"),
    # a loop that skips expert 0
    (("[0..EXPERTS) carry (y)", "[1..EXPERTS) carry (y)"), {}, "sum over experts"),
    # the same parameters for every expert
    (("y <- y + MoE.expert_weight w idx e * gated h EXPERT_FFN",
      "y <- y + MoE.expert_weight w idx e * gated@@blocks.one h EXPERT_FFN"), {}, "sum over experts"),
    (("  x, new_i <- dense_layer x pos mask past_i", "  x, new_i <- moe_layer x pos mask past_i"), {},
     "leading dense"),
    (("w, idx <- MoE.softmax_topk_router@router h top_k=TOPK",
      "w, idx <- MoE.softmax_topk_router@router (h * 2.0) top_k=TOPK"), {}, "router"),
    (("mixture h = do", "mixture h = do\n  h <- Tensor.dropout h"), {}, "post-attention norm"),
    (("  g <- NN.linear@w_gate x dim=width", "  g <- NN.linear@w_gate x dim=width scale=2.0"), {}, "scale"),
])
def test_moe_modules_outside_the_kernels_are_refused(src, cfg, msg):
    text = MOE if src is None else _moe_variant(*src)
    with pytest.raises(fe.LoweringError, match=msg):
        fe.compile_decoder(text, dict(MOE_CFG, **cfg))


def _llama_variants():
    """q/k/v biases, qk-norm, the tanh gelu gate and a tied head."""
    src = LLAMA
    for proj in ("wq", "wk", "wv"):
        src = re.sub(rf"(NN\.linear@{proj} h dim=\([A-Z_]+ \* HEAD_DIM\))", r"\1 bias=true", src)
    src = src.replace("  q <- rope q pos theta=THETA", "  q <- NN.rmsnorm@q_norm q eps=EPS\n  q <- rope q pos theta=THETA")
    src = src.replace("  k <- rope k pos theta=THETA", "  k <- NN.rmsnorm@k_norm k eps=EPS\n  k <- rope k pos theta=THETA")
    return src.replace("Act.silu g", "Act.gelu_tanh g").replace("NN.linear@output dim=VOCAB",
                                                              "NN.linear@tok_embeddings dim=VOCAB")


def _moe_shared_first():
    """The experts' sum accumulated onto the shared MLP's output instead of
    zeros, the router weights renormalised."""
    src = MOE.replace("  y <- Tensor.zeros_like h\n", "  y <- gated@shared h (SHARED * EXPERT_FFN)\n")
    return src.replace("  s <- gated@shared h (SHARED * EXPERT_FFN)\n  return y + s", "  return y")


def _llama_layer_mask():
    """The mask built inside the layer from q and k (the attention built-ins'
    self-attention pattern), windowed."""
    return LLAMA.replace("  y <- attention q k v mask |>",
                         "  keep <- Masking.causal_mask q k window=5\n  y <- attention q k v keep |>")


def test_mask_built_in_the_layer_is_plumbing_with_its_window():
    low = fe.compile_decoder(_llama_layer_mask(), CFG)
    assert low.shape["window"] == 5 and low.names == fe.compile_decoder(LLAMA, CFG).names


def _llama_fused(bias=True):
    """The attention's q, k, v as one projection cut by Attention.split_qkv,
    and the MLP in the composition idiom linear@up |> swiglu |> linear@down."""
    src = LLAMA.replace(
        "  q <- NN.linear@wq h dim=(HEADS * HEAD_DIM) |> reshape_heads heads=HEADS\n"
        "  k <- NN.linear@wk h dim=(KV_HEADS * HEAD_DIM) |> reshape_heads heads=KV_HEADS\n"
        "  v <- NN.linear@wv h dim=(KV_HEADS * HEAD_DIM) |> reshape_heads heads=KV_HEADS\n",
        f"  qkv <- NN.linear@wqkv h dim=((HEADS + 2 * KV_HEADS) * HEAD_DIM){' bias=true' if bias else ''}\n"
        "  q, k, v <- Attention.split_qkv qkv heads=HEADS kv_heads=KV_HEADS\n")
    src = src.replace("  g <- NN.linear@w1 x dim=FFN\n  u <- NN.linear@w3 x dim=FFN\n"
                      "  return Act.silu g * u |> NN.linear@w2 dim=HIDDEN",
                      "  return NN.linear@w13 x dim=(2 * FFN) |> Act.swiglu |> NN.linear@w2 dim=HIDDEN")
    assert "split_qkv" in src and "swiglu" in src
    return src


def _moe_fused():
    """Experts and shared MLP in the swiglu idiom (one gate/up projection each)."""
    src = MOE.replace("gated x width = do\n  g <- NN.linear@w_gate x dim=width\n  u <- NN.linear@w_up x dim=width\n"
                      "  return Act.silu g * u |> NN.linear@w_down dim=HIDDEN",
                      "gated x width = NN.linear@w_gate_up x dim=(2 * width) |> Act.swiglu |> NN.linear@w_down dim=HIDDEN")
    assert "w_gate_up" in src
    return src


def test_fused_projections_map_to_row_ranges():
    low = fe.compile_decoder(_llama_fused(), CFG)
    assert low.shape["bias"] and (low.shape["H"], low.shape["G"], low.shape["d"], low.shape["F"]) == (4, 2, 32, 192)
    assert set(low.names) == set(si.weight_shapes(low.shape))
    p = "model.layers.1."
    assert low.names[p + "self_attn.k_proj.weight"] == "layers.1.attention.wqkv.weight"
    assert low.rows[p + "self_attn.q_proj.weight"] == (0, 128)
    assert low.rows[p + "self_attn.k_proj.bias"] == (128, 192)
    assert low.rows[p + "self_attn.v_proj.weight"] == (192, 256)
    assert (low.rows[p + "mlp.gate_proj.weight"], low.rows[p + "mlp.up_proj.weight"]) == ((0, 192), (192, 384))
    lib = {k: np.full(tuple(v), float(i)) for i, (k, v) in enumerate(si.weight_shapes(low.shape).items())}
    mod = low.module_weights(lib)
    assert mod["layers.1.attention.wqkv.weight"].shape == (256, 128)
    back = low.library_weights(mod)
    assert set(back) == set(lib) and all(np.array_equal(back[k], lib[k]) for k in lib)
    lowm = fe.compile_decoder(_moe_fused(), MOE_CFG)
    assert set(lowm.names) == set(si.weight_shapes(lowm.shape)) and lowm.shape["moe_F"] == 16
    assert lowm.rows["model.layers.2.mlp.experts.4.up_proj.weight"] == (16, 32)
    assert lowm.rows["model.layers.1.mlp.shared_experts.up_proj.weight"] == (32, 64)
    assert lowm.rows["model.layers.0.mlp.up_proj.weight"] == (48, 96)


@pytest.mark.parametrize("old,new,msg", [
    ("dim=((HEADS + 2 * KV_HEADS) * HEAD_DIM)", "dim=((HEADS + 2 * KV_HEADS) * HEAD_DIM + 1)", "fused q/k/v"),
    ("dim=(2 * FFN)", "dim=(2 * FFN + 1)", "even"),
    ("  q, k, v <- Attention.split_qkv qkv heads=HEADS kv_heads=KV_HEADS\n",
     "  q, k, v0 <- Attention.split_qkv qkv heads=HEADS kv_heads=KV_HEADS\n"
     "  v <- NN.linear@wv h dim=(KV_HEADS * HEAD_DIM) bias=true |> reshape_heads heads=KV_HEADS\n", "split_qkv"),
    ("  q, k, v <- Attention.split_qkv qkv heads=HEADS kv_heads=KV_HEADS\n",
     "  k, q, v <- Attention.split_qkv qkv heads=HEADS kv_heads=KV_HEADS\n", "order"),
])
def test_fused_projections_that_do_not_fit_are_refused(old, new, msg):
    src = _llama_fused()
    assert old in src
    with pytest.raises(fe.LoweringError, match=msg):
        fe.compile_decoder(src.replace(old, new), CFG)


@pytest.mark.parametrize("case", ["llama", "llama_variants_window", "llama_layer_mask", "llama_fused", "moe",
                                  "moe_normalised_all_moe", "moe_shared_first", "moe_fused"])
def test_lowered_modules_compute_what_the_oracle_computes(case):
    """The module's own Graph IR on its own parameter paths against the
    oracle on the lowered shape and the re-keyed checkpoint (float64 both),
    for a prompt and then three KV-cached decode steps through the cache the
    module threads: the lowering keeps the module's meaning. For MoE modules
    both the literal loop over experts and its stacked-experts rewrite are
    evaluated."""
    src, cfg = {"llama": (LLAMA, dict(CFG, num_hidden_layers=2)),
                "llama_variants_window": (_llama_variants(), dict(CFG, sliding_window=3)),
                "llama_layer_mask": (_llama_layer_mask(), CFG),
                "llama_fused": (_llama_fused(), CFG),
                "moe_fused": (_moe_fused(), dict(MOE_CFG, norm_topk_prob=True)),
                "moe": (MOE, MOE_CFG),
                "moe_normalised_all_moe": (MOE, dict(MOE_CFG, norm_topk_prob=True, first_k_dense_replace=0)),
                "moe_shared_first": (_moe_shared_first(), dict(MOE_CFG, norm_topk_prob=True))}[case]
    low = fe.compile_decoder(src, cfg)
    if case == "moe_shared_first":
        assert "zeros_like" not in src and low.shape["n_shared"] == 2 and low.shape["norm_topk"]
    if case == "llama_variants_window":
        s = low.shape
        assert s["bias"] and s["qk_norm"] and s["act"] == "gelu_tanh" and s["tie"] and s["window"] == 3
    w = si.make_weights(low.shape, seed=11)
    lib = si.weights_as_f32_numpy(w)
    mod = low.module_weights(lib)
    ids = si.make_ids(2, 7, low.shape["V"], seed=12)
    fed = si.make_ids(2, 3, low.shape["V"], seed=13)  # the decode steps' input tokens
    o = oracle_for(low.shape, w)
    g = fe.build_graph(sx.parse_module(src), cfg)
    graphs = [g]
    if "moe" in case:
        g2 = fe.build_graph(sx.parse_module(src), cfg)
        assert rw.stack_experts(g2) == 1
        graphs.append(g2)

    def close(got, ref):
        assert got.shape == ref.shape
        err = float(np.max(np.abs(got - ref)))
        assert err < 1e-10 * max(1.0, float(np.max(np.abs(ref)))), err

    for gg in graphs:
        cache = o.new_contiguous_cache(2, 16)
        ev = GraphEval(mod)
        got, work = ev.run(gg, ids)
        close(got, o.prefill(ids, cache))
        past, lens = ev.next_past(work, ids), np.full(2, 7)
        for t in range(fed.shape[1]):
            step = fed[:, t:t + 1]
            got, work = ev.run(gg, step, past)
            close(got[:, 0], o.decode_step(fed[:, t], cache, lens))
            past, lens = ev.next_past(work, step), lens + 1


def test_lowered_moe_shape_fills_the_config_the_library_reads():
    """The lowered MoE shape through make_config (host-side ctypes struct,
    no library call): the config.json keys the module read land in the
    C config's mixture-of-experts fields."""
    import paper_2608_19889_gb300 as ax
    low = fe.compile_decoder(MOE, dict(MOE_CFG, norm_topk_prob=True))
    c = ax.make_config(low.shape, max_batch=4, max_context=64)
    assert (c.num_hidden_layers, c.hidden_size, c.intermediate_size, c.vocab_size) == (3, 32, 48, 64)
    assert (c.n_routed_experts, c.num_experts_per_tok, c.moe_intermediate_size, c.n_shared_experts,
            c.first_k_dense_replace, c.norm_topk_prob) == (6, 2, 16, 2, 1, 1)
    assert (c.num_attention_heads, c.num_key_value_heads, c.head_dim, c.hidden_act) == (4, 2, 8, ax.AXON_ACT_SILU)


# ------------------------------------------------------------ conditionals
COND = """import NN
USE <- Config.value @@use_norm default=true
expr_if x = if USE then NN.rmsnorm@a x eps=0.1 else x
ternary x = USE ? NN.rmsnorm@b x eps=0.1 : null
stmt_if x = do
  if USE then do
    return x
  else do
    y <- NN.rmsnorm@c x eps=0.1
    return y
inline x = do h <- NN.rmsnorm@d x eps=0.1; return h
"""


@pytest.mark.parametrize("use", [True, False])
def test_conditional_forms_build_only_the_taken_branch(use):
    mod = sx.parse_module(COND)
    ops = {e: [n.op + ("@" + n.path if n.path else "") for n in fe.build_graph(mod, {"use_norm": use}, entry=e).nodes]
           for e in ("expr_if", "ternary", "stmt_if", "inline")}
    norm = ["input", "NN.rmsnorm@{}"]
    assert ops["expr_if"] == ([norm[0], norm[1].format("a")] if use else ["input"])
    assert ops["ternary"] == ([norm[0], norm[1].format("b")] if use else ["input"])
    assert ops["stmt_if"] == (["input"] if use else [norm[0], norm[1].format("c")])
    assert ops["inline"] == [norm[0], norm[1].format("d")]


def test_statement_if_needs_an_else():
    with pytest.raises(fe.AxonSyntaxError, match="else"):
        sx.parse_module("f x = do\n  if true then do\n    return x\n  y <- x\n  return y\n")


@pytest.mark.parametrize("qk", [True, False])
def test_a_config_switch_in_the_module_selects_the_variant(qk):
    """qk-norm behind a configuration flag, written with the statement-level
    conditional: the lowering sees only the taken branch."""
    src = LLAMA.replace("WINDOW <- Config.value @@sliding_window default=0",
                        "WINDOW <- Config.value @@sliding_window default=0\nQK_NORM <- Config.value @@qk_norm default=false")
    src = src.replace("  q <- rope q pos theta=THETA\n  k <- rope k pos theta=THETA\n",
                      "  q, k <- qk_norm_rope q k pos\n")
    src = src.replace("ffn :: ", "qk_norm_rope q k pos = do\n"
                      "  if QK_NORM then do\n"
                      "    return rope (NN.rmsnorm@q_norm q eps=EPS) pos theta=THETA, "
                      "rope (NN.rmsnorm@k_norm k eps=EPS) pos theta=THETA\n"
                      "  else do\n"
                      "    return rope q pos theta=THETA, rope k pos theta=THETA\n\n"
                      "ffn :: ")
    low = fe.compile_decoder(src, dict(CFG, qk_norm=qk))
    assert low.shape["qk_norm"] == qk
    assert ("model.layers.0.self_attn.q_norm.weight" in low.names) == qk


def test_exports_type_aliases_and_a_scope_on_the_signature():
    src = ("import NN\nexport layer Twin\n\ntype Twin[T] = (T, T)\n\nwidth <- 64\n\n"
           "layer@blk :: Tensor[B,S,D] -> ?Tensor[B,K] -> Tensor[B,S,D]\n"
           "layer x m = do\n  h <- NN.rmsnorm@norm x eps=0.5\n  return x + h\n")
    mod = sx.parse_module(src)
    assert mod.exports == ["layer", "Twin"] and "Twin" in mod.types
    assert mod.definitions["layer"].scope == "blk"
    g = fe.build_graph(mod, {}, entry="layer")
    assert [n.path for n in g.nodes if n.path] == ["blk.norm"]
    assert [n.op for n in g.nodes if n.op == "input"] == ["input", "input"]  # the optional argument too
    with pytest.raises(fe.AxonSyntaxError, match="type alias"):
        sx.parse_module("type Twin T\n")


def test_loops_with_a_step():
    src = ("import NN\nf x = do\n  y <- for i <- [0..7) step=2 carry (x) do\n    x <- x + 1.0\n    yield x\n"
           "  return y\n")
    g = fe.build_graph(sx.parse_module(src), {}, entry="f")
    loop = [n for n in g.nodes if n.op == "loop"][0]
    assert (loop.attrs["start"], loop.attrs["stop"], loop.attrs["step"]) == (0, 7, 2)
    assert GraphEval({}).run(g, np.zeros((1, 1)))[0] == 4.0  # i = 0, 2, 4, 6
    with pytest.raises(fe.AxonGraphError, match="step"):
        fe.build_graph(sx.parse_module(src.replace("step=2", "step=0")), {}, entry="f")
    with pytest.raises(fe.LoweringError, match="one layer per iteration"):
        fe.compile_decoder(LLAMA.replace("[0..LAYERS) carry", "[0..LAYERS) step=2 carry"), CFG)
