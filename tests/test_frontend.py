"""CPU tests of the Axon-subset front end: lexing and parsing, Graph IR
building (definition inlining, scoped parameter paths, loops, configuration
reads), and the lowering of a decoder module onto the library's kernels
(shape and checkpoint-name map), including the variants it accepts and the
modules it must refuse."""
import os
import re

import pytest

from paper_2608_19889_gb300 import frontend as fe
from paper_2608_19889_gb300.frontend import syntax as sx

HERE = os.path.dirname(os.path.abspath(__file__))
LLAMA = open(os.path.join(HERE, "data", "llama_decoder.axon")).read()
CFG = dict(hidden_size=128, num_hidden_layers=2, num_attention_heads=4, num_key_value_heads=2, head_dim=32,
           intermediate_size=192, vocab_size=1000, rope_theta=10000.0, rms_norm_eps=1e-5)


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
