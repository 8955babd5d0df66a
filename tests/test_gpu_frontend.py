"""The Axon-subset front end end to end on the GPU: a decoder written in the
Axon subset is parsed, built into a Graph IR and lowered onto the library's
kernels; the model is created from a checkpoint stored under the module's
own parameter paths, and its prefill and decode logits are compared with
the oracle (which reads the same tensors under the HF names)."""
import os
import re

import numpy as np
import pytest

import synth_inputs as si
from helpers import oracle_for, tiny_tol
from test_gpu_parity import _ax, check, decode_steps, oracle_decode, run_prefill

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

HERE = os.path.dirname(os.path.abspath(__file__))
LLAMA = open(os.path.join(HERE, "data", "llama_decoder.axon")).read()


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_19889_gb300 import build
    build.build()


def _qk_norm_bias_variant(src):
    for proj in ("wq", "wk", "wv"):
        src = re.sub(rf"(NN\.linear@{proj} h dim=\([A-Z_]+ \* HEAD_DIM\))", r"\1 bias=true", src)
    src = src.replace("  q <- rope q pos theta=THETA", "  q <- NN.rmsnorm@q_norm q eps=EPS\n  q <- rope q pos theta=THETA")
    return src.replace("  k <- rope k pos theta=THETA", "  k <- NN.rmsnorm@k_norm k eps=EPS\n  k <- rope k pos theta=THETA")


@pytest.mark.parametrize("variant,prec", [("plain", "bf16"), ("qk_norm_bias", "fp16")])
def test_axon_module_through_the_kernels(variant, prec):
    from paper_2608_19889_gb300 import frontend as fe
    ax = _ax()
    src = LLAMA if variant == "plain" else _qk_norm_bias_variant(LLAMA)
    config = dict(hidden_size=256, num_hidden_layers=2, num_attention_heads=8, num_key_value_heads=2, head_dim=64,
                  intermediate_size=320, vocab_size=1000, rope_theta=10000.0, rms_norm_eps=1e-5)
    low = fe.compile_decoder(src, config)
    shape = low.shape
    assert shape["qk_norm"] == (variant != "plain") and shape["bias"] == (variant != "plain")
    w_lib = si.make_weights(shape, device="cuda")       # library (HF) names, for the oracle
    checkpoint = low.module_weights(w_lib)                # the module's own names, for the front end
    assert "layers.1.feed_forward.w2.weight" in checkpoint
    B, S = 2, 80
    m = fe.create_model(low, checkpoint, max_batch=B, max_context=128,
                        precision=ax.AXON_FP16 if prec == "fp16" else ax.AXON_BF16)
    try:
        ids = si.make_ids(B, S, shape["V"], seed=37)
        lg, nxt = run_prefill(m, ids, ax.AXON_LOGITS_ALL, shape["V"])
        o = oracle_for(shape, w_lib)
        cache = o.new_contiguous_cache(B, 128)
        check(lg, o.prefill(ids, cache), tol=tiny_tol(prec), what=f"axon module ({variant}) prefill")
        dl, fed = decode_steps(m, nxt, [S] * B, 5, shape["V"])
        check(dl, oracle_decode(o, cache, fed, [S] * B), tol=tiny_tol(prec), what=f"axon module ({variant}) decode")
        assert ax.axon_check_device(m)[0] == 0
    finally:
        ax.axon_free(m)
