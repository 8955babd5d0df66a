"""CPU oracle for the Llama-family decoder forward (prefill + KV-cached greedy decode).

TEST INFRASTRUCTURE ONLY. Nothing in the product path imports this package:
only `tests/`, `__graft_entry__.smoke()` and the CPU-baseline leg of `bench.py`
use it. It shares no code with the CUDA library: it reads HF-named weights,
computes in float64 with numpy, and keeps its own KV caches.

Every function cites the passage of the Axon paper (arxiv 2608.19889) whose
built-in operation it restates. The paper names the operations (NN.rmsnorm,
NN.linear, Attention.attention with grouped-query heads, Positions with
past_length, Cache.update/append, Act.swiglu) but prints no formulas for them;
the readings taken where it is silent are listed in `decoder.READINGS`.
`gpt2` holds the GPT-2 causal LM of the paper's complete model definition
(LayerNorm, learned positions, fused biased projections, gelu_new MLP), with
its own READINGS.
"""
from .decoder import (  # noqa: F401
    DecoderConfig,
    READINGS,
    rmsnorm,
    linear,
    rope_inv_freq,
    rope,
    silu,
    swiglu,
    softmax,
    attention_one_query,
    causal_attention,
    ContiguousKV,
    PagedKV,
    slot_of,
    Oracle,
    argmax_lowest,
    moe_route,
    topk_lowest,
)
