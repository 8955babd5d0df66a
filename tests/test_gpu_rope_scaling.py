"""GPU parity with RoPE frequency scaling (the stretch of Llama-3.1-family
configs) against the oracle: an original context of 64 puts the rotary
frequencies in all three bands (kept, blended, stretched), and prompts of
150 tokens rotate far past it. The q and k projections are scaled by 8
(exact in bf16) so that attention is sharp enough for the rotary
frequencies to move the logits by far more than the tolerance; fp16 operand
mode keeps the rounding of those larger scores inside it."""
import numpy as np
import pytest

import synth_inputs as si
from helpers import create, gpu_weights, oracle_for
from test_gpu_parity import TINY, TINY128, _ax, check, decode_steps, oracle_decode, run_prefill

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

SCALED = dict(rope_factor=8.0, rope_low=1.0, rope_high=4.0, rope_orig=64)


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_19889_gb300 import build
    build.build()


@pytest.mark.parametrize("base", [TINY128, TINY])
def test_rope_scaling_prefill_and_decode(base):
    ax = _ax()
    shape = dict(base, **SCALED)
    B, S = 2, 150
    w = gpu_weights(shape)
    for k in w:
        if k.endswith(("q_proj.weight", "k_proj.weight")):
            w[k] = w[k] * 8
    m = create(shape, w, max_batch=B, max_context=176, fp16=True)
    try:
        ids = si.make_ids(B, S, shape["V"], seed=13)
        lg, nxt = run_prefill(m, ids, ax.AXON_LOGITS_ALL, shape["V"])
        o = oracle_for(shape, w)
        cache = o.new_contiguous_cache(B, 176)
        ref = o.prefill(ids, cache)
        check(lg, ref, what=f"rope scaling d={shape['d']} prefill")
        # the scaling matters here: the unscaled oracle is farther off than the tolerance
        plain = oracle_for(base, w)
        far = np.max(np.abs(plain.prefill(ids, plain.new_contiguous_cache(B, 176)) - ref))
        assert far > 0.5, far
        dl, fed = decode_steps(m, nxt, [S] * B, 8, shape["V"])
        check(dl, oracle_decode(o, cache, fed, [S] * B), what=f"rope scaling d={shape['d']} decode")
        assert ax.axon_check_device(m)[0] == 0
    finally:
        ax.axon_free(m)
