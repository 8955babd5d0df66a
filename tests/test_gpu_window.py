"""GPU parity of sliding-window attention (the `window=` argument of the
causal mask) against the oracle: windows not aligned to the 16-token cache
blocks, prompts shorter and longer than the window, decode through the
persistent step and through the launch chain, long contexts whose window
starts many blocks in (split-KV decode), variable-length chunks after a long
past, and the fp32 debug mode."""
import numpy as np
import pytest

import synth_inputs as si
from helpers import FP32_REL_TOL, create, gpu_weights, oracle_for
from test_gpu_parity import TINY, TINY128, _ax, check, decode_steps, oracle_decode, run_prefill
from test_gpu_persistent import _create, _kinds
from test_gpu_varlen import _case

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

WIN = dict(TINY, window=24)
WIN128 = dict(TINY128, window=40)


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_19889_gb300 import build
    build.build()


@pytest.mark.parametrize("persistent", [True, False])
@pytest.mark.parametrize("shape,B,S,max_ctx", [(WIN, 2, 100, 128), (WIN128, 3, 70, 128), (WIN, 2, 20, 128),
                                               (dict(TINY, window=200), 2, 600, 640)])
def test_window_prefill_all_positions_and_decode(shape, B, S, max_ctx, persistent):
    ax = _ax()
    w = gpu_weights(shape)
    m = _create(shape, w, persistent, max_batch=B, max_context=max_ctx, max_prefill_tokens=B * S)
    try:
        ids = si.make_ids(B, S, shape["V"], seed=31)
        lg, nxt = run_prefill(m, ids, ax.AXON_LOGITS_ALL, shape["V"])
        o = oracle_for(shape, w)
        cache = o.new_contiguous_cache(B, max_ctx)
        ref = o.prefill(ids, cache)
        check(lg, ref, what=f"window {shape['window']} prefill S={S}")
        assert np.array_equal(nxt, lg[:, -1].argmax(-1))
        kinds = _kinds(m, B, [max_ctx - 2] * B)  # which decode path runs (the step writes past the test's range)
        assert ("decode_persistent" in kinds) == persistent
        steps = 10
        dl, fed = decode_steps(m, nxt, [S] * B, steps, shape["V"])
        check(dl, oracle_decode(o, cache, fed, [S] * B), what=f"window {shape['window']} decode "
              f"({'persistent' if persistent else 'launch chain'})")
        assert ax.axon_check_device(m)[0] == 0
    finally:
        ax.axon_free(m)


@pytest.mark.parametrize("layout", ["contiguous", "paged"])
def test_window_varlen_chunks_after_a_long_past(layout):
    _case(WIN, layout, "bf16", first=[90, 40, 1], second=[30, 1, 64])


def test_window_fp32_debug_mode():
    ax = _ax()
    shape = WIN
    B, S = 2, 70
    w = gpu_weights(shape)
    m = create(shape, w, max_batch=B, max_context=128, fp32=True)
    try:
        ids = si.make_ids(B, S, shape["V"], seed=9)
        lg, nxt = run_prefill(m, ids, ax.AXON_LOGITS_ALL, shape["V"])
        o = oracle_for(shape, w)
        cache = o.new_contiguous_cache(B, 128)
        ref = o.prefill(ids, cache)
        rel = np.max(np.abs(lg - ref)) / np.max(np.abs(ref))
        print("fp32 window prefill rel", rel)
        assert rel <= FP32_REL_TOL
        dl, fed = decode_steps(m, nxt, [S] * B, 4, shape["V"])
        refd = oracle_decode(o, cache, fed, [S] * B)
        reld = np.max(np.abs(dl - refd)) / np.max(np.abs(refd))
        print("fp32 window decode rel", reld)
        assert reld <= FP32_REL_TOL
    finally:
        ax.axon_free(m)
