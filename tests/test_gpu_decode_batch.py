"""Decode with 9-32 sequences (the launch chain with its per-batch projection
choices) at tiny shapes, and a model created from host-resident weights,
against the oracle through the C ABI."""
import numpy as np
import pytest

import synth_inputs as si
from helpers import create, gpu_weights, oracle_for, tiny_tol
from test_gpu_parity import TINY, TINY128, _ax, check, decode_steps, oracle_decode, run_prefill
from test_gpu_persistent import _kinds

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_19889_gb300 import build
    build.build()


@pytest.mark.parametrize("prec", ["bf16", "fp16"])
@pytest.mark.parametrize("shape,B", [(TINY128, 12), (TINY, 16), (TINY128, 32)])
def test_decode_batch_9_to_32(shape, B, prec):
    """More than 8 sequences: no persistent step; the launch chain decodes
    (GEMV projections up to 32 tokens, split-K GEMM for O and down where it
    applies). Prefill of B x 24 rows on the tcgen05 GEMM, then 6 steps."""
    ax = _ax()
    S, n = 24, 6
    w = gpu_weights(shape)
    m = create(shape, w, max_batch=B, max_context=64, fp16=prec == "fp16")
    try:
        assert "decode_persistent" not in _kinds(m, B, [S] * B)
        ids = si.make_ids(B, S, shape["V"], seed=23)
        lg, nxt = run_prefill(m, ids, ax.AXON_LOGITS_LAST, shape["V"])
        o = oracle_for(shape, w)
        cache = o.new_contiguous_cache(B, 64)
        check(lg, o.prefill(ids, cache, last_only=True)[:, -1], tol=tiny_tol(prec), what=f"B={B} prefill")
        dl, fed = decode_steps(m, nxt, [S] * B, n, shape["V"])
        check(dl, oracle_decode(o, cache, fed, [S] * B), tol=tiny_tol(prec), what=f"B={B} decode ({prec})")
        assert ax.axon_check_device(m)[0] == 0
    finally:
        ax.axon_free(m)


def test_model_from_host_resident_weights():
    """axon_model_create reads weight tensors through host pointers as well
    as device pointers: the model built from host tensors gives the same
    logits, bit for bit, as one built from device copies of them, and both
    match the oracle."""
    ax = _ax()
    shape = TINY
    B, S = 2, 40
    w_host = si.make_weights(shape, device="cpu")
    assert all(not t.is_cuda for t in w_host.values())
    w_dev = {k: v.cuda() for k, v in w_host.items()}
    mh = create(shape, w_host, max_batch=B, max_context=64)
    md = create(shape, w_dev, max_batch=B, max_context=64)
    try:
        ids = si.make_ids(B, S, shape["V"], seed=29)
        lh, nh = run_prefill(mh, ids, ax.AXON_LOGITS_ALL, shape["V"])
        ld, nd = run_prefill(md, ids, ax.AXON_LOGITS_ALL, shape["V"])
        assert np.array_equal(lh, ld) and np.array_equal(nh, nd)
        o = oracle_for(shape, w_host)
        cache = o.new_contiguous_cache(B, 64)
        check(lh, o.prefill(ids, cache), tol=tiny_tol("bf16"), what="host-weight model prefill")
        dl, fed = decode_steps(mh, nh, [S] * B, 4, shape["V"])
        check(dl, oracle_decode(o, cache, fed, [S] * B), tol=tiny_tol("bf16"), what="host-weight model decode")
    finally:
        ax.axon_free(mh)
        ax.axon_free(md)
