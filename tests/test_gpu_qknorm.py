"""GPU parity of per-head qk-norm (Qwen3-family layers: RMSNorm over each
head's d values of q and k, with gains, before RoPE) against the oracle:
prefill on the decode GEMV (few rows) and on the tcgen05 GEMM (many rows),
decode with few and with more than 8 sequences, contiguous and paged caches,
a variable-length batch, and the three precision modes. Normalised q and k
change the attention far beyond the tolerance, so a missing, misplaced or
mis-scaled norm fails."""
import numpy as np
import pytest

import synth_inputs as si
from helpers import FP32_REL_TOL, create, gpu_weights, oracle_for, tiny_tol
from test_gpu_parity import TINY, TINY128, _ax, check, decode_steps, oracle_decode, run_prefill
from test_gpu_persistent import _kinds
from test_gpu_varlen import _case

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_19889_gb300 import build
    build.build()


@pytest.mark.parametrize("base,B,S,prec", [(TINY, 2, 20, "bf16"), (TINY, 2, 100, "bf16"), (TINY128, 2, 100, "fp16"),
                                           (TINY128, 12, 24, "fp16"), (TINY128, 1, 40, "fp32")])
def test_qk_norm_prefill_and_decode(base, B, S, prec):
    ax = _ax()
    shape = dict(base, qk_norm=True)
    w = gpu_weights(shape)
    m = create(shape, w, max_batch=B, max_context=128, fp16=prec == "fp16", fp32=prec == "fp32")
    try:
        if prec != "fp32":  # qk-norm models decode on the launch chain
            assert "decode_persistent" not in _kinds(m, B, [S] * B)
        ids = si.make_ids(B, S, shape["V"], seed=23)
        lg, nxt = run_prefill(m, ids, ax.AXON_LOGITS_ALL, shape["V"])
        o = oracle_for(shape, w)
        cache = o.new_contiguous_cache(B, 128)
        ref = o.prefill(ids, cache)
        plain = oracle_for(base, w)
        far = float(np.max(np.abs(ref - plain.prefill(ids, plain.new_contiguous_cache(B, 128)))))
        assert far > 0.1, far  # the norm changes the logits by far more than the tolerance
        dl, fed = decode_steps(m, nxt, [S] * B, 5, shape["V"])
        refd = oracle_decode(o, cache, fed, [S] * B)
        if prec == "fp32":
            for what, got, want in (("prefill", lg, ref), ("decode", dl, refd)):
                rel = np.max(np.abs(got - want)) / np.max(np.abs(want))
                print(f"qk-norm fp32 {what}: relative error {rel:.3e}")
                assert rel <= FP32_REL_TOL
        else:
            check(lg, ref, tol=tiny_tol(prec), what=f"qk-norm prefill d={shape['d']} S={S} {prec}")
            check(dl, refd, tol=tiny_tol(prec), what=f"qk-norm decode d={shape['d']} B={B} {prec}")
        assert ax.axon_check_device(m)[0] == 0
    finally:
        ax.axon_free(m)


@pytest.mark.parametrize("layout", ["contiguous", "paged"])
def test_qk_norm_varlen_chunks(layout):
    _case(dict(TINY, qk_norm=True), layout, "bf16", first=[37, 5, 70, 1], second=[20, 1, 3, 17])
