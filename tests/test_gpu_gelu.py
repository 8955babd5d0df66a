"""GPU parity of the gated-GELU MLP (hidden_act gelu_tanh, the gelu_new of
the GPT-2 listing on the gate) against the oracle, in the prefill GEMMs, the
decode launch chain and the persistent decode step. The gate projection is
scaled by 8 (exact in bf16) so that the two activations differ by far more
than the tolerance: the same run is also checked to be far from SiLU."""
import numpy as np
import pytest

import synth_inputs as si
from helpers import LOGIT_TOL, gpu_weights, oracle_for
from test_gpu_parity import TINY, TINY128, _ax, check, decode_steps, oracle_decode, run_prefill
from test_gpu_persistent import _create, _kinds

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_19889_gb300 import build
    build.build()


@pytest.mark.parametrize("base,persistent,prec", [(TINY, True, "bf16"), (TINY, False, "bf16"),
                                                  (TINY128, True, "fp16"), (TINY128, False, "fp16")])
def test_gated_gelu_prefill_and_decode(base, persistent, prec):
    ax = _ax()
    shape = dict(base, act="gelu_tanh")
    B, S = 2, 100  # 200 rows: the prefill projections run on the tcgen05 GEMM
    w = gpu_weights(shape)
    for k in w:
        if k.endswith("gate_proj.weight"):
            w[k] = w[k] * 8
    m = _create(shape, w, persistent, max_batch=B, max_context=128, fp16=prec == "fp16")
    try:
        assert ("decode_persistent" in _kinds(m, B, [120] * B)) == persistent
        ids = si.make_ids(B, S, shape["V"], seed=41)
        lg, nxt = run_prefill(m, ids, ax.AXON_LOGITS_ALL, shape["V"])
        o = oracle_for(shape, w)
        cache = o.new_contiguous_cache(B, 128)
        ref = o.prefill(ids, cache)
        check(lg, ref, what=f"gated gelu prefill d={shape['d']} {prec}")
        silu = oracle_for(base, w)
        far = float(np.max(np.abs(lg - silu.prefill(ids, silu.new_contiguous_cache(B, 128)))))
        assert far > 2 * LOGIT_TOL, far
        dl, fed = decode_steps(m, nxt, [S] * B, 6, shape["V"])
        check(dl, oracle_decode(o, cache, fed, [S] * B),
              what=f"gated gelu decode ({'persistent' if persistent else 'launch chain'})")
        assert ax.axon_check_device(m)[0] == 0
    finally:
        ax.axon_free(m)
