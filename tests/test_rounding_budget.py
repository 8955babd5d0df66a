"""CPU checks of the rounding-budget forward (tests/rounding_budget.py): with
no rounding it is the oracle's prompt pass, and at each rounding point the
fp16 error is below the bf16 one (10 vs 7 mantissa bits)."""
import numpy as np
import pytest

import synth_inputs as si
from oracle import decoder as od
from rounding_budget import POINTS, forward, table

torch = pytest.importorskip("torch")

SHAPE = dict(L=2, D=64, H=4, G=2, d=16, F=96, V=80, tie=False, bias=True, theta=1e4, eps=1e-5)


def _case(shape):
    W = {k: np.asarray(v, dtype=np.float64) for k, v in si.weights_as_f32_numpy(si.make_weights(shape)).items()}
    return od.DecoderConfig.from_dict(shape), W, si.make_ids(2, 9, shape["V"], seed=4)


@pytest.mark.parametrize("shape", [SHAPE, dict(SHAPE, bias=False, tie=True, qk_norm=True, window=4,
                                               act="gelu_tanh")])
def test_no_rounding_is_the_oracle(shape):
    cfg, W, ids = _case(shape)
    o = od.Oracle(cfg, W)
    ref = o.prefill(ids, o.new_contiguous_cache(2, 16))
    got = forward(cfg, W, ids)
    assert np.max(np.abs(got - ref)) <= 1e-12 * np.max(np.abs(ref))


def test_fp16_rounding_costs_less_than_bf16_at_every_point():
    cfg, W, ids = _case(SHAPE)
    t = table(cfg, W, ids)
    for pt in POINTS + ("all",):
        f_rms, b_rms = t["fp16"][pt][0], t["bf16"][pt][0]
        assert 0 < f_rms < b_rms, (pt, f_rms, b_rms)


def test_two_term_rounding_keeps_about_twice_the_bits():
    from rounding_budget import rounder
    # magnitudes in [0.25, 4): the second fp16 term stays out of fp16's subnormal range
    rng = np.random.Generator(np.random.PCG64(8))
    x = rng.choice([-1.0, 1.0], size=10000) * 2.0 ** rng.uniform(-2, 2, size=10000)
    for kind, one, two in (("bf16", 2.0 ** -8, 2.0 ** -16), ("fp16", 2.0 ** -11, 2.0 ** -21)):
        e1 = np.max(np.abs(rounder(kind)(x) - x) / np.abs(x))
        e2 = np.max(np.abs(rounder(kind + "x2")(x) - x) / np.abs(x))
        assert e1 <= one and 0 < e2 <= two, (kind, e1, e2)
