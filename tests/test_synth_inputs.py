"""The seeded input generators shared by the oracle and the CUDA path:
ranges, shapes, determinism, and the block table's integer structure."""
import numpy as np
import pytest

import synth_inputs as si


def test_block_table_is_a_partial_permutation_of_the_pool():
    caps = [33, 16, 1, 70]
    bt = si.make_block_table(caps, 16, 6, 40, seed=3)
    assert bt.shape == (4, 6) and bt.dtype == np.int32
    need = [3, 1, 1, 5]
    used = []
    for b, n in enumerate(need):
        assert np.all(bt[b, :n] >= 0) and np.all(bt[b, :n] < 40)
        assert np.all(bt[b, n:] == -1)
        used += list(bt[b, :n])
    assert len(set(used)) == len(used) == sum(need)  # no pool block serves two slots
    assert np.array_equal(bt, si.make_block_table(caps, 16, 6, 40, seed=3))
    assert not np.array_equal(bt, si.make_block_table(caps, 16, 6, 40, seed=4))
    with pytest.raises(ValueError):
        si.make_block_table(caps, 16, 6, 9, seed=3)


def test_ids_and_context_lengths_stay_in_range_and_repeat_by_seed():
    ids = si.make_ids(3, 500, 1000, seed=5)
    assert ids.shape == (3, 500) and ids.dtype == np.int32
    assert ids.min() >= 0 and ids.max() < 1000
    assert np.array_equal(ids, si.make_ids(3, 500, 1000, seed=5))
    lens = si.make_context_lens(64, 512, 4096, seed=2)
    assert lens.min() >= 512 and lens.max() <= 4096
    assert np.array_equal(lens, si.make_context_lens(64, 512, 4096, seed=2))


def test_weights_by_name_are_deterministic_bf16_with_gains_near_one():
    torch = pytest.importorskip("torch")
    m = dict(L=1, D=64, H=2, G=1, d=32, F=96, V=50, tie=False, bias=True, theta=1e4, eps=1e-5)
    w = si.make_weights(m, seed=0)
    w2 = si.make_weights(m, seed=0)
    assert all(t.dtype == torch.bfloat16 for t in w.values())
    assert all(torch.equal(w[k], w2[k]) for k in w)
    assert set(si.weight_shapes(m)) == set(w)
    q = w["model.layers.0.self_attn.q_proj.weight"].float()
    assert tuple(q.shape) == (64, 64) and 0.015 < float(q.std()) < 0.025
    g = w["model.layers.0.input_layernorm.weight"].float()
    assert abs(float(g.mean()) - 1.0) < 0.02
    other = si.make_weights(m, seed=1)
    assert not torch.equal(w["lm_head.weight"], other["lm_head.weight"])
