"""Change detector for the oracle: tests/golden/tiny_decoder.json holds what
tests/golden/make_golden.py wrote from the oracle itself (the paper prints no
worked numbers for this forward). It catches unintended changes to the
oracle's arithmetic but pins the oracle only to itself; the other oracle
tests pin it to the paper and to mathematics. The tolerance leaves room for
the summation order of another BLAS build or thread count (float64 sums of
a few hundred terms); the greedy tokens must match exactly."""
import json
import os

import numpy as np
import pytest

import synth_inputs as si
from oracle import decoder as od

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "tiny_decoder.json")
DATA = json.load(open(GOLDEN))


@pytest.mark.parametrize("name", sorted(DATA["cases"]))
def test_oracle_reproduces_the_stored_generation(name):
    c = DATA["cases"][name]
    shape = c["shape"]
    w = si.weights_as_f32_numpy(si.make_weights(shape, seed=0))
    o = od.Oracle(od.DecoderConfig.from_dict(shape), w)
    ids = np.array(c["ids"])
    assert np.array_equal(ids, si.make_ids(DATA["batch"], DATA["prompt"], shape["V"], seed=1))
    cache = o.new_contiguous_cache(DATA["batch"], DATA["prompt"] + DATA["decode_steps"])
    toks, logits = o.generate(ids, DATA["decode_steps"] + 1, cache)
    assert np.array_equal(toks, np.array(c["tokens"]))
    assert np.allclose(logits, np.array(c["logits"]), rtol=1e-9, atol=1e-9)


def test_cases_differ_from_each_other():
    # every variant changes the result, so each case pins its own feature
    base = np.array(DATA["cases"]["llama_bias_untied"]["logits"])
    for name, c in DATA["cases"].items():
        if name != "llama_bias_untied":
            assert not np.allclose(np.array(c["logits"]), base), name
