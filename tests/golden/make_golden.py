"""Writes tests/golden/tiny_decoder.json: the oracle's logits for small
seeded decoders (prefill of the last position, then greedy cached decode
steps), for the regression pin in tests/test_golden.py.

The paper prints no worked numbers for the decoder forward, so these values
are not the paper's: they are the oracle's own output, written by this
script, which calls only oracle/ and the seeded input module. A later change
to the oracle's arithmetic shows up as a mismatch; regenerate the file only
with a commit that names the passage of the paper (or the reading of it)
that justifies the change.

Run from the repository root:  python tests/golden/make_golden.py
"""
import json
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

import synth_inputs as si  # noqa: E402
from oracle import decoder as od  # noqa: E402

BASE = dict(L=2, D=32, H=4, G=2, d=8, F=48, V=64, tie=False, bias=True, theta=1e4, eps=1e-5)
CASES = {
    "llama_bias_untied": BASE,
    "tied_no_bias": dict(BASE, tie=True, bias=False),
    "sliding_window_3": dict(BASE, window=3),
    "gelu_gate": dict(BASE, act="gelu_tanh"),
    "rope_scaling": dict(BASE, rope_factor=4.0, rope_low=1.0, rope_high=2.0, rope_orig=16),
    "qk_norm": dict(BASE, qk_norm=True),
}
B, S, STEPS = 2, 7, 3


def case(shape):
    w = si.weights_as_f32_numpy(si.make_weights(shape, seed=0))
    o = od.Oracle(od.DecoderConfig.from_dict(shape), w)
    ids = si.make_ids(B, S, shape["V"], seed=1)
    cache = o.new_contiguous_cache(B, S + STEPS)
    toks, logits = o.generate(ids, STEPS + 1, cache)
    return {"ids": ids.tolist(), "tokens": toks.tolist(), "logits": [[[float(x) for x in row] for row in seq]
                                                                      for seq in logits]}


def main():
    out = {"shape_base": BASE, "batch": B, "prompt": S, "decode_steps": STEPS,
           "cases": {name: dict(shape=shape, **case(shape)) for name, shape in CASES.items()}}
    path = os.path.join(os.path.dirname(os.path.abspath(__file__)), "tiny_decoder.json")
    with open(path, "w") as f:
        json.dump(out, f, indent=None, separators=(",", ":"))
    print(path)


if __name__ == "__main__":
    main()
