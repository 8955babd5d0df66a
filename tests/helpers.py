"""Shared test machinery: model construction through the C ABI, the oracle
side of a comparison, and the parity statistics.

The oracle and the CUDA library never see each other: both receive the same
seeded inputs from `synth_inputs`, and only the comparison below looks at
both results."""
from __future__ import annotations

import numpy as np

import synth_inputs as si

LOGIT_TOL = 5e-2  # bf16 weights, fp32 accumulation: max |delta logit|
FP32_REL_TOL = 1e-4  # fp32 debug mode: max |delta| / max |oracle logit|
TOP1_MIN = 0.99
# Tiny shapes (D <= 256, two layers): a few times the largest error observed
# there (bf16 operands 5.0e-3, fp16 operands 5.8e-4), so that a regression in
# a tensor-core epilogue fails long before the model-scale bound above.
TINY_TOL = {"bf16": 1e-2, "fp16": 2e-3}


def tiny_tol(prec: str) -> float:
    return TINY_TOL[prec]


def parity(gpu: np.ndarray, ref: np.ndarray):
    """(max |delta|, top-1 agreement, hard mismatches). A hard mismatch is a
    top-1 disagreement where the oracle's top-2 gap exceeds twice the
    observed max |delta|. It cannot occur: a flip needs a delta of at least
    half the gap (tests/test_parity_stats.py), so the count is a diagnostic
    and the binding checks are max |delta| against the tolerance and the
    raw top-1 floors."""
    gpu = np.asarray(gpu, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    maxd = float(np.max(np.abs(gpu - ref)))
    g_top = gpu.argmax(-1)
    r_top = ref.argmax(-1)
    agree = g_top == r_top
    srt = np.sort(ref, axis=-1)
    gap = srt[..., -1] - srt[..., -2]
    hard = int(np.sum(~agree & (gap > 2 * maxd)))
    return maxd, float(agree.mean()), hard


def gpu_weights(shape: dict, seed: int = si.SEED_WEIGHTS):
    import torch
    return si.make_weights(shape, seed=seed, device="cuda" if torch.cuda.is_available() else "cpu")


def create(shape, weights, max_batch, max_context, layout="contiguous", num_blocks=0, fp32=False,
           max_prefill_tokens=0, fp16=False):
    import paper_2608_19889_gb300 as ax
    prec = ax.AXON_FP32_DEBUG if fp32 else (ax.AXON_FP16 if fp16 else ax.AXON_BF16)
    cfg = ax.make_config(shape, max_batch, max_context,
                         kv_layout=ax.AXON_KV_PAGED if layout == "paged" else ax.AXON_KV_CONTIGUOUS,
                         kv_num_blocks=num_blocks, precision=prec, max_prefill_tokens=max_prefill_tokens)
    return ax.axon_model_create(cfg, weights)


def oracle_for(shape, weights, keep_f64=True):
    from oracle import decoder as od
    return od.Oracle(od.DecoderConfig.from_dict(shape), si.weights_as_f32_numpy(weights), keep_f64=keep_f64)
