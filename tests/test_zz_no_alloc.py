"""The allocation-free decode step (axon_decode_step_noalloc) through the C
ABI, on two calls in a row, against the regular decode step and the oracle.

Some callers cannot allocate on their call path: their device memory pool is
owned by another component, or their allocator is locked once serving has
started. The regular decode step instantiates a CUDA graph the first time it
meets a new pointer set, and instantiation allocates. The allocation-free
step launches the same kernels directly and takes the split-KV attention's
merge scratch (partial softmax states and tickets) from one fixed device
array owned by the library.

Each case below is chosen so that the attention really splits the keys, and
so really writes and merges partial states in that shared array:
  * launch chain (B > 8) over 10 key blocks of capacity: 2 key splits per
    (sequence, kv head), the same count as the regular step, so results must
    be bit-identical;
  * launch chain with more splits than the fixed array holds: the model is
    created with a grid budget of 1024 attention CTAs (AXON_ATTN_TARGET_CTAS),
    which gives the regular step 32 splits of its 128 blocks of capacity; the
    fixed array keeps 256 / (B * kv heads) = 8, so the 94 blocks of context
    fall into 8 splits of 12 blocks instead of 12 splits of 8, and the fp32
    merge order and the 16-bit rounding of the attention output differ;
  * the persistent single-launch step (B <= 8) over more than 64 key blocks,
    which it cuts into items of 16 blocks: 5 splits, bit-identical.
The second call checks that what the first call left in the shared array
does not leak into its result. This file is collected last so a failure
here comes after every other test."""
import os

import numpy as np
import pytest

import synth_inputs as si
from helpers import create, gpu_weights, oracle_for, parity, tiny_tol

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

SHAPE = dict(L=2, D=256, H=8, G=2, d=128, F=320, V=1000, tie=False, bias=True, theta=1e4, eps=1e-5)

# (case, B, prompt length, max_context, bit-identical to the regular step,
#  attention grid budget at creation or None)
CASES = [
    ("chain_2_splits", 12, 140, 160, True, None),
    ("chain_splits_clamped", 16, 1500, 2048, False, 1024),
    ("persistent_5_splits", 2, 1100, 1280, True, None),
]


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_19889_gb300 import build
    build.build()


@pytest.mark.parametrize("prec", ["bf16", "fp16"])
@pytest.mark.parametrize("case,B,S,max_ctx,identical,target", CASES)
def test_noalloc_decode_two_calls(case, B, S, max_ctx, identical, target, prec):
    import paper_2608_19889_gb300 as ax
    V = SHAPE["V"]
    w = gpu_weights(SHAPE)
    old = os.environ.pop("AXON_ATTN_TARGET_CTAS", None)
    try:
        if target:
            os.environ["AXON_ATTN_TARGET_CTAS"] = str(target)
        m = create(SHAPE, w, max_batch=B, max_context=max_ctx, fp16=prec == "fp16")
    finally:
        os.environ.pop("AXON_ATTN_TARGET_CTAS", None)
        if old is not None:
            os.environ["AXON_ATTN_TARGET_CTAS"] = old
    try:
        ids = si.make_ids(B, S, V, seed=11)
        tok = torch.empty(B, dtype=torch.int32, device="cuda")
        ax.axon_prefill(m, torch.from_numpy(ids).cuda(), next_tokens=tok)
        o = oracle_for(SHAPE, w)
        cache = o.new_contiguous_cache(B, max_ctx)
        o.prefill(ids, cache, last_only=True)
        for call in range(2):
            pos = S + call
            fed = tok.cpu().numpy().copy()
            ref_logits = torch.empty(B, V, device="cuda")
            ref_next = torch.empty(B, dtype=torch.int32, device="cuda")
            ctx = torch.full((B,), pos, dtype=torch.int32, device="cuda")
            ax.axon_decode_step(m, tok.clone(), ctx, logits=ref_logits, next_tokens=ref_next)
            # The same step again from the same cache state (position pos is
            # rewritten with the same K/V) through the allocation-free entry point.
            got_logits = torch.full((B, V), float("nan"), device="cuda")
            got_next = torch.empty(B, dtype=torch.int32, device="cuda")
            ctx2 = torch.full((B,), pos, dtype=torch.int32, device="cuda")
            ax.axon_decode_step_noalloc(m, tok.clone(), ctx2, logits=got_logits, next_tokens=got_next)
            torch.cuda.synchronize()
            a, b = ref_logits.cpu().numpy(), got_logits.cpu().numpy()
            assert np.isfinite(b).all()
            d_reg = float(np.max(np.abs(b - a)))
            want = o.decode_step(fed, cache, np.full(B, pos))
            d_orc, agree, hard = parity(b, want)
            print(f"{case} {prec} call {call}: vs axon_decode_step {d_reg:.3e}, vs oracle {d_orc:.3e} "
                  f"(top1 {agree:.3f})")
            if identical:
                assert d_reg == 0.0, f"{case}: same key splits, results must be bit-identical"
            else:
                assert d_reg <= tiny_tol(prec)
            assert d_orc <= tiny_tol(prec) and hard == 0
            assert np.array_equal(got_next.cpu().numpy(), b.argmax(-1))
            assert np.array_equal(ctx2.cpu().numpy(), np.full(B, pos + 1))
            tok = got_next
        assert ax.axon_check_device(m)[0] == 0
    finally:
        ax.axon_free(m)
