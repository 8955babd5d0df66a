"""The allocation-free decode step (axon_decode_step_noalloc) against the
regular one, through the C ABI, on two calls in a row.

Some callers cannot allocate on their call path (their allocator is owned by
someone else or locked after start-up); for them the library offers a decode
step that instantiates no CUDA graph and takes its attention merge scratch
from a fixed library-owned device array. The second call checks that what
the first call left in that shared array does not leak into the result.
This file is collected last so a failure here comes after every other test."""
import numpy as np
import pytest

import synth_inputs as si
from helpers import LOGIT_TOL, create, gpu_weights, parity

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

SHAPE = dict(L=2, D=256, H=8, G=2, d=128, F=320, V=1000, tie=False, bias=True, theta=1e4, eps=1e-5)


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_19889_gb300 import build
    build.build()


def test_noalloc_decode_matches_regular_decode_two_calls():
    import paper_2608_19889_gb300 as ax
    B, S = 3, 150  # 10 key blocks: several key splits, so the merge scratch is used
    w = gpu_weights(SHAPE)
    m = create(SHAPE, w, max_batch=B, max_context=256)
    try:
        ids = torch.from_numpy(si.make_ids(B, S, SHAPE["V"], seed=11)).cuda()
        tok = torch.empty(B, dtype=torch.int32, device="cuda")
        ax.axon_prefill(m, ids, next_tokens=tok)
        for step in range(2):
            pos = S + step
            ref_logits = torch.empty(B, SHAPE["V"], device="cuda")
            ref_next = torch.empty(B, dtype=torch.int32, device="cuda")
            ctx = torch.full((B,), pos, dtype=torch.int32, device="cuda")
            ax.axon_decode_step(m, tok.clone(), ctx, logits=ref_logits, next_tokens=ref_next)
            # Same step again from the same cache state (position pos is rewritten
            # with the same K/V) through the allocation-free entry point.
            got_logits = torch.full((B, SHAPE["V"]), float("nan"), device="cuda")
            got_next = torch.empty(B, dtype=torch.int32, device="cuda")
            ctx2 = torch.full((B,), pos, dtype=torch.int32, device="cuda")
            ax.axon_decode_step_noalloc(m, tok.clone(), ctx2, logits=got_logits, next_tokens=got_next)
            torch.cuda.synchronize()
            a, b = ref_logits.cpu().numpy(), got_logits.cpu().numpy()
            maxd, agree, hard = parity(b, a)
            print(f"call {step}: max|dlogit| vs axon_decode_step {maxd:.3e}, top1 {agree:.3f}")
            assert np.isfinite(b).all()
            assert maxd <= LOGIT_TOL
            assert hard == 0
            assert np.array_equal(got_next.cpu().numpy(), b.argmax(-1))
            assert np.array_equal(ctx2.cpu().numpy(), np.full(B, pos + 1))
            tok = ref_next
        assert ax.axon_check_device(m)[0] == 0
    finally:
        ax.axon_free(m)
