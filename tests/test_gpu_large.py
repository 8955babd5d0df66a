"""Parity at the paper's 8B- and 32B-class widths: full-width layers with
few layers (prefill through the tensor-core GEMM, B=64 paged decode), and
the full-depth models on a short prompt. Slow (the float64 oracle does the
same work on the host).

These run in AXON_FP16 (the bf16 checkpoint converted to fp16 operands):
at these widths the random-init logits have a standard deviation of 1.3-1.4,
and rounding GEMM operands and the KV cache to bf16 alone moves the largest
of the 128k-152k logits past the 5e-2 bound (about 0.06-0.07 on the
two-layer 8B-width case below). fp16 operands cut that rounding 8x. The
bf16 mode is run on the same case under a looser regression bound; parity
at these widths is claimed for fp16 mode only."""
import numpy as np
import pytest

import synth_inputs as si
from helpers import create, oracle_for
from test_gpu_parity import check, decode_steps, oracle_decode, run_prefill

torch = pytest.importorskip("torch")
pytestmark = [pytest.mark.gpu, pytest.mark.slow]


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_19889_gb300 import build
    build.build()


def shape(name, **over):
    m = dict(si.MODEL_SHAPES[name])
    m.update(over)
    return m


class LazyF32(dict):
    """HF name -> bf16 torch tensor on the host, widened to float32 numpy on
    each access (the oracle's lazy mode widens it further to float64)."""

    def __getitem__(self, k):
        return super().__getitem__(k).float().numpy()


BF16_FLOOR_8B_WIDTH = 8e-2  # regression bound for bf16 mode at 8B width (no parity claim; measured 0.057-0.073)


@pytest.mark.parametrize("prec", ["fp16", "bf16"])
def test_8b_width_two_layers_tensor_core_prefill_and_decode(prec):
    import paper_2608_19889_gb300 as ax
    m = shape("8b", L=2)
    B, S = 2, 130  # 260 rows: three 128-row tiles, ragged
    tol = 5e-2 if prec == "fp16" else BF16_FLOOR_8B_WIDTH
    w = si.make_weights(m, device="cuda")
    model = create(m, w, max_batch=B, max_context=160, max_prefill_tokens=B * S, fp16=prec == "fp16")
    try:
        ids = si.make_ids(B, S, m["V"], seed=21)
        lg, nxt = run_prefill(model, ids, ax.AXON_LOGITS_LAST, m["V"])
        dl, fed = decode_steps(model, nxt, [S] * B, 3, m["V"])
        o = oracle_for(m, w)
        cache = o.new_contiguous_cache(B, 160)
        ref = o.prefill(ids, cache, last_only=True)[:, -1]
        check(lg, ref, tol=tol, what=f"8b-width prefill ({prec})")
        check(dl, oracle_decode(o, cache, fed, [S] * B), tol=tol, what=f"8b-width decode ({prec})")
    finally:
        ax.axon_free(model)


def test_8b_width_paged_batch64_decode():
    """B=64 decode (the 64-token projection path) over a shuffled paged cache
    with ragged contexts, each sequence prefilled on its own block-table row."""
    import paper_2608_19889_gb300 as ax
    m = shape("8b", L=1)
    B, n_new = 64, 3
    lens = si.make_context_lens(B, 16, 100, seed=si.SEED_CTX)
    max_ctx = 112
    caps = lens + n_new
    num_blocks = int(sum(-(-int(c) // 16) for c in caps)) + 16
    bt_np = si.make_block_table(caps, 16, max_ctx // 16, num_blocks, seed=si.SEED_BLOCKS)
    w = si.make_weights(m, device="cuda")
    model = create(m, w, max_batch=B, max_context=max_ctx, layout="paged", num_blocks=num_blocks,
                   max_prefill_tokens=max_ctx, fp16=True)
    try:
        bt = torch.from_numpy(bt_np).cuda()
        first = []
        o = oracle_for(m, w)
        cache = o.new_paged_cache(num_blocks, 16, bt_np)
        ref_first = []
        for b in range(B):
            ids = si.make_ids(1, int(lens[b]), m["V"], seed=100 + b)
            lg, nxt = run_prefill(model, ids, ax.AXON_LOGITS_LAST, m["V"], block_table=bt[b:b + 1])
            first.append(int(nxt[0]))
            # the oracle's paged cache addresses sequence b through row b of the table
            sub = o.new_paged_cache(num_blocks, 16, bt_np[b:b + 1])
            sub.K, sub.V = cache.K, cache.V
            ref_first.append(o.prefill(ids, sub, last_only=True)[0, -1])
            if b < 4:
                check(lg, ref_first[-1][None], what=f"paged prefill seq {b}")
        dl, fed = decode_steps(model, np.array(first), lens, n_new, m["V"], block_table=bt)
        check(dl, oracle_decode(o, cache, fed, lens), what="B=64 paged decode", top1=True)
    finally:
        ax.axon_free(model)


def test_32b_width_one_layer():
    import paper_2608_19889_gb300 as ax
    m = shape("32b", L=1)
    B, S = 1, 70
    w = si.make_weights(m, device="cuda")
    model = create(m, w, max_batch=B, max_context=96, max_prefill_tokens=B * S, fp16=True)
    try:
        ids = si.make_ids(B, S, m["V"], seed=31)
        lg, nxt = run_prefill(model, ids, ax.AXON_LOGITS_ALL, m["V"])
        dl, fed = decode_steps(model, nxt, [S] * B, 3, m["V"])
        o = oracle_for(m, w)
        cache = o.new_contiguous_cache(B, 96)
        check(lg, o.prefill(ids, cache), what="32b-width prefill (all positions)", top1=True)
        check(dl, oracle_decode(o, cache, fed, [S] * B), what="32b-width decode")
    finally:
        ax.axon_free(model)


@pytest.mark.parametrize("name", ["8b", "32b"])
def test_full_depth_short_prompt(name):
    """All layers at full width: B=1, 80-token prompt (tensor-core prefill), 2 decode steps."""
    import paper_2608_19889_gb300 as ax
    m = shape(name)
    B, S = 1, 80
    w = si.make_weights(m, device="cuda")
    model = create(m, w, max_batch=B, max_context=96, max_prefill_tokens=B * S, fp16=True)
    try:
        ids = si.make_ids(B, S, m["V"], seed=41)
        lg, nxt = run_prefill(model, ids, ax.AXON_LOGITS_LAST, m["V"])
        dl, fed = decode_steps(model, nxt, [S] * B, 2, m["V"])
        host = LazyF32({k: v.cpu() for k, v in w.items()})
        del w
        from oracle import decoder as od
        o = od.Oracle(od.DecoderConfig.from_dict(m), host, keep_f64=False)
        cache = o.new_contiguous_cache(B, 96)
        check(lg, o.prefill(ids, cache, last_only=True)[:, -1], what=f"{name} full-depth prefill")
        check(dl, oracle_decode(o, cache, fed, [S] * B), what=f"{name} full-depth decode")
    finally:
        ax.axon_free(model)
