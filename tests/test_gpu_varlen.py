"""GPU parity of the variable-length batch (axon_prefill_varlen) against the
oracle's forward_varlen: sequences of different lengths, each appending one
chunk after its own cached tokens (whole prompts, further pieces of a prompt
and single decode tokens mixed in one call), on contiguous and shuffled paged
caches, followed by a regular decode step on the advanced context lengths."""
import numpy as np
import pytest

import synth_inputs as si
from helpers import FP32_REL_TOL, LOGIT_TOL, create, gpu_weights, oracle_for, parity

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

TINY = dict(L=2, D=128, H=4, G=2, d=64, F=192, V=1000, tie=False, bias=True, theta=1e4, eps=1e-5)
TINY128 = dict(L=2, D=256, H=6, G=2, d=128, F=320, V=777, tie=True, bias=False, theta=5e5, eps=1e-6)


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_19889_gb300 import build
    build.build()


def _ax():
    import paper_2608_19889_gb300 as ax
    return ax


def _check(gpu, ref, what, fp32=False):
    gpu = np.asarray(gpu, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert np.isfinite(gpu).all(), f"{what}: non-finite logits"
    if fp32:
        rel = float(np.max(np.abs(gpu - ref)) / np.max(np.abs(ref)))
        print(f"{what}: fp32 relative error {rel:.3e}")
        assert rel <= FP32_REL_TOL
        return
    maxd, agree, hard = parity(gpu, ref)
    print(f"{what}: max|dlogit| {maxd:.3e}  top1 {agree:.4f}  hard mismatches {hard}")
    assert maxd <= LOGIT_TOL, f"{what}: max|dlogit| {maxd} > {LOGIT_TOL}"
    assert hard == 0


def _chunks(lengths, V, seed):
    return [si.make_ids(1, int(n), V, seed=seed + 100 * i)[0] for i, n in enumerate(lengths)]


def _run_varlen(m, chunks, ctx, mode, V, block_table=None):
    """One axon_prefill_varlen call; returns (logits, next, ctx after)."""
    ax = _ax()
    ids = torch.from_numpy(np.concatenate(chunks).astype(np.int32)).cuda()
    cu_np = np.concatenate([[0], np.cumsum([len(c) for c in chunks])]).astype(np.int32)
    cu = torch.from_numpy(cu_np).cuda()
    B, T = len(chunks), int(cu_np[-1])
    logits = torch.full((T, V) if mode == ax.AXON_LOGITS_ALL else (B, V), float("nan"), device="cuda")
    nxt = torch.full((B,), -1, dtype=torch.int32, device="cuda")
    ax.axon_prefill_varlen(m, ids, cu, ctx, max(len(c) for c in chunks), block_table=block_table,
                           logits_mode=mode, logits=logits, next_tokens=nxt)
    torch.cuda.synchronize()
    return logits.cpu().numpy(), nxt.cpu().numpy(), cu_np


def _case(shape, layout, prec, first, second, max_ctx=256):
    """first: chunk lengths of a call from an empty cache (LAST logits);
    second: the next chunk of every sequence (ALL logits); then one decode
    step with axon_decode_step on the context lengths the calls advanced."""
    ax = _ax()
    B = len(first)
    V = shape["V"]
    w = gpu_weights(shape)
    bt_np, bt, nb = None, None, 0
    if layout == "paged":
        nb = B * (max_ctx // 16) + 7
        bt_np = si.make_block_table([max_ctx] * B, 16, max_ctx // 16, nb, seed=si.SEED_BLOCKS)
        bt = torch.from_numpy(bt_np).cuda()
    T_max = max(sum(first), sum(second))
    m = create(shape, w, max_batch=B, max_context=max_ctx, layout=layout, num_blocks=nb,
               fp32=prec == "fp32", fp16=prec == "fp16", max_prefill_tokens=T_max)
    fp32 = prec == "fp32"
    try:
        o = oracle_for(shape, w)
        cache = o.new_paged_cache(nb, 16, bt_np) if layout == "paged" else o.new_contiguous_cache(B, max_ctx)
        ctx = torch.zeros(B, dtype=torch.int32, device="cuda")
        past = np.zeros(B, dtype=np.int64)

        c1 = _chunks(first, V, seed=21)
        lg, nxt, _ = _run_varlen(m, c1, ctx, ax.AXON_LOGITS_LAST, V, bt)
        ref = np.stack(o.forward_varlen(c1, cache, past, last_only=True))
        _check(lg, ref, f"varlen {layout} {prec} first chunks {first}", fp32)
        assert np.array_equal(nxt, lg.argmax(-1))
        past += np.asarray(first)
        assert np.array_equal(ctx.cpu().numpy(), past)

        c2 = _chunks(second, V, seed=57)
        lg2, nxt2, cu2 = _run_varlen(m, c2, ctx, ax.AXON_LOGITS_ALL, V, bt)
        ref2 = np.concatenate(o.forward_varlen(c2, cache, past, last_only=False))
        _check(lg2, ref2, f"varlen {layout} {prec} next chunks {second} (all rows)", fp32)
        assert np.array_equal(nxt2, lg2[cu2[1:] - 1].argmax(-1))
        past += np.asarray(second)
        assert np.array_equal(ctx.cpu().numpy(), past)

        tok = torch.from_numpy(nxt2).cuda()
        dl = torch.full((B, V), float("nan"), device="cuda")
        dn = torch.empty(B, dtype=torch.int32, device="cuda")
        ax.axon_decode_step(m, tok, ctx, block_table=bt, logits=dl, next_tokens=dn)
        torch.cuda.synchronize()
        refd = o.decode_step(nxt2, cache, past)
        _check(dl.cpu().numpy(), refd, f"decode after varlen {layout} {prec}", fp32)
        assert ax.axon_check_device(m)[0] == 0
    finally:
        ax.axon_free(m)


@pytest.mark.parametrize("prec", ["bf16", "fp16"])
@pytest.mark.parametrize("layout", ["contiguous", "paged"])
def test_varlen_tensor_core_then_gemv_rows(layout, prec):
    """First call 113 rows (tcgen05 GEMM, ragged 128-row tail), lengths
    crossing 16-token blocks and a 1-token prompt; second call 41 rows
    (decode GEMV) mixing prompt pieces with single decode tokens."""
    _case(TINY, layout, prec, first=[37, 5, 70, 1], second=[20, 1, 3, 17])


@pytest.mark.parametrize("layout", ["contiguous", "paged"])
def test_varlen_head_dim_128(layout):
    _case(TINY128, layout, "bf16", first=[96, 33, 2], second=[1, 40, 64])


def test_varlen_fp32_debug_mode():
    _case(TINY, "contiguous", "fp32", first=[37, 5, 70, 1], second=[20, 1, 3, 17])


def test_varlen_chunked_prompt_matches_whole_prompt_prefill():
    """A 150-token prompt through three varlen calls of one sequence (64, 50,
    36 tokens) gives the same last-position logits as axon_prefill of the
    whole prompt, and both match the oracle."""
    ax = _ax()
    shape, V = TINY, TINY["V"]
    w = gpu_weights(shape)
    ids = si.make_ids(1, 150, V, seed=77)
    m = create(shape, w, max_batch=1, max_context=160, max_prefill_tokens=150)
    try:
        whole = torch.full((1, V), float("nan"), device="cuda")
        ax.axon_prefill(m, torch.from_numpy(ids.astype(np.int32)).cuda(), logits=whole)
        ctx = torch.zeros(1, dtype=torch.int32, device="cuda")
        lg = None
        for a, b in [(0, 64), (64, 114), (114, 150)]:
            lg, _, _ = _run_varlen(m, [ids[0, a:b]], ctx, ax.AXON_LOGITS_LAST, V)
        assert int(ctx.item()) == 150
        o = oracle_for(shape, w)
        ref = o.prefill(ids, o.new_contiguous_cache(1, 160), last_only=True)[:, -1]
        _check(lg, ref, "chunked 64+50+36 vs oracle")
        _check(whole.cpu().numpy(), ref, "whole prompt vs oracle")
        assert np.max(np.abs(lg - whole.cpu().numpy())) <= LOGIT_TOL
    finally:
        ax.axon_free(m)


def test_varlen_more_than_64_sequences_last_rows():
    """70 sequences of 1-3 tokens: the LM head runs over the gathered last
    rows in groups of at most 64."""
    ax = _ax()
    shape, V = TINY, TINY["V"]
    rng = np.random.default_rng(5)
    lens = rng.integers(1, 4, size=70)
    w = gpu_weights(shape)
    m = create(shape, w, max_batch=70, max_context=32, max_prefill_tokens=int(lens.sum()))
    try:
        ch = _chunks(lens, V, seed=91)
        ctx = torch.zeros(70, dtype=torch.int32, device="cuda")
        lg, nxt, _ = _run_varlen(m, ch, ctx, ax.AXON_LOGITS_LAST, V)
        o = oracle_for(shape, w)
        ref = np.stack(o.forward_varlen(ch, o.new_contiguous_cache(70, 32), np.zeros(70), last_only=True))
        _check(lg, ref, "70 sequences, last rows")
        assert np.array_equal(nxt, lg.argmax(-1))
        assert np.array_equal(ctx.cpu().numpy(), lens)
    finally:
        ax.axon_free(m)


def test_varlen_inconsistent_offsets_are_reported():
    """Row offsets that end before T and a chunk longer than max_chunk: the
    device check reports them (every access of the affected rows is skipped
    by the kernels' own range checks), and a following valid call is clean."""
    ax = _ax()
    shape, V = TINY, TINY["V"]
    w = gpu_weights(shape)
    m = create(shape, w, max_batch=2, max_context=64, max_prefill_tokens=16)
    try:
        ids = torch.from_numpy(si.make_ids(1, 10, V, seed=3)[0].astype(np.int32)).cuda()
        ctx = torch.zeros(2, dtype=torch.int32, device="cuda")
        cu = torch.tensor([0, 5, 9], dtype=torch.int32, device="cuda")  # row 9 belongs to no sequence
        ax.axon_prefill_varlen(m, ids, cu, ctx, 5)
        rc, bits = ax.axon_check_device(m)
        assert rc == ax.AXON_ERR_DEVICE_CHECK and bits & 16
        ctx.zero_()
        cu = torch.tensor([0, 7, 10], dtype=torch.int32, device="cuda")  # first chunk 7 > max_chunk 5
        ax.axon_prefill_varlen(m, ids, cu, ctx, 5)
        rc, bits = ax.axon_check_device(m)
        assert rc == ax.AXON_ERR_DEVICE_CHECK and bits & 16
        with pytest.raises(ax.AxonError):  # host-side: T < B
            ax.axon_prefill_varlen(m, ids[:1], cu, ctx, 1)
        ax.axon_reset(m)
        ctx.zero_()
        cu = torch.tensor([0, 5, 10], dtype=torch.int32, device="cuda")
        ax.axon_prefill_varlen(m, ids, cu, ctx, 5)
        assert ax.axon_check_device(m)[0] == 0
    finally:
        ax.axon_free(m)
