"""Parity at the paper's 8B- and 32B-class widths: full-width layers with
few layers (prefill through the tensor-core GEMM at the configs' prompt
lengths, decode at batch 12/16 and the B=64 paged decode), and the
full-depth models with 100 teacher-forced decode tokens. Slow (the float64
oracle does the same work on the host).

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


def sampled_rows(S, n, seed):
    """n distinct positions of an S-token prompt, always including the first
    and the last."""
    rng = np.random.Generator(np.random.PCG64(seed))
    mid = rng.choice(np.arange(1, S - 1), size=n - 2, replace=False)
    return np.sort(np.concatenate([[0, S - 1], mid])).astype(np.int64)


def prefill_long_case(m, B, S, seed, n_rows, fp16=True, decode_n=3):
    """Prefill B x S at full width through the tensor-core path in ALL mode;
    the oracle recomputes the LAST logits of every sequence and a sample of
    n_rows positions per sequence; then decode_n greedy steps."""
    import paper_2608_19889_gb300 as ax
    max_ctx = (S + decode_n + 15) // 16 * 16
    w = si.make_weights(m, device="cuda")
    model = create(m, w, max_batch=B, max_context=max_ctx, max_prefill_tokens=B * S, fp16=fp16)
    try:
        ids = si.make_ids(B, S, m["V"], seed=seed)
        idt = torch.from_numpy(ids).cuda()
        lg = torch.empty(B, S, m["V"], device="cuda")
        nxt = torch.empty(B, dtype=torch.int32, device="cuda")
        ax.axon_prefill(model, idt, logits_mode=ax.AXON_LOGITS_ALL, logits=lg, next_tokens=nxt)
        rows = sampled_rows(S, n_rows, seed)
        got = lg[:, torch.from_numpy(rows).cuda()].cpu().numpy()
        del lg
        nxt = nxt.cpu().numpy()
        dl, fed = decode_steps(model, nxt, [S] * B, decode_n, m["V"])
        o = oracle_for(m, w)
        del w
        cache = o.new_contiguous_cache(B, max_ctx)
        ref = o.prefill(ids, cache, rows=rows)
        assert np.array_equal(nxt, got[:, -1].argmax(-1))
        return got, ref, dl, oracle_decode(o, cache, fed, [S] * B)
    finally:
        ax.axon_free(model)


def test_8b_width_prefill_batch8_s1024():
    """The 8B config's batched prefill shape: 8 x 1024 = 8192 rows through the
    tcgen05 GEMMs and the d=128 flash attention over 1024 keys, two layers;
    LAST logits and 8 sampled positions per sequence, then 3 decode steps."""
    m = shape("8b", L=2)
    got, ref, dl, refd = prefill_long_case(m, B=8, S=1024, seed=51, n_rows=8)
    check(got, ref, what="8b-width B=8 S=1024 prefill, sampled rows")
    check(got[:, -1], ref[:, -1], what="8b-width B=8 S=1024 prefill, last rows")
    check(dl, refd, what="8b-width B=8 decode after S=1024")


def test_32b_width_prefill_s2048():
    """The 32B config's prompt length: 2048 rows, one 32B-width layer with QKV
    biases; LAST logits and 16 sampled positions, then 3 decode steps."""
    m = shape("32b", L=1)
    got, ref, dl, refd = prefill_long_case(m, B=1, S=2048, seed=52, n_rows=16)
    check(got, ref, what="32b-width S=2048 prefill, sampled rows")
    check(dl, refd, what="32b-width decode after S=2048")


@pytest.mark.parametrize("name,B", [("8b", 12), ("32b", 16)])
def test_wide_decode_batch_9_to_32(name, B):
    """Decode with 9-32 sequences at full width, one layer: the launch chain
    with gate/up and the LM head on the tcgen05 GEMM, QKV, O and down on its
    split-K mode at up to 16 tokens (the plan the 32B batch-16 config decodes
    with)."""
    import paper_2608_19889_gb300 as ax
    m = shape(name, L=1)
    S, n = 48, 4
    w = si.make_weights(m, device="cuda")
    model = create(m, w, max_batch=B, max_context=64, max_prefill_tokens=B * S, fp16=True)
    try:
        ids = si.make_ids(B, S, m["V"], seed=61)
        lg, nxt = run_prefill(model, ids, ax.AXON_LOGITS_LAST, m["V"])
        tok = torch.zeros(B, dtype=torch.int32, device="cuda")
        ctx = torch.full((B,), S, dtype=torch.int32, device="cuda")
        kinds = {r["name"] for r in ax.axon_profile_decode_step(model, tok, ctx, next_tokens=tok.clone())}
        assert "decode_persistent" not in kinds and "decode_gateup" in kinds
        dl, fed = decode_steps(model, nxt, [S] * B, n, m["V"])
        o = oracle_for(m, w)
        del w
        cache = o.new_contiguous_cache(B, 64)
        check(lg, o.prefill(ids, cache, last_only=True)[:, -1], what=f"{name}-width B={B} prefill")
        check(dl, oracle_decode(o, cache, fed, [S] * B), what=f"{name}-width B={B} decode (launch chain)")
    finally:
        ax.axon_free(model)


def top1_report(gpu, ref, maxd):
    """Raw greedy agreement, and how many disagreements fall where the
    oracle's top-2 gap is within 2 max|delta| (near ties)."""
    g = np.asarray(gpu).argmax(-1)
    r = np.asarray(ref).argmax(-1)
    srt = np.sort(np.asarray(ref), axis=-1)
    gap = srt[..., -1] - srt[..., -2]
    flips = g != r
    return float(np.mean(~flips)), int(np.sum(flips & (gap <= 2 * maxd))), int(np.sum(flips & (gap > 2 * maxd)))


def decode_forced(model, fed, ctx0, V):
    """Decode steps that consume the given tokens fed[:, t] (teacher forcing
    on the GPU side too); returns the logits of every step [B, n, V]."""
    import paper_2608_19889_gb300 as ax
    B, n = fed.shape
    ctx = torch.from_numpy(np.asarray(ctx0, dtype=np.int32)).cuda()
    outs = []
    for t in range(n):
        tok = torch.from_numpy(fed[:, t].astype(np.int32)).cuda()
        lg = torch.empty(B, V, device="cuda")
        ax.axon_decode_step(model, tok, ctx, logits=lg, next_tokens=torch.empty_like(tok))
        outs.append(lg.cpu().numpy())
    return np.stack(outs, 1)


@pytest.mark.parametrize("name", ["8b", "32b"])
def test_full_depth_teacher_forced_100_tokens(name):
    """All layers at full width, B=1: a 64-token prompt and 100 greedy decode
    steps in fp16 operand mode; then the fp32 mode (the bf16 weights widened,
    fp32 activations and accumulation: the paper's fp32 fallback) consumes
    the same 100 tokens. Teacher-forced: the oracle reads those tokens in one
    pass over prompt + tokens (cached decode = full recompute, an oracle pin)
    and returns the logits of the 101 positions the GPU produced.

    fp16 mode: max|dlogit| <= 5e-2, and every greedy disagreement lies where
    the oracle's top-2 gap is within 2 max|dlogit| (a near tie). Its raw
    agreement is bounded by the 16-bit rounding of q, k, v, P, o and u
    (about 5e-4 rms each per pair of layers at 8B width, measured by
    emulating them in the float64 forward): at 32B full depth that leaves
    about 1e-2 rms logit noise against a median top-2 gap of ~0.3, i.e. a few
    percent of positions flip, so 95% is asserted and the count reported.
    fp32 mode: relative error <= 1e-4 and raw top-1 >= 99%."""
    import paper_2608_19889_gb300 as ax
    m = shape(name)
    B, S, n = 1, 64, 100
    w = si.make_weights(m, device="cuda")
    model = create(m, w, max_batch=B, max_context=176, max_prefill_tokens=B * S, fp16=True)
    try:
        ids = si.make_ids(B, S, m["V"], seed=41)
        lg, nxt = run_prefill(model, ids, ax.AXON_LOGITS_LAST, m["V"])
        dl, fed = decode_steps(model, nxt, [S] * B, n, m["V"])
    finally:
        ax.axon_free(model)
    g16 = np.concatenate([lg[:, None], dl], 1)  # [1, 101, V]
    model = create(m, w, max_batch=B, max_context=176, max_prefill_tokens=B * S, fp32=True)
    try:
        lg32, _ = run_prefill(model, ids, ax.AXON_LOGITS_LAST, m["V"])
        g32 = np.concatenate([lg32[:, None], decode_forced(model, fed, [S] * B, m["V"])], 1)
    finally:
        ax.axon_free(model)
    host = LazyF32({k: v.cpu() for k, v in w.items()})
    del w
    from oracle import decoder as od
    o = od.Oracle(od.DecoderConfig.from_dict(m), host, keep_f64=False)
    seq = np.concatenate([ids, fed], 1)  # the prompt, then the 100 fed tokens
    ref = o.prefill(seq, o.new_contiguous_cache(B, 176), rows=np.arange(S - 1, S + n))
    maxd = float(np.max(np.abs(g16 - ref)))
    raw, near_flips, hard_flips = top1_report(g16, ref, maxd)
    print(f"{name} full depth fp16, {n + 1} positions: max|dlogit| {maxd:.3e}  raw top-1 {raw:.4f}  "
          f"flips at near ties {near_flips}  other flips {hard_flips}")
    rel = float(np.max(np.abs(g32 - ref)) / np.max(np.abs(ref)))
    raw32, near32, hard32 = top1_report(g32, ref, float(np.max(np.abs(g32 - ref))))
    print(f"{name} full depth fp32, same tokens: relative error {rel:.3e}  raw top-1 {raw32:.4f}  "
          f"flips {near32 + hard32}")
    assert np.isfinite(g16).all() and np.isfinite(g32).all()
    assert maxd <= 5e-2
    assert hard_flips == 0
    assert raw >= 0.95
    assert rel <= 1e-4
    assert raw32 >= 0.99
