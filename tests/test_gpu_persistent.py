"""The persistent decode step (one cooperative launch per step, B <= 8)
against the oracle and against the multi-kernel decode path on the same
model: tiny shapes with ragged vocabularies and K spans that leave ring stages
partly filled, both head dims, both 16-bit modes, contiguous and paged
caches, token counts from 1 to the maximum of 8."""
import os

import numpy as np
import pytest

import synth_inputs as si
from helpers import create, gpu_weights, oracle_for, tiny_tol
from test_gpu_parity import TINY, TINY128, _ax, check, decode_steps, oracle_decode, run_prefill

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_19889_gb300 import build
    build.build()


def _create(shape, w, persistent, **kw):
    """Model with the persistent decode step (the default) or with the launch
    chain (AXON_NO_PERSIST=1 at creation)."""
    old = os.environ.pop("AXON_NO_PERSIST", None)
    try:
        if not persistent:
            os.environ["AXON_NO_PERSIST"] = "1"
        return create(shape, w, **kw)
    finally:
        os.environ.pop("AXON_NO_PERSIST", None)
        if old is not None:
            os.environ["AXON_NO_PERSIST"] = old


def _kinds(m, B, ctx0, bt=None):
    """Profiler kinds of one decode step (which path ran)."""
    ax = _ax()
    tok = torch.zeros(B, dtype=torch.int32, device="cuda")
    ctx = torch.tensor(ctx0, dtype=torch.int32, device="cuda")
    nxt = torch.empty(B, dtype=torch.int32, device="cuda")
    rows = ax.axon_profile_decode_step(m, tok, ctx, block_table=bt, next_tokens=nxt)
    return {r["name"] for r in rows}


@pytest.mark.parametrize("prec", ["bf16", "fp16"])
@pytest.mark.parametrize("shape,B,S", [(TINY, 1, 40), (TINY, 5, 30), (TINY128, 8, 20), (TINY128, 3, 70)])
def test_persistent_decode_matches_oracle_and_multi_kernel_path(shape, B, S, prec):
    ax = _ax()
    w = gpu_weights(shape)
    fp16 = prec == "fp16"
    mp = _create(shape, w, True, max_batch=8, max_context=128, fp16=fp16)
    mk = _create(shape, w, False, max_batch=8, max_context=128, fp16=fp16)
    try:
        assert "decode_persistent" in _kinds(mp, B, [S] * B)
        assert "decode_persistent" not in _kinds(mk, B, [S] * B)
        ids = si.make_ids(B, S, shape["V"], seed=7)
        _, nxt = run_prefill(mp, ids, ax.AXON_LOGITS_LAST, shape["V"])
        _, nxt_k = run_prefill(mk, ids, ax.AXON_LOGITS_LAST, shape["V"])
        assert np.array_equal(nxt, nxt_k)
        n = 8
        dl, fed = decode_steps(mp, nxt, [S] * B, n, shape["V"])
        o = oracle_for(shape, w)
        cache = o.new_contiguous_cache(B, 128)
        o.prefill(ids, cache)
        ref = oracle_decode(o, cache, fed, [S] * B)
        check(dl, ref, tol=tiny_tol(prec), what=f"persistent decode B={B}")
        # the multi-kernel path on the same fed tokens
        ctx = torch.full((B,), S, dtype=torch.int32, device="cuda")
        outs = []
        for t in range(n):
            tok = torch.from_numpy(fed[:, t].astype(np.int32)).cuda()
            lg = torch.empty(B, shape["V"], device="cuda")
            nx = torch.empty(B, dtype=torch.int32, device="cuda")
            ax.axon_decode_step(mk, tok, ctx, logits=lg, next_tokens=nx)
            outs.append(lg.cpu().numpy())
        torch.cuda.synchronize()
        dk = np.stack(outs, 1)
        check(dk, ref, tol=tiny_tol(prec), what=f"multi-kernel decode B={B}")
        diff = float(np.max(np.abs(dl - dk)))
        print(f"persistent vs multi-kernel: max|dlogit| {diff:.3e}")
        assert diff <= tiny_tol(prec)
        assert ax.axon_check_device(mp)[0] == 0
        assert ax.axon_check_device(mk)[0] == 0
    finally:
        ax.axon_free(mp)
        ax.axon_free(mk)


@pytest.mark.parametrize("prec", ["bf16", "fp16"])
def test_persistent_decode_paged_cache(prec):
    """Paged cache with a shuffled block table, head_dim 128: the persistent
    step reads and writes the blocks the table names."""
    ax = _ax()
    shape = TINY128
    B, S, n_new, max_ctx = 6, 37, 6, 64
    num_blocks = 3 * B * (max_ctx // 16)
    w = gpu_weights(shape)
    bt_np = si.make_block_table([max_ctx] * B, 16, max_ctx // 16, num_blocks, seed=si.SEED_BLOCKS)
    m = _create(shape, w, True, max_batch=B, max_context=max_ctx, layout="paged", num_blocks=num_blocks,
                fp16=prec == "fp16")
    try:
        bt = torch.from_numpy(bt_np).cuda()
        assert "decode_persistent" in _kinds(m, B, [S] * B, bt)
        ids = si.make_ids(B, S, shape["V"], seed=13)
        lg, nxt = run_prefill(m, ids, ax.AXON_LOGITS_LAST, shape["V"], block_table=bt)
        o = oracle_for(shape, w)
        cache = o.new_paged_cache(num_blocks, 16, bt_np)
        check(lg, o.prefill(ids, cache, last_only=True)[:, -1], tol=tiny_tol(prec), what="paged prefill")
        dl, fed = decode_steps(m, nxt, [S] * B, n_new, shape["V"], block_table=bt)
        check(dl, oracle_decode(o, cache, fed, [S] * B), tol=tiny_tol(prec), what="persistent paged decode")
        assert ax.axon_check_device(m)[0] == 0
    finally:
        ax.axon_free(m)


@pytest.mark.parametrize("shape", [TINY, TINY128])
def test_persistent_decode_split_kv_long_context(shape):
    """A context of more than 64 key blocks: the persistent step splits each
    sequence's keys into items of 16 blocks (8 in the head_dim-128 small
    layout, one staged block per warp) and merges them across CTAs."""
    ax = _ax()
    B, S, max_ctx = 2, 1100, 1152  # 72 key blocks of capacity: 5 splits
    w = gpu_weights(shape)
    m = _create(shape, w, True, max_batch=B, max_context=max_ctx, max_prefill_tokens=B * S)
    try:
        assert "decode_persistent" in _kinds(m, B, [max_ctx - 2] * B)
        ids = si.make_ids(B, S, shape["V"], seed=17)
        _, nxt = run_prefill(m, ids, ax.AXON_LOGITS_LAST, shape["V"])
        dl, fed = decode_steps(m, nxt, [S] * B, 6, shape["V"])
        o = oracle_for(shape, w)
        cache = o.new_contiguous_cache(B, max_ctx)
        o.prefill(ids, cache, last_only=True)
        check(dl, oracle_decode(o, cache, fed, [S] * B), tol=tiny_tol("bf16"),
              what=f"persistent split-KV decode d={shape['d']}")
        assert ax.axon_check_device(m)[0] == 0
    finally:
        ax.axon_free(m)
