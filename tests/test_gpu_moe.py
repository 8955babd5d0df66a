"""GPU parity of the mixture-of-experts decoder (routing, the stable sort
into expert segments, the grouped tcgen05 expert GEMMs, the combine, shared
experts, leading dense layers) against the oracle, through the C ABI.

The routing is a discrete decision taken from 16-bit activations on the GPU
and from float64 ones in the oracle, so a near tie between the k-th and the
next expert may legitimately go either way. The test therefore (1) records
the GPU's expert choices (axon_moe_routing_record), (2) checks that every
choice is a valid top-k under the oracle's own router probabilities -- k
distinct experts, none of the others more probable than the least probable
chosen one by more than a small band -- and (3) compares the logits with
the oracle run on those same choices (teacher-forced routing)."""
import numpy as np
import pytest

import synth_inputs as si
from helpers import create, gpu_weights, oracle_for, tiny_tol
from oracle import decoder as od
from test_gpu_parity import _ax, check, run_prefill

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

# three layers, the first dense; 8 experts, 2 per token, one shared expert
MOE = dict(L=3, D=256, H=4, G=2, d=64, F=384, V=1000, tie=False, bias=False, theta=1e4, eps=1e-5,
           n_experts=8, top_k=2, moe_F=128, n_shared=1, first_dense=1, norm_topk=False)
# 16 experts, 4 per token, renormalised weights, no shared expert (the
# combine is the layer's residual producer)
MOE2 = dict(MOE, n_experts=16, top_k=4, moe_F=192, n_shared=0, norm_topk=True, bias=True)
BAND = 1e-2  # probability band for a valid top-k choice


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_19889_gb300 import build
    build.build()


def _moe_layers(shape):
    return [l for l in range(shape["L"]) if l >= shape["first_dense"]]


def _check_routing(o, chosen, shape, what):
    """chosen[l] [rows, k]: valid top-k under the oracle's probabilities of
    its last (forced) pass; returns how many rows differ from its own top-k."""
    differ = 0
    k = shape["top_k"]
    for l in _moe_layers(shape):
        _, _, prob = o.last_routing[f"model.layers.{l}."]
        c = chosen[l]
        assert c.shape == prob.shape[:1] + (k,)
        for t in range(c.shape[0]):
            sel = [int(e) for e in c[t]]
            assert len(set(sel)) == k and min(sel) >= 0 and max(sel) < shape["n_experts"], (what, l, t, sel)
            rest = np.delete(prob[t], sel)
            assert rest.max() <= prob[t][sel].min() + BAND, (what, l, t, sel, prob[t])
            differ += set(sel) != set(od.topk_lowest(prob[t], k).tolist())
    return differ


@pytest.mark.parametrize("shape,prec", [(MOE, "bf16"), (MOE, "fp16"), (MOE2, "fp16")])
def test_moe_decoder_prefill_and_decode_teacher_forced_routing(shape, prec):
    ax = _ax()
    B, S, steps = 2, 72, 4  # 144 prefill rows: the dense projections on the tcgen05 GEMM
    L, k, V = shape["L"], shape["top_k"], shape["V"]
    w = gpu_weights(shape)
    m = create(shape, w, max_batch=B, max_context=96, fp16=prec == "fp16")
    try:
        rec = torch.full((L, B * S, k), -1, dtype=torch.int32, device="cuda")
        ax.axon_moe_routing_record(m, rec, B * S)
        ids = si.make_ids(B, S, V, seed=43)
        lg, nxt = run_prefill(m, ids, ax.AXON_LOGITS_ALL, V)
        route = rec.cpu().numpy()
        assert (route[0] == -1).all()  # the dense first layer records nothing
        o = oracle_for(shape, w)
        o.forced_routing = {l: route[l] for l in _moe_layers(shape)}
        cache = o.new_contiguous_cache(B, 96)
        ref = o.prefill(ids, cache)
        differ = _check_routing(o, route, shape, "prefill")
        print(f"moe prefill: {differ} of {B * S * len(_moe_layers(shape))} token-layers routed differently "
              f"from the oracle's own top-{k} (near ties)")
        check(lg, ref, tol=tiny_tol(prec), what=f"moe prefill ({prec}, E={shape['n_experts']})")
        assert np.array_equal(nxt, lg[:, -1].argmax(-1))

        rec_d = torch.full((L, B, k), -1, dtype=torch.int32, device="cuda")
        ax.axon_moe_routing_record(m, rec_d, B)
        tok = torch.from_numpy(nxt.astype(np.int32)).cuda()
        ctx = torch.full((B,), S, dtype=torch.int32, device="cuda")
        lens = np.full(B, S)
        outs, refs = [], []
        for _ in range(steps):
            fed = tok.cpu().numpy()
            logits = torch.empty(B, V, device="cuda")
            nx = torch.empty(B, dtype=torch.int32, device="cuda")
            ax.axon_decode_step(m, tok, ctx, logits=logits, next_tokens=nx)
            torch.cuda.synchronize()
            rd = rec_d.cpu().numpy()
            o.forced_routing = {l: rd[l] for l in _moe_layers(shape)}
            refs.append(o.decode_step(fed, cache, lens))
            _check_routing(o, rd, shape, "decode")
            outs.append(logits.cpu().numpy())
            assert np.array_equal(nx.cpu().numpy(), outs[-1].argmax(-1))
            lens = lens + 1
            tok = nx
        check(np.stack(outs, 1), np.stack(refs, 1), tol=tiny_tol(prec), what=f"moe decode ({prec})")
        kinds = {r["name"] for r in ax.axon_profile_decode_step(m, tok, ctx, next_tokens=tok.clone())}
        assert {"decode_moe_route", "decode_moe_gateup", "decode_moe_down", "decode_moe_combine"} <= kinds
        assert ax.axon_check_device(m)[0] == 0
    finally:
        ax.axon_free(m)
