"""CPU checks of bench.py's accounting and of its reference-arm JSON line:
the algorithmic byte and FLOP counts on shapes small enough to count by hand
(dense and mixture-of-experts, against the checkpoint's own matrix shapes
and, for the expected number of routed experts, exact enumeration), the
DRAM-traffic record lookup (valid only for the CUDA sources it was taken
on), the peak and clock bookkeeping, and `--impl reference` on the 135M
workload."""
import json
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402

SHAPE = dict(L=2, D=64, H=4, G=2, d=16, F=96, V=100, bias=True)


def test_model_bytes_counts_every_linear_weight():
    lin, head = bench.model_bytes(SHAPE)
    per_layer = (4 + 2 * 2) * 16 * 64 + 64 * 4 * 16 + 2 * 96 * 64 + 64 * 96
    assert lin == 2 * per_layer
    assert head == 100 * 64


def test_decode_bytes_per_step_by_hand():
    # B = 2 sequences whose new tokens sit at positions 5 and 9
    lin, head = bench.model_bytes(SHAPE)
    kv_tok = 2 * 2 * 2 * 16 * 2          # L * (K, V) * G * d * bf16
    small = (2 * 2 + 1) * 64 * 4 + 2 * (4 + 2 * 2) * 16 * 4  # norm gains + qkv biases, fp32
    want = 2 * (lin + head) + small + (6 + 10) * kv_tok + 2 * kv_tok + 2 * 100 * 4
    assert bench.decode_bytes_per_step(SHAPE, 2, [5, 9]) == want


def test_prefill_flops_by_hand():
    lin, head = bench.model_bytes(SHAPE)
    B, S = 3, 7
    attn = 2 * B * 4 * 4 * 16 * S * (S + 1) / 2
    assert bench.prefill_flops(SHAPE, B, S) == 2 * B * S * lin + attn + 2 * B * head


def test_recorded_traffic_is_tied_to_the_sources(tmp_path, monkeypatch):
    prof = tmp_path / "profiles"
    prof.mkdir()
    sha = bench.kernel_source_sha()
    (prof / "dram_w_bf16.md").write_text(
        "text\n```\nsource_sha256: %s\ntraffic decode_persistent: 12345\ntraffic prefill_qkv: 77\n```\n" % sha)
    (prof / "dram_old_bf16.md").write_text("```\nsource_sha256: 0000\ntraffic decode_persistent: 1\n```\n")
    real_dirname = os.path.dirname

    def fake_dirname(p):
        if p == os.path.abspath(bench.__file__):
            return str(tmp_path)
        return real_dirname(p)

    monkeypatch.setattr(bench.os.path, "dirname", fake_dirname)
    # the sha is computed over the real sources: point it back at the repository
    monkeypatch.setattr(bench, "kernel_source_sha", lambda: sha)
    assert bench.recorded_traffic("w", "bf16", "decode_persistent") == 12345.0
    assert bench.recorded_traffic("w", "bf16", "prefill_qkv") == 77.0
    assert bench.recorded_traffic("w", "bf16", "decode_o") is None
    assert bench.recorded_traffic("old", "bf16", "decode_persistent") is None  # other sources
    assert bench.recorded_traffic("missing", "bf16", "decode_persistent") is None


def test_reference_arm_json_line():
    out = subprocess.run(
        [sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--steps", "1", "--warmup", "0",
         "--workload", "135m_b1_s16_n16"],
        capture_output=True, text=True, timeout=600, cwd=ROOT)
    assert out.returncode == 0, out.stderr[-2000:]
    line = json.loads(out.stdout.strip().splitlines()[-1])
    assert line["impl"] == "reference"
    assert line["metric"] == bench.METRIC
    assert line["unit"] == "tokens/s" and line["value"] > 0
    assert line["higher_is_better"] is True
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["value"] == line["value"]
    assert line["cpu_baseline"]["cores"] >= 1
    assert line["e2e"] == {"value": line["value"], "unit": "tokens/s", "h2d_bytes_per_step": 0,
                           "d2h_bytes_per_step": 0}
    assert line["config"]["workload"] == "135m_b1_s16_n16"


def test_chunk_plan_covers_every_token_once_within_the_budget():
    lens = [5, 3, 9, 2]
    calls = bench.plan_chunks(lens, 6)
    assert calls == [(0, [(0, 5), (0, 1)]), (1, [(1, 2), (0, 4)]), (2, [(4, 5), (0, 1)]), (3, [(1, 1)])]
    got = {}
    for first, chunks in calls:
        assert sum(n for _, n in chunks) <= 6
        for i, (past, n) in enumerate(chunks):
            b = first + i
            assert past == got.get(b, 0)  # each chunk continues where the last one stopped
            got[b] = past + n
    assert got == {0: 5, 1: 3, 2: 9, 3: 2}


def test_varlen_prefill_flops_by_hand():
    lin, head = bench.model_bytes(SHAPE)
    # one whole prompt of 7 tokens counts like prefill_flops with B = 1
    assert bench.varlen_prefill_flops(SHAPE, [[(0, 7)]]) == bench.prefill_flops(SHAPE, 1, 7)
    # 3 new tokens after 4 cached ones attend 5 + 6 + 7 keys; a 1-token chunk after 9 attends 10
    want = 2 * 4 * lin + 2 * 4 * 4 * 16 * (5 + 6 + 7 + 10) + 2 * 2 * head
    assert bench.varlen_prefill_flops(SHAPE, [[(4, 3), (9, 1)]]) == want


def test_sliding_window_counts_only_the_visible_keys():
    W = dict(SHAPE, window=3)
    lin, head = bench.model_bytes(SHAPE)
    kv_tok = 2 * 2 * 2 * 16 * 2
    # new tokens at positions 5 and 1: 3 and 2 keys visible
    assert bench.decode_bytes_per_step(W, 2, [5, 1]) - bench.decode_bytes_per_step(SHAPE, 2, [5, 1]) == \
        (3 + 2 - 6 - 2) * kv_tok
    # a 7-token prompt sees 1 + 2 + 3 + 3 + 3 + 3 + 3 keys
    assert bench.prefill_flops(W, 1, 7) == 2 * 7 * lin + 2 * 4 * 4 * 16 * 18 + 2 * head
    assert bench.varlen_prefill_flops(W, [[(4, 3)]]) == 2 * 3 * lin + 2 * 4 * 4 * 16 * 9 + 2 * head
    assert bench.keys_seen_by_run(4, 3, 0) == 5 + 6 + 7


# mixture of experts: the decode step's weight bytes and the prefill FLOPs
MOE_SHAPE = dict(L=3, D=32, H=4, G=2, d=8, F=48, V=64, tie=False, bias=False, n_experts=6, top_k=2, moe_F=16,
                 n_shared=2, first_dense=1)


def _matrices(shape):
    """Weight elements of every per-layer matrix, by its HF name."""
    import numpy as np
    import synth_inputs as si
    return {k: int(np.prod(v)) for k, v in si.weight_shapes(shape).items() if ".layers." in k and len(v) == 2}


@pytest.mark.parametrize("shape", [dict(SHAPE, tie=False), MOE_SHAPE])
def test_model_bytes_match_the_checkpoints_matrices(shape):
    """All experts counted (active None): the per-layer matrices of the
    checkpoint the library reads, counted from their shapes."""
    lin, head = bench.model_bytes(shape)
    assert lin == sum(_matrices(shape).values())
    assert head == shape["V"] * shape["D"]


def test_moe_model_bytes_with_some_experts_active():
    m = _matrices(MOE_SHAPE)
    one_expert = sum(v for k, v in m.items() if ".layers.1.mlp.experts.0." in k)
    lin_all, _ = bench.model_bytes(MOE_SHAPE)
    lin_3, _ = bench.model_bytes(MOE_SHAPE, active_experts=3)
    assert lin_all - lin_3 == 2 * (6 - 3) * one_expert  # two MoE layers, three experts fewer each


def test_expected_active_experts_against_enumeration():
    """E (1 - (1 - k/E)^T) against the exact mean over every assignment of
    T tokens to k-subsets of E experts (uniform, independent)."""
    import itertools
    E, k = 6, 2
    subsets = list(itertools.combinations(range(E), k))
    for T in (1, 2, 3):
        total = sum(len(set().union(*pick)) for pick in itertools.product(subsets, repeat=T))
        exact = total / len(subsets) ** T
        assert abs(bench.expected_active_experts(dict(n_experts=E, top_k=k), T) - exact) < 1e-12


def test_moe_linear_flops_per_token_by_hand():
    """Per token: every attention matrix, the dense layer's MLP, and in each
    MoE layer the router, the shared MLP and top_k experts, 2 FLOPs per
    weight element."""
    m = _matrices(MOE_SHAPE)
    per = sum(v for k, v in m.items() if ".experts." not in k)
    per += 2 * MOE_SHAPE["top_k"] * sum(v for k, v in m.items() if ".layers.1.mlp.experts.0." in k)
    assert bench.linear_flops_per_token(MOE_SHAPE) == 2 * per


def test_tensor_peak_takes_the_sustained_figure_for_long_phases():
    assert bench.tensor_peak(1900.0, 1700.0, 99.9) == (1900.0, "burst")
    assert bench.tensor_peak(1900.0, 1700.0, 100.0) == (1700.0, "sustained")
    assert bench.tensor_peak(1900.0, None, 5000.0) == (1900.0, "burst")


def test_clock_sampler_reads_median_clock_and_active_reasons():
    class FakeProc:
        def terminate(self):
            pass

        def communicate(self, timeout=None):
            rows = ["0, 2070, 2070, 900.1, 0x0, Not Active, Not Active, Not Active, Not Active",
                    "0, 1980, 2070, 1390.5, 0x4, Not Active, Not Active, Not Active, Active",
                    "0, 2070, 2070, 1200.0, 0x0, Not Active, Not Active, Not Active, Not Active",
                    "garbled line"]
            return "\n".join(rows) + "\n", ""

    s = bench.ClockSampler.__new__(bench.ClockSampler)
    s.p = FakeProc()
    c = s.stop()
    assert c == {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "reasons": ["sw_power_cap"], "samples": 3}


def test_default_precision_by_width():
    assert bench.default_precision("32b_b16_s2048_n256") == "fp16"
    assert bench.default_precision("8b_paged_b64_ctx512-4096_n128") == "fp16"
    assert bench.default_precision("0.5b_b1_s512_n128") == "bf16"
