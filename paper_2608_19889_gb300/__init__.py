"""GB300 (sm_103a) Llama-family decoder forward behind a C ABI.

This module is the thin Python binding of `libaxon_gb300.so` (see
`include/axon.h`): functions with the C names that marshal torch tensors
into pointers and raise on a non-zero status. Every step of the forward pass
runs in the library's CUDA kernels; torch only provides device memory and
streams. There is no CPU fallback: if the library was not built, the first
call raises.
"""
from __future__ import annotations

import ctypes
import os

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libaxon_gb300.so")

AXON_OK = 0
AXON_ERR_INVALID_ARG = 1
AXON_ERR_SHAPE_MISMATCH = 2
AXON_ERR_MISSING_WEIGHT = 3
AXON_ERR_UNSUPPORTED = 4
AXON_ERR_OOM = 5
AXON_ERR_CUDA = 6
AXON_ERR_TIMEOUT = 7
AXON_ERR_DEVICE_CHECK = 8
AXON_KV_CONTIGUOUS, AXON_KV_PAGED = 0, 1
AXON_BF16, AXON_FP32_DEBUG, AXON_FP16 = 0, 1, 2
AXON_DTYPE_BF16, AXON_DTYPE_F32 = 0, 1
AXON_LOGITS_LAST, AXON_LOGITS_ALL = 0, 1
AXON_ACT_SILU, AXON_ACT_GELU_TANH = 0, 1

EXPORTED = ["axon_model_create", "axon_prefill", "axon_prefill_varlen", "axon_decode_step", "axon_reset",
            "axon_check_device", "axon_kv_view_get", "axon_profile_decode_step", "axon_profile_prefill",
            "axon_decode_step_noalloc", "axon_moe_routing_record", "axon_free", "axon_status_string"]


class axon_config(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in (
        "num_hidden_layers", "hidden_size", "num_attention_heads", "num_key_value_heads", "head_dim",
        "intermediate_size", "vocab_size", "tie_word_embeddings", "attention_bias")] + [
        ("rope_theta", ctypes.c_float), ("rms_norm_eps", ctypes.c_float)] + [
        (n, ctypes.c_int32) for n in ("max_batch", "max_context", "max_prefill_tokens", "kv_layout",
                                      "kv_block_size", "kv_num_blocks", "precision", "sliding_window")] + [
        (n, ctypes.c_float) for n in ("rope_scaling_factor", "rope_low_freq_factor", "rope_high_freq_factor")] + [
        ("rope_original_max_position", ctypes.c_int32), ("hidden_act", ctypes.c_int32), ("qk_norm", ctypes.c_int32)] + [
        (n, ctypes.c_int32) for n in ("n_routed_experts", "num_experts_per_tok", "moe_intermediate_size",
                                      "n_shared_experts", "first_k_dense_replace", "norm_topk_prob")]


class axon_tensor(ctypes.Structure):
    _fields_ = [("name", ctypes.c_char_p), ("data", ctypes.c_void_p), ("dtype", ctypes.c_int32),
                ("ndim", ctypes.c_int32), ("shape", ctypes.c_int64 * 4)]


class axon_kv_view(ctypes.Structure):
    _fields_ = [("k_pool", ctypes.c_void_p), ("v_pool", ctypes.c_void_p), ("num_blocks", ctypes.c_int64),
                ("blocks_per_seq", ctypes.c_int32), ("block_size", ctypes.c_int32), ("elem_bytes", ctypes.c_int32)]


class axon_kernel_time(ctypes.Structure):
    _fields_ = [("name", ctypes.c_char * 32), ("launches", ctypes.c_int32), ("total_ms", ctypes.c_float),
                ("bytes", ctypes.c_double), ("flops", ctypes.c_double)]


class AxonError(RuntimeError):
    def __init__(self, fn, status):
        self.status = status
        super().__init__(f"{fn} failed: {status} ({axon_status_string(status)})")


_lib = None


def lib() -> ctypes.CDLL:
    """Load the CUDA library (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with paper_2608_19889_gb300.build.build()")
        L = ctypes.CDLL(LIB_PATH)
        vp, i32, p_i32 = ctypes.c_void_p, ctypes.c_int32, ctypes.POINTER(ctypes.c_int32)
        L.axon_model_create.argtypes = [ctypes.POINTER(axon_config), ctypes.POINTER(axon_tensor), i32, vp,
                                        ctypes.POINTER(vp)]
        L.axon_prefill.argtypes = [vp, vp, i32, i32, vp, i32, vp, vp, vp]
        L.axon_prefill_varlen.argtypes = [vp, vp, i32, i32, vp, vp, i32, vp, i32, vp, vp, vp]
        L.axon_decode_step.argtypes = [vp, vp, i32, vp, vp, vp, vp, vp]
        L.axon_decode_step_noalloc.argtypes = [vp, vp, i32, vp, vp, vp, vp, vp]
        L.axon_moe_routing_record.argtypes = [vp, vp, i32]
        L.axon_reset.argtypes = [vp]
        L.axon_check_device.argtypes = [vp, vp, p_i32]
        L.axon_kv_view_get.argtypes = [vp, ctypes.POINTER(axon_kv_view)]
        L.axon_profile_decode_step.argtypes = [vp, vp, i32, vp, vp, vp, vp, ctypes.POINTER(axon_kernel_time), i32,
                                               p_i32]
        L.axon_profile_prefill.argtypes = [vp, vp, i32, i32, vp, vp, vp, ctypes.POINTER(axon_kernel_time), i32, p_i32]
        L.axon_free.argtypes = [vp]
        L.axon_free.restype = None
        L.axon_status_string.argtypes = [ctypes.c_int]
        L.axon_status_string.restype = ctypes.c_char_p
        for n in ("axon_model_create", "axon_prefill", "axon_prefill_varlen", "axon_decode_step", "axon_reset",
                  "axon_check_device", "axon_kv_view_get", "axon_profile_decode_step", "axon_profile_prefill",
                  "axon_decode_step_noalloc", "axon_moe_routing_record"):
            getattr(L, n).restype = ctypes.c_int
        _lib = L
    return _lib


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        import torch
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream))


def _check(fn, rc):
    if rc != AXON_OK:
        raise AxonError(fn, rc)


def axon_status_string(status: int) -> str:
    return lib().axon_status_string(status).decode()


def make_config(m: dict, max_batch: int, max_context: int, kv_layout=AXON_KV_CONTIGUOUS, kv_num_blocks=0,
                precision=AXON_BF16, max_prefill_tokens=0) -> axon_config:
    """axon_config from a shape dict with keys L, D, H, G, d, F, V, tie, bias, theta, eps (and optionally
    window, the sliding window, rope_factor / rope_low / rope_high / rope_orig, the RoPE frequency
    scaling, 0 or absent = none; act, "silu" (default) or "gelu_tanh"; qk_norm, per-head RMSNorm of q and k;
    n_experts, top_k, moe_F, n_shared, first_dense, norm_topk: the mixture-of-experts MLP)."""
    return axon_config(m["L"], m["D"], m["H"], m["G"], m["d"], m["F"], m["V"], int(m["tie"]), int(m["bias"]),
                       float(m["theta"]), float(m["eps"]), max_batch, max_context, max_prefill_tokens, kv_layout, 16,
                       kv_num_blocks, precision, int(m.get("window", 0)), float(m.get("rope_factor", 0.0)),
                       float(m.get("rope_low", 1.0)), float(m.get("rope_high", 4.0)), int(m.get("rope_orig", 8192)),
                       AXON_ACT_GELU_TANH if m.get("act", "silu") == "gelu_tanh" else AXON_ACT_SILU,
                       int(bool(m.get("qk_norm", False))), int(m.get("n_experts", 0)), int(m.get("top_k", 0)),
                       int(m.get("moe_F", 0)), int(m.get("n_shared", 0)), int(m.get("first_dense", 0)),
                       int(bool(m.get("norm_topk", False))))


def axon_model_create(cfg: axon_config, weights: dict, stream=None) -> ctypes.c_void_p:
    """Create a model from {HF name: torch tensor (bf16 or fp32, host or device)}."""
    import torch
    names = list(weights.keys())
    arr = (axon_tensor * len(names))()
    keep = []
    for i, n in enumerate(names):
        t = weights[n].contiguous()
        keep.append(t)
        if t.dtype == torch.bfloat16:
            dt = AXON_DTYPE_BF16
        elif t.dtype == torch.float32:
            dt = AXON_DTYPE_F32
        else:
            raise TypeError(f"{n}: unsupported dtype {t.dtype}")
        shape = (ctypes.c_int64 * 4)(*(list(t.shape) + [0] * (4 - t.dim())))
        arr[i] = axon_tensor(n.encode(), t.data_ptr(), dt, t.dim(), shape)
    h = ctypes.c_void_p()
    _check("axon_model_create", lib().axon_model_create(ctypes.byref(cfg), arr, len(names), _stream(stream),
                                                        ctypes.byref(h)))
    return h


def axon_prefill(m, ids, block_table=None, logits_mode=AXON_LOGITS_LAST, logits=None, next_tokens=None,
                 stream=None):
    """ids: int32 [B, S] on the device; outputs written into the given tensors."""
    B, S = ids.shape
    _check("axon_prefill", lib().axon_prefill(m, _ptr(ids), B, S, _ptr(block_table), logits_mode, _ptr(logits),
                                              _ptr(next_tokens), _stream(stream)))


def axon_prefill_varlen(m, ids, cu_seqlens, context_lens, max_chunk, block_table=None, logits_mode=AXON_LOGITS_LAST,
                        logits=None, next_tokens=None, stream=None):
    """ids: int32 [T] packed chunks; cu_seqlens: int32 [B+1] row offsets;
    context_lens: int32 [B] tokens cached before each chunk (advanced by the
    chunk lengths); max_chunk: host bound on the longest chunk. All device
    tensors; outputs written into the given tensors."""
    T = ids.shape[0]
    B = cu_seqlens.shape[0] - 1
    _check("axon_prefill_varlen", lib().axon_prefill_varlen(
        m, _ptr(ids), B, T, _ptr(cu_seqlens), _ptr(context_lens), int(max_chunk), _ptr(block_table), logits_mode,
        _ptr(logits), _ptr(next_tokens), _stream(stream)))


def axon_decode_step(m, tokens, context_lens, block_table=None, logits=None, next_tokens=None, stream=None):
    """tokens, context_lens: int32 [B] on the device (context_lens advances by one)."""
    B = tokens.shape[0]
    _check("axon_decode_step", lib().axon_decode_step(m, _ptr(tokens), B, _ptr(context_lens), _ptr(block_table),
                                                      _ptr(logits), _ptr(next_tokens), _stream(stream)))


def axon_moe_routing_record(m, experts=None, rows=0):
    """experts: int32 device tensor [L, rows, k] that later passes fill with
    each MoE layer's chosen experts (see include/axon.h), or None to stop."""
    _check("axon_moe_routing_record", lib().axon_moe_routing_record(m, _ptr(experts), int(rows)))


def axon_decode_step_noalloc(m, tokens, context_lens, block_table=None, logits=None, next_tokens=None, stream=None):
    """Allocation-free decode step (see include/axon.h): same contract as
    axon_decode_step, direct launches, fixed library-owned merge scratch."""
    B = tokens.shape[0]
    _check("axon_decode_step_noalloc", lib().axon_decode_step_noalloc(
        m, _ptr(tokens), B, _ptr(context_lens), _ptr(block_table), _ptr(logits), _ptr(next_tokens), _stream(stream)))


def axon_reset(m):
    _check("axon_reset", lib().axon_reset(m))


def axon_check_device(m, stream=None) -> tuple[int, int]:
    """(status, raw error bits) after synchronising the stream."""
    bits = ctypes.c_int32(0)
    rc = lib().axon_check_device(m, _stream(stream), ctypes.byref(bits))
    return rc, bits.value


def axon_kv_view_get(m) -> axon_kv_view:
    v = axon_kv_view()
    _check("axon_kv_view_get", lib().axon_kv_view_get(m, ctypes.byref(v)))
    return v


def _profile_result(arr, n):
    return [dict(name=arr[i].name.decode(), launches=arr[i].launches, total_ms=arr[i].total_ms,
                 bytes=arr[i].bytes, flops=arr[i].flops) for i in range(n.value)]


def axon_profile_decode_step(m, tokens, context_lens, block_table=None, next_tokens=None, stream=None):
    """Per-kernel-kind timing of one decode step (runs the step)."""
    arr = (axon_kernel_time * 16)()
    n = ctypes.c_int32(0)
    B = tokens.shape[0]
    _check("axon_profile_decode_step", lib().axon_profile_decode_step(
        m, _ptr(tokens), B, _ptr(context_lens), _ptr(block_table), _ptr(next_tokens), _stream(stream), arr, 16,
        ctypes.byref(n)))
    return _profile_result(arr, n)


def axon_profile_prefill(m, ids, block_table=None, next_tokens=None, stream=None):
    """Per-kernel-kind timing of one prefill (LAST-position logits not stored)."""
    arr = (axon_kernel_time * 16)()
    n = ctypes.c_int32(0)
    B, S = ids.shape
    _check("axon_profile_prefill", lib().axon_profile_prefill(
        m, _ptr(ids), B, S, _ptr(block_table), _ptr(next_tokens), _stream(stream), arr, 16, ctypes.byref(n)))
    return _profile_result(arr, n)


def axon_free(m):
    lib().axon_free(m)
