"""CPU-side checks of the C ABI: the library loads without a GPU and exports
every function include/axon.h declares; the binding's structs match the
header's field order."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_functions():
    src = open(os.path.join(ROOT, "include", "axon.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:int|void|const char\*)\s+(axon_\w+)\s*\(", src, flags=re.M)))


@pytest.fixture(scope="module")
def built():
    from paper_2608_19889_gb300 import build
    build.build()
    import paper_2608_19889_gb300 as ax
    return ax


def test_header_declares_the_boundary():
    fns = declared_functions()
    for f in ("axon_model_create", "axon_prefill", "axon_decode_step", "axon_free"):
        assert f in fns


def test_library_exports_every_declared_symbol(built):
    lib = built.lib()
    for f in declared_functions():
        assert hasattr(lib, f), f"missing export {f}"
    assert sorted(built.EXPORTED) == declared_functions()


def test_status_strings_without_gpu(built):
    assert built.axon_status_string(0) == "ok"
    assert "argument" in built.axon_status_string(built.AXON_ERR_INVALID_ARG)
    assert built.axon_status_string(12345) == "unknown status"


def test_null_arguments_are_rejected_without_touching_the_device(built):
    lib = built.lib()
    out = ctypes.c_void_p()
    assert lib.axon_model_create(None, None, 0, None, ctypes.byref(out)) == built.AXON_ERR_INVALID_ARG
    assert lib.axon_prefill(None, None, 1, 1, None, 0, None, None, None) == built.AXON_ERR_INVALID_ARG
    assert lib.axon_decode_step(None, None, 1, None, None, None, None, None) == built.AXON_ERR_INVALID_ARG
    assert lib.axon_prefill_varlen(None, None, 1, 1, None, None, 1, None, 0, None, None, None) == \
        built.AXON_ERR_INVALID_ARG
    lib.axon_free(None)


def test_config_struct_layout_matches_header():
    import paper_2608_19889_gb300 as ax
    src = open(os.path.join(ROOT, "include", "axon.h")).read()
    body = src[src.index("typedef struct axon_config {"):src.index("} axon_config;")]
    names = re.findall(r"(\w+);", re.sub(r"/\*.*?\*/", "", body, flags=re.S))
    # fields declared several per line: expand "int32_t a, b, c;"
    fields = []
    for decl in re.sub(r"/\*.*?\*/", "", body, flags=re.S).split(";")[:-1]:
        decl = decl.replace("typedef struct axon_config {", "")
        parts = decl.split()
        if not parts:
            continue
        fields += [p.strip(",") for p in " ".join(parts[1:]).split(",")]
    assert [f[0] for f in ax.axon_config._fields_] == [f.strip() for f in fields]
    assert names


def test_invalid_configs_are_rejected_before_any_device_work(built):
    """axon_model_create validates the config on the host before its first
    CUDA call, so every rejection below runs without a GPU."""
    import ctypes as C
    ax = built
    shape = dict(L=1, D=128, H=4, G=2, d=64, F=192, V=100, tie=True, bias=False, theta=1e4, eps=1e-5)
    cases = [
        (dict(sliding_window=-1), ax.AXON_ERR_INVALID_ARG),
        (dict(hidden_act=5), ax.AXON_ERR_INVALID_ARG),
        (dict(qk_norm=2), ax.AXON_ERR_INVALID_ARG),
        (dict(rope_scaling_factor=8.0, rope_low_freq_factor=4.0, rope_high_freq_factor=1.0,
              rope_original_max_position=8192), ax.AXON_ERR_INVALID_ARG),
        (dict(rope_scaling_factor=-1.0), ax.AXON_ERR_INVALID_ARG),
        (dict(precision=7), ax.AXON_ERR_INVALID_ARG),
        (dict(kv_layout=ax.AXON_KV_PAGED, kv_num_blocks=0), ax.AXON_ERR_INVALID_ARG),
        (dict(head_dim=96), ax.AXON_ERR_UNSUPPORTED),
        (dict(num_key_value_heads=3), ax.AXON_ERR_UNSUPPORTED),
        (dict(kv_block_size=32), ax.AXON_ERR_UNSUPPORTED),
        (dict(max_context=100), ax.AXON_ERR_UNSUPPORTED),
        (dict(hidden_size=100), ax.AXON_ERR_UNSUPPORTED),
    ]
    for change, want in cases:
        cfg = ax.make_config(shape, max_batch=2, max_context=128)
        for k, v in change.items():
            setattr(cfg, k, v)
        out = C.c_void_p(1234)
        rc = ax.lib().axon_model_create(C.byref(cfg), None, 0, None, C.byref(out))
        assert rc == want, (change, rc)
        assert out.value is None, change
