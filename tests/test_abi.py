"""The C-ABI library builds, loads, exports every declared symbol and rejects
bad arguments before touching the device (no GPU needed)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2608_08086_gb300 import build
    return ctypes.CDLL(build.build())


def declared_functions():
    names = []
    for fn in os.listdir(os.path.join(ROOT, "include")):
        if fn.endswith(".h"):
            text = open(os.path.join(ROOT, "include", fn)).read()
            text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
            names += re.findall(r"\b(archer_[a-z0-9_]+)\s*\(", text)
    return sorted(set(names))


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert len(names) >= 10
    missing = [n for n in names if not hasattr(lib, n)]
    assert not missing, f"declared but not exported: {missing}"


def test_status_strings_and_version(lib):
    lib.archer_status_string.restype = ctypes.c_char_p
    assert lib.archer_status_string(0) == b"ok"
    assert lib.archer_status_string(-4) == b"device wait timed out"
    assert lib.archer_version() >= 200      # 0.2.0: step graph, decoder stand-in, row scatter


class Shape(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int), ("prompt_len", ctypes.c_int), ("resp_len", ctypes.c_int),
                ("n_heads", ctypes.c_int), ("n_kv_heads", ctypes.c_int), ("head_dim", ctypes.c_int),
                ("softmax_scale", ctypes.c_float)]


def _attn_step(lib, shape, ptr=0x10000):
    f = lib.archer_attn_step
    f.argtypes = [ctypes.POINTER(Shape)] + [ctypes.c_void_p] * 8 + [ctypes.c_size_t, ctypes.c_void_p]
    f.restype = ctypes.c_int
    p = ctypes.c_void_p(ptr)
    return f(ctypes.byref(shape), p, p, p, p, p, p, None, None, 0, None)


def test_bad_shapes_rejected_before_any_launch(lib):
    lib.archer_last_error.restype = ctypes.c_char_p
    assert _attn_step(lib, Shape(1, 4, 4, 3, 2, 128, 0.0)) == -1          # Hq % Hkv != 0
    assert b"multiple" in lib.archer_last_error()
    assert _attn_step(lib, Shape(1, 4, 0, 2, 2, 128, 0.0)) == -1          # G = 0
    assert _attn_step(lib, Shape(1, 4, 4, 2, 2, 96, 0.0)) == -2           # D unsupported
    assert _attn_step(lib, Shape(1, 4, 4, 2, 2, 128, float("nan"))) == -1
    assert _attn_step(lib, Shape(1, 4, 4, 2, 2, 128, 0.0), ptr=0x10008) == -1   # misaligned
    assert b"aligned" in lib.archer_last_error()
    f = lib.archer_attn_step
    s = Shape(1, 4, 4, 2, 2, 128, 0.0)
    assert f(ctypes.byref(s), None, None, None, None, None, None, None, None, 0, None) == -1
    assert _attn_step(lib, Shape(0, 4, 4, 2, 2, 128, 0.0)) == 0            # empty batch: no-op


def test_bad_scoring_and_rule_arguments_rejected(lib):
    f = lib.archer_decode_scores
    f.argtypes = [ctypes.c_int] * 4 + [ctypes.c_void_p, ctypes.c_int64] + [ctypes.c_void_p] * 7 + [
        ctypes.c_size_t, ctypes.c_void_p]
    p = ctypes.c_void_p(0x10000)
    assert f(1, 4, 100, 0, p, 50, None, None, p, p, p, None, None, 0, None) == -1     # stride < vocab
    assert f(1, 4, 100, 0, ctypes.c_void_p(0x10001), 100, None, None, p, p, p, None, None, 0, None) == -1  # odd
    assert f(1, 4, 104, 7, p, 104, None, None, p, p, p, None, None, 0, None) == -2    # dtype
    assert f(1, 4, 104, 0, p, 104, None, None, None, p, p, None, None, 0, None) == -1  # null output
    g = lib.archer_should_refresh
    g.argtypes = [ctypes.c_int, ctypes.c_int] + [ctypes.c_void_p] * 3 + [ctypes.c_int] * 3 + [ctypes.c_void_p] * 3
    assert g(-1, 4, p, p, p, 1, 0, 1, p, p, None) == -1
    assert g(2, 4, None, p, p, 1, 0, 1, p, p, None) == -1
    assert g(0, 4, None, None, None, 1, 0, 1, None, None, None) == 0


def test_step_graph_arguments_rejected_before_any_cuda_call(lib):
    c = lib.archer_step_graph_create
    c.argtypes = [ctypes.c_void_p, ctypes.c_void_p]
    out = ctypes.c_void_p(0x1234)
    assert c(None, ctypes.byref(out)) == -1 and out.value is None      # NULL desc; *out cleared
    assert c(None, None) == -1                                          # NULL out
    lib.archer_step_graph_launch.argtypes = [ctypes.c_void_p, ctypes.c_void_p]
    assert lib.archer_step_graph_launch(None, None) == -1
    lib.archer_step_graph_destroy.argtypes = [ctypes.c_void_p]
    assert lib.archer_step_graph_destroy(None) == 0


def test_decoder_update_arguments_rejected(lib):
    f = lib.archer_decoder_update
    f.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_float, ctypes.c_float, ctypes.c_int32] + [ctypes.c_void_p] * 6
    p = ctypes.c_void_p(0x10000)
    assert f(-1, 4, 0.9, 0.05, -1, p, p, p, p, p, None) == -1
    assert f(2, 4, 0.9, 0.05, -1, None, p, p, p, p, None) == -1
    assert f(2, 4, float("nan"), 0.05, -1, p, p, p, p, p, None) == -1
    assert f(0, 4, 0.9, 0.05, -1, None, None, None, None, None, None) == 0


def test_scatter_rows_arguments_rejected(lib):
    f = lib.archer_scatter_rows
    f.argtypes = [ctypes.c_int] * 3 + [ctypes.c_size_t] + [ctypes.c_void_p] * 3 + [ctypes.c_int] * 2 + [
        ctypes.c_void_p] + [ctypes.c_int] * 2 + [ctypes.c_void_p]
    p = ctypes.c_void_p(0x10000)
    assert f(1, 1, 1, 24, p, p, p, 4, 0, None, 0, 0, None) == -1          # row_bytes % 16
    assert f(1, 1, 1, 32, None, p, p, 4, 0, None, 0, 0, None) == -1       # NULL src
    assert f(1, 1, 1, 32, p, p, ctypes.c_void_p(0x10008), 4, 0, None, 0, 0, None) == -1   # misaligned
    assert f(-1, 1, 1, 32, p, p, p, 4, 0, None, 0, 0, None) == -1
    assert f(0, 1, 1, 32, None, None, None, 0, 0, None, 0, 0, None) == 0   # nothing to do


def test_refresh_and_cache_rewrite_arguments_rejected(lib):
    lib.archer_last_error.restype = ctypes.c_char_p
    p, odd = ctypes.c_void_p(0x10000), ctypes.c_void_p(0x10008)
    f = lib.archer_prompt_refresh
    f.argtypes = [ctypes.POINTER(Shape)] + [ctypes.c_void_p] * 11 + [ctypes.c_size_t, ctypes.c_void_p]
    s = Shape(1, 4, 4, 2, 2, 128, 0.0)
    assert f(ctypes.byref(s), p, p, p, p, p, p, None, None, p, None, None, 0, None) == -1   # NULL v_cache
    assert f(ctypes.byref(s), p, p, p, p, p, p, None, p, odd, None, None, 0, None) == -1     # misaligned
    assert b"aligned" in lib.archer_last_error()
    bad = Shape(1, 4, 4, 3, 2, 128, 0.0)
    assert f(ctypes.byref(bad), p, p, p, p, p, p, None, p, p, None, None, 0, None) == -1     # Hq % Hkv
    assert f(None, p, p, p, p, p, p, None, p, p, None, None, 0, None) == -1                  # NULL shape
    empty = Shape(0, 4, 4, 2, 2, 128, 0.0)
    assert f(ctypes.byref(empty), p, p, p, p, p, p, None, p, p, None, None, 0, None) == 0    # empty batch
    g = lib.archer_cache_rewrite
    g.argtypes = [ctypes.POINTER(Shape)] + [ctypes.c_void_p] * 6
    assert g(ctypes.byref(s), p, None, p, p, None, None) == -1                               # NULL v_src
    assert g(ctypes.byref(s), p, p, odd, p, None, None) == -1                                # misaligned
    assert g(ctypes.byref(Shape(1, 4, 4, 2, 2, 96, 0.0)), p, p, p, p, None, None) == -2      # D 96
    assert g(ctypes.byref(Shape(1, 0, 4, 2, 2, 128, 0.0)), None, None, None, None, None, None) == 0  # P 0


def test_workspace_queries_of_bad_shapes_are_zero(lib):
    w = lib.archer_attn_workspace_size
    w.argtypes = [ctypes.POINTER(Shape), ctypes.c_int]
    w.restype = ctypes.c_size_t
    assert w(ctypes.byref(Shape(1, 4, 4, 3, 2, 128, 0.0)), 8) == 0       # Hq % Hkv
    assert w(ctypes.byref(Shape(1, 4, 4, 2, 2, 128, 0.0)), 0) == 0       # no queries
    assert w(None, 8) == 0
    lib.archer_status_string.restype = ctypes.c_char_p
    assert lib.archer_status_string(12345)                                # any code has a string


def test_no_cpu_path_the_binding_and_smoke_fail_loudly(tmp_path):
    # the binding refuses to import where its library is missing
    import importlib.util
    import shutil
    src = os.path.join(ROOT, "paper_2608_08086_gb300", "archer.py")
    shutil.copy(src, tmp_path / "archer.py")
    spec = importlib.util.spec_from_file_location("archer_without_library", tmp_path / "archer.py")
    mod = importlib.util.module_from_spec(spec)
    with pytest.raises(ImportError, match="no CPU fallback"):
        spec.loader.exec_module(mod)
    # smoke() on a machine without a GPU raises instead of passing on the CPU
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    import __graft_entry__
    with pytest.raises(RuntimeError, match="cuda:0"):
        __graft_entry__.smoke()
