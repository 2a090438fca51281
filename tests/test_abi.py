"""The C ABI library loads and exports every function include/gnn.h declares (no GPU calls)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_functions():
    text = open(os.path.join(ROOT, "include", "gnn.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(gnn_[a-z_]+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for n in ("gnn_create", "gnn_infer", "gnn_destroy", "gnn_status", "gnn_error_string"):
        assert n in names


def test_library_exports_every_declared_symbol():
    from paper_2402_09633_gb300 import build
    path = build.build()
    lib = ctypes.CDLL(path)
    missing = [n for n in declared_functions() if not hasattr(lib, n)]
    assert not missing, missing


def test_error_strings_without_gpu():
    from paper_2402_09633_gb300 import binding
    lib = binding.load_library()
    assert lib.gnn_error_string(0) == b"ok"
    assert lib.gnn_error_string(-5) == b"edge endpoint out of range"


def test_invalid_arguments_rejected_on_host():
    """Host-side validation returns codes before touching the device."""
    from paper_2402_09633_gb300 import binding
    lib = binding.load_library()
    h = ctypes.c_void_p()
    cfg = binding.GnnConfig(1, 3, 2, 96, 2, 2, 0, 1e-5)      # H = 96 unsupported
    assert lib.gnn_create(ctypes.byref(cfg), ctypes.c_char_p(b"x" * 64), 64, ctypes.byref(h)) == -1
    assert lib.gnn_create(None, None, 0, ctypes.byref(h)) == -1
    assert lib.gnn_infer(None, None, None, 0, 0, None, None) == -1
    assert lib.gnn_reserve(None, 1, 1) == -1
    lib.gnn_track_labels.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int64,
                                     ctypes.c_int64, ctypes.c_float, ctypes.c_void_p, ctypes.c_void_p]
    assert lib.gnn_track_labels(None, None, None, 5, 3, 0.5, None, None) == -1


def test_python_path_fails_loudly_without_library(tmp_path):
    from paper_2402_09633_gb300 import binding
    saved = binding._lib
    binding._lib = None
    try:
        with pytest.raises(RuntimeError):
            binding.load_library(str(tmp_path / "missing.so"))
    finally:
        binding._lib = saved


def test_counts_beyond_the_limit_rejected_before_device_work():
    """Every count above GNN_MAX_COUNT (2^31 - 1 - 8192: the kernels round rows up to whole blocks
    and radix tiles of up to 8192 in 32-bit arithmetic) is INVALID_ARG, checked before the context
    is read or any device call is made.  The context pointer here is a zeroed host buffer, which a
    call that got past its size checks would misuse."""
    from paper_2402_09633_gb300 import binding
    lib = binding.load_library()
    text = open(os.path.join(ROOT, "include", "gnn.h")).read()
    limit = int(re.search(r"#define GNN_MAX_COUNT (\d+)", text).group(1))
    assert limit == 2 ** 31 - 1 - 8192
    vp, i64, f32 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_float
    fake = ctypes.create_string_buffer(4096)
    ctx, buf = ctypes.cast(fake, vp), ctypes.cast(ctypes.create_string_buffer(64), vp)
    big, bad = limit + 1, -1
    lib.gnn_track_labels.argtypes = [vp, vp, vp, i64, i64, f32, vp, vp]
    lib.gnn_csr_build_noalloc.argtypes = [vp, i64, i64, vp, vp, vp, vp]
    lib.gnn_filter_edges.argtypes = [vp, vp, vp, i64, i64, f32, vp, vp, vp, vp, vp]
    lib.gnn_embed.argtypes = [vp, vp, i64, vp, vp]
    lib.gnn_build_graph.argtypes = [vp, vp, ctypes.c_int, vp, i64, f32, i64, vp, vp, vp]
    for n in (big, bad, 2 ** 31 - 1):
        assert lib.gnn_reserve(ctx, n, 1) == -1 and lib.gnn_reserve(ctx, 1, n) == -1
        assert lib.gnn_infer(ctx, buf, buf, n, 4, buf, None) == -1
        assert lib.gnn_infer(ctx, buf, buf, 4, n, buf, None) == -1
        assert lib.gnn_infer_host(ctx, buf, buf, 4, n, buf, None) == -1
        assert lib.gnn_track_labels(ctx, buf, buf, n, 1, 0.5, buf, None) == -1
        assert lib.gnn_track_labels(ctx, buf, buf, 4, n, 0.5, buf, None) == -1
        assert lib.gnn_filter_edges(ctx, buf, buf, 4, n, 0.5, buf, buf, buf, buf, None) == -1
        assert lib.gnn_embed(ctx, buf, n, buf, None) == -1
        assert lib.gnn_build_graph(ctx, buf, 8, buf, n, 0.1, 4, buf, buf, None) == -1
        assert lib.gnn_build_graph(ctx, buf, 8, buf, 4, 0.1, n, buf, buf, None) == -1
        assert lib.gnn_csr_build_noalloc(buf, n, 4, buf, buf, buf, None) == -1
