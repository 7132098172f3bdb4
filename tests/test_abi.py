"""The C ABI library on the CPU: it builds, loads, exports every declared symbol, and its
host-side argument validation answers before any device work."""

import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "gs_sketch.h")


@pytest.fixture(scope="module")
def lib():
    import paper_2108_06004_gb300 as gs
    if not os.path.exists(gs.LIB_PATH):
        from paper_2108_06004_gb300 import _build
        _build.build()
    return gs.load_library()


def declared_functions():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"^(?:gs_status|const char\*)\s+(gs_\w+)\s*\(", text, re.M)))


def test_header_declares_the_pipeline():
    names = declared_functions()
    for need in ("gs_sketch_create", "gs_accumulate", "gs_sketch_insert", "gs_sketch_merge_tree",
                 "gs_query_topk", "gs_gather_and_zero", "gs_accumulate_insert", "gs_step"):
        assert need in names


def test_library_exports_every_declared_symbol(lib):
    import paper_2108_06004_gb300 as gs
    names = declared_functions()
    missing = [n for n in names if not hasattr(lib, n)]
    assert not missing, missing
    assert set(names) == set(gs.SIGNATURES), "binding and header disagree"


def test_binding_has_same_names():
    import paper_2108_06004_gb300 as gs
    for n in declared_functions():
        assert callable(getattr(gs, n)), n


def _status(fn, *args):
    return fn(*args)


def test_validation_before_device_work(lib):
    import paper_2108_06004_gb300 as gs
    out = ctypes.c_void_p()
    bad_create = [(0, 16, 1, 4, 0), (17, 16, 1, 4, 0), (5, 0, 1, 4, 0), (5, (1 << 26) + 1, 1, 4, 0),
                  (5, 16, 1, 0, 0), (5, 16, 1, 65, 0), (5, 16, 1, 4, 3)]
    for a in bad_create:
        assert lib.gs_sketch_create(*a, ctypes.byref(out)) == gs.GS_ERR_INVALID_ARG, a
    assert lib.gs_sketch_create(5, 16, 1, 4, 0, None) == gs.GS_ERR_INVALID_ARG
    assert b"out is NULL" in lib.gs_last_error()
    sz = ctypes.c_size_t()
    assert lib.gs_query_topk_workspace_size(0, 1, ctypes.byref(sz)) == gs.GS_ERR_INVALID_ARG
    assert lib.gs_query_topk_workspace_size(10, 11, ctypes.byref(sz)) == gs.GS_ERR_INVALID_ARG
    assert lib.gs_query_topk_workspace_size(1 << 31, 1, ctypes.byref(sz)) == gs.GS_ERR_INVALID_ARG
    assert lib.gs_query_topk_workspace_size(1000, 10, ctypes.byref(sz)) == gs.GS_OK and sz.value >= 4000
    assert lib.gs_step_workspace_size(1000, 10, ctypes.byref(sz)) == gs.GS_OK
    assert lib.gs_accumulate(None, None, None, 10, 0.9, None) == gs.GS_ERR_INVALID_ARG
    assert lib.gs_accumulate(8, 16, 2, 10, 0.9, None) == gs.GS_ERR_INVALID_ARG  # misaligned
    assert lib.gs_accumulate(16, 32, 48, 0, 0.9, None) == gs.GS_ERR_INVALID_ARG  # d = 0
    assert lib.gs_sketch_merge_tree(None, 1, None) == gs.GS_ERR_INVALID_ARG
    assert lib.gs_sketch_destroy(None) == gs.GS_OK
    arr = (ctypes.c_void_p * 2)(16, 32)
    assert lib.gs_gather_and_zero(arr, arr, 0, 10, 64, 1, 128, None) == gs.GS_ERR_INVALID_ARG
    assert lib.gs_gather_and_zero(arr, arr, 65, 10, 64, 1, 128, None) == gs.GS_ERR_INVALID_ARG
    assert lib.gs_gather_and_zero(arr, arr, 2, 10, 64, 11, 128, None) == gs.GS_ERR_INVALID_ARG
    # plans: argument errors before any capture
    plan = ctypes.c_void_p(12345)
    assert lib.gs_step_plan_create(None, arr, arr, arr, 10, 0.9, 1, 64, 128, None, None, 0.0, 256, 1 << 20, 0,
                                   ctypes.byref(plan)) == gs.GS_ERR_INVALID_ARG
    assert plan.value is None and b"sketch is NULL" in lib.gs_last_error()
    assert lib.gs_sketched_state_plan_create(None, None, None, arr, 10, 0.9, 1, 64, 128, None, 0.0, 256, 1 << 20, 0,
                                             ctypes.byref(plan)) == gs.GS_ERR_INVALID_ARG
    assert lib.gs_step_host_plan_create(None, arr, arr, arr, arr, 10, 0.9, 1, 64, 128, 256, 1 << 20, 0,
                                        ctypes.byref(plan)) == gs.GS_ERR_INVALID_ARG
    assert lib.gs_plan_launch(None, None) == gs.GS_ERR_INVALID_ARG
    n_out = ctypes.c_int32()
    assert lib.gs_plan_insert_times(None, None, 1, ctypes.byref(n_out)) == gs.GS_ERR_INVALID_ARG
    assert lib.gs_plan_destroy(None) == gs.GS_OK


def test_binding_raises_on_error(lib):
    import paper_2108_06004_gb300 as gs
    with pytest.raises(gs.GsError) as ei:
        gs.gs_sketch_create(0, 16, 1, 4)
    assert ei.value.status == gs.GS_ERR_INVALID_ARG and "r must lie" in str(ei.value)


def test_no_cpu_fallback_when_library_missing(tmp_path, monkeypatch):
    import paper_2108_06004_gb300 as gs
    monkeypatch.setattr(gs, "_lib", None)
    monkeypatch.setattr(gs, "LIB_PATH", str(tmp_path / "absent.so"))
    with pytest.raises(ImportError):
        gs.gs_sketch_create(5, 16, 1, 4)


def test_validation_of_the_later_entry_points(lib):
    """The entry points added for merging separate sketches, the HEAVYMIX step, the staged
    insert, the measurement aids and the plan query timings reject bad arguments on the host."""
    import paper_2108_06004_gb300 as gs
    arr = (ctypes.c_void_p * 2)(16, 32)
    assert lib.gs_sketch_merge_sketches(None, 1, None) == gs.GS_ERR_INVALID_ARG
    none2 = (ctypes.c_void_p * 2)(None, None)
    assert lib.gs_sketch_merge_sketches(none2, 0, None) == gs.GS_ERR_INVALID_ARG
    assert lib.gs_sketch_merge_sketches(none2, 65, None) == gs.GS_ERR_INVALID_ARG
    assert lib.gs_sketch_merge_sketches(none2, 2, None) == gs.GS_ERR_INVALID_ARG   # NULL sketch
    sz = ctypes.c_size_t()
    assert lib.gs_heavymix_step_workspace_size(0, 1, ctypes.byref(sz)) == gs.GS_ERR_INVALID_ARG
    assert lib.gs_heavymix_step_workspace_size(1000, 10, ctypes.byref(sz)) == gs.GS_OK and sz.value >= 8000
    assert lib.gs_heavymix_step(None, arr, arr, arr, 10, 0.9, 1, 7, 64, 128, None, 256, 1 << 20, None) \
        == gs.GS_ERR_INVALID_ARG
    plan = ctypes.c_void_p(1)
    assert lib.gs_heavymix_step_plan_create(None, arr, arr, arr, 10, 0.9, 1, 7, 64, 128, None, 256, 1 << 20, 0,
                                            ctypes.byref(plan)) == gs.GS_ERR_INVALID_ARG
    assert plan.value is None
    assert lib.gs_accumulate_insert_staged(None, 0, 1, arr, arr, arr, 10, 0.9, None) == gs.GS_ERR_INVALID_ARG
    ms = ctypes.c_float()
    assert lib.gs_insert_request_ceiling(None, 10, 256, 1 << 20, ctypes.byref(ms), None) == gs.GS_ERR_INVALID_ARG
    assert lib.gs_insert_request_ceiling_window_size(None, ctypes.byref(sz)) == gs.GS_ERR_INVALID_ARG
    assert lib.gs_query_request_ceiling(None, 10, 256, 1 << 20, ctypes.byref(ms), None) == gs.GS_ERR_INVALID_ARG
    n_out = ctypes.c_int32()
    assert lib.gs_plan_query_times(None, None, None, 1, ctypes.byref(n_out)) == gs.GS_ERR_INVALID_ARG
    assert lib.gs_query_topk_noalloc(None, 10, 1, 64, 128, None) == gs.GS_ERR_INVALID_ARG
