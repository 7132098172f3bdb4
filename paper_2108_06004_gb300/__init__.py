"""Python binding of libgs_sketch, the GB300 gs-SGD gradient-compression library.

The functions below carry the names of the C ABI declared in ``include/gs_sketch.h`` and
only marshal arguments: tensors become device pointers (``tensor.data_ptr()``), lists of
tensors become host arrays of device pointers, and the stream defaults to PyTorch's
current stream.  Every step of the computation runs in the library's CUDA kernels; there
is no fallback.  A non-OK status raises ``GsError`` with the library's message.
"""

from __future__ import annotations

import ctypes
import os

LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libgs_sketch.so")

GS_OK = 0
GS_ERR_INVALID_ARG = 1
GS_ERR_MISMATCH = 2
GS_ERR_OOM = 3
GS_ERR_CUDA = 4
GS_ERR_TIMEOUT = 5
GS_MAX_ROWS = 16
GS_MAX_COLS = 1 << 26
GS_MAX_WORKERS = 64
GS_MAX_DIM = (1 << 31) - 1
GS_NOALLOC_MAX_DIM = 1 << 30
GS_CEILING_WINDOW_FLOATS = 1 << 17

_lib = None

_vp = ctypes.c_void_p
_i32, _i64, _u64, _f32, _sz = ctypes.c_int32, ctypes.c_int64, ctypes.c_uint64, ctypes.c_float, ctypes.c_size_t
_PP = ctypes.POINTER(ctypes.c_void_p)

# name -> argument types (all return gs_status / int32 unless listed in _RESTYPES)
SIGNATURES = {
    "gs_sketch_create": [_i32, _i32, _u64, _i32, _i32, ctypes.POINTER(_vp)],
    "gs_sketch_destroy": [_vp],
    "gs_sketch_info": [_vp, ctypes.POINTER(_i32), ctypes.POINTER(_i32), ctypes.POINTER(_i32),
                       ctypes.POINTER(_i32), ctypes.POINTER(_i32)],
    "gs_sketch_coefficients": [_vp, ctypes.POINTER(_u64)],
    "gs_sketch_zero": [_vp, _vp],
    "gs_accumulate": [_vp, _vp, _vp, _i64, _f32, _vp],
    "gs_sketch_insert": [_vp, _i32, _vp, _i64, _vp],
    "gs_accumulate_insert": [_vp, _i32, _i32, _PP, _PP, _PP, _i64, _f32, _vp],
    "gs_accumulate_insert_staged": [_vp, _i32, _i32, _PP, _PP, _PP, _i64, _f32, _vp],
    "gs_sketch_merge_tree": [_vp, _i32, _vp],
    "gs_sketch_merge_sketches": [_PP, _i32, _vp],
    "gs_query_topk_workspace_size": [_i64, _i64, ctypes.POINTER(_sz)],
    "gs_query_topk": [_vp, _i64, _i64, _vp, _vp, _vp, _sz, _vp],
    "gs_query_topk_noalloc": [_vp, _i64, _i64, _vp, _vp, _vp],
    "gs_query_heavymix_workspace_size": [_i64, _i64, ctypes.POINTER(_sz)],
    "gs_query_heavymix": [_vp, _i64, _i64, _u64, _vp, _vp, _vp, _vp, _sz, _vp],
    "gs_gather_and_zero": [_PP, _PP, _i32, _i64, _vp, _i64, _vp, _vp],
    "gs_apply_update": [_vp, _i64, _vp, _vp, _i64, _f32, _vp],
    "gs_gather_zero_update": [_PP, _PP, _i32, _i64, _vp, _i64, _vp, _vp, _f32, _vp],
    "gs_train_step": [_vp, _vp, _f32, _PP, _PP, _PP, _i64, _f32, _i64, _vp, _vp, _vp, _vp, _sz, _vp],
    "gs_heavymix_step_workspace_size": [_i64, _i64, ctypes.POINTER(_sz)],
    "gs_heavymix_step": [_vp, _PP, _PP, _PP, _i64, _f32, _i64, _u64, _vp, _vp, _vp, _vp, _sz, _vp],
    "gs_heavymix_step_plan_create": [_vp, _PP, _PP, _PP, _i64, _f32, _i64, _u64, _vp, _vp, _vp, _vp, _sz, _i32,
                                     ctypes.POINTER(_vp)],
    "gs_sketch_merged_table": [_vp, ctypes.POINTER(_vp)],
    "gs_sketch_query_at": [_vp, _vp, _i64, _vp, _vp],
    "gs_sketch_add_sparse": [_vp, _vp, _vp, _i64, _f32, _vp],
    "gs_sketched_state_step": [_vp, _vp, _vp, _PP, _i64, _f32, _i64, _vp, _vp, _vp, _f32, _vp, _sz, _vp],
    "gs_step_plan_create": [_vp, _PP, _PP, _PP, _i64, _f32, _i64, _vp, _vp, _vp, _vp, _f32, _vp, _sz, _i32,
                            ctypes.POINTER(_vp)],
    "gs_step_host_plan_create": [_vp, _PP, _PP, _PP, _PP, _i64, _f32, _i64, _vp, _vp, _vp, _sz, _i32,
                                 ctypes.POINTER(_vp)],
    "gs_sketched_state_plan_create": [_vp, _vp, _vp, _PP, _i64, _f32, _i64, _vp, _vp, _vp, _f32, _vp, _sz, _i32,
                                      ctypes.POINTER(_vp)],
    "gs_plan_launch": [_vp, _vp],
    "gs_plan_insert_times": [_vp, _vp, _i32, ctypes.POINTER(_i32)],
    "gs_plan_query_times": [_vp, _vp, _vp, _i32, ctypes.POINTER(_i32)],
    "gs_plan_destroy": [_vp],
    "gs_step_workspace_size": [_i64, _i64, ctypes.POINTER(_sz)],
    "gs_step": [_vp, _PP, _PP, _PP, _i64, _f32, _i64, _vp, _vp, _vp, _vp, _sz, _vp],
    "gs_step_host": [_vp, _PP, _PP, _PP, _PP, _i64, _f32, _i64, _vp, _vp, _vp, _sz, _vp],
    "gs_insert_request_ceiling_window_size": [_vp, ctypes.POINTER(_sz)],
    "gs_insert_request_ceiling": [_vp, _i64, _vp, _sz, ctypes.POINTER(_f32), _vp],
    "gs_query_request_ceiling": [_vp, _i64, _vp, _sz, ctypes.POINTER(_f32), _vp],
    "gs_hash_eval": [_vp, _vp, _i64, _vp, _vp, _vp],
    "gs_sketch_copy_to_host": [_vp, _i32, _vp],
    "gs_last_error": [],
}
_RESTYPES = {"gs_last_error": ctypes.c_char_p}


class GsError(RuntimeError):
    def __init__(self, status: int, func: str, msg: str):
        super().__init__(f"{func} failed with status {status}: {msg}")
        self.status = status


def load_library():
    """Load libgs_sketch.so (built by ``paper_2108_06004_gb300._build``); raise if absent."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise ImportError(
                f"{LIB_PATH} is missing: build it with `python -c \"import __graft_entry__ as g; g.build()\"` "
                "(the CUDA library is required; there is no CPU fallback)")
        lib = ctypes.CDLL(LIB_PATH)
        for name, args in SIGNATURES.items():
            fn = getattr(lib, name)
            fn.argtypes = args
            fn.restype = _RESTYPES.get(name, _i32)
        _lib = lib
    return _lib


def _check(status: int, func: str):
    if status != GS_OK:
        msg = load_library().gs_last_error().decode(errors="replace")
        raise GsError(status, func, msg)


def _ptr(x) -> int | None:
    if x is None:
        return None
    if hasattr(x, "data_ptr"):
        return x.data_ptr()
    return int(x)


def _ptr_array(xs):
    return (ctypes.c_void_p * len(xs))(*[_ptr(x) for x in xs])


def _stream(stream):
    if stream is not None:
        return _ptr(getattr(stream, "cuda_stream", stream))
    import torch
    return torch.cuda.current_stream().cuda_stream


# ---- C ABI, same names ------------------------------------------------------------------

def gs_sketch_create(r: int, c: int, seed: int, workers: int, group_width: int = 0) -> int:
    out = _vp()
    _check(load_library().gs_sketch_create(r, c, seed, workers, group_width, ctypes.byref(out)),
           "gs_sketch_create")
    return out.value


def gs_sketch_destroy(sketch: int) -> None:
    _check(load_library().gs_sketch_destroy(sketch), "gs_sketch_destroy")


def gs_sketch_info(sketch: int) -> dict:
    r, c, w, g, rp = _i32(), _i32(), _i32(), _i32(), _i32()
    _check(load_library().gs_sketch_info(sketch, ctypes.byref(r), ctypes.byref(c), ctypes.byref(w),
                                         ctypes.byref(g), ctypes.byref(rp)), "gs_sketch_info")
    return {"r": r.value, "c": c.value, "workers": w.value, "group_width": g.value,
            "rows_per_pass": rp.value}


def gs_sketch_coefficients(sketch: int):
    """(a, b, a2, b2) lists of Python ints, one entry per row."""
    r = gs_sketch_info(sketch)["r"]
    buf = (_u64 * (4 * r))()
    _check(load_library().gs_sketch_coefficients(sketch, buf), "gs_sketch_coefficients")
    v = list(buf)
    return v[0::4], v[1::4], v[2::4], v[3::4]


def gs_sketch_zero(sketch: int, stream=None) -> None:
    _check(load_library().gs_sketch_zero(sketch, _stream(stream)), "gs_sketch_zero")


def gs_accumulate(momentum, error, grad, d: int, rho: float, stream=None) -> None:
    _check(load_library().gs_accumulate(_ptr(momentum), _ptr(error), _ptr(grad), d, rho,
                                        _stream(stream)), "gs_accumulate")


def gs_sketch_insert(sketch: int, worker: int, vec, d: int, stream=None) -> None:
    _check(load_library().gs_sketch_insert(sketch, worker, _ptr(vec), d, _stream(stream)),
           "gs_sketch_insert")


def gs_accumulate_insert(sketch: int, first_worker: int, momentum, error, grad, d: int,
                         rho: float, stream=None) -> None:
    n = len(grad)
    _check(load_library().gs_accumulate_insert(sketch, first_worker, n, _ptr_array(momentum),
                                               _ptr_array(error), _ptr_array(grad), d, rho,
                                               _stream(stream)), "gs_accumulate_insert")


def gs_accumulate_insert_staged(sketch: int, first_worker: int, momentum, error, grad, d: int,
                                rho: float, stream=None) -> None:
    n = len(grad)
    _check(load_library().gs_accumulate_insert_staged(sketch, first_worker, n, _ptr_array(momentum),
                                                      _ptr_array(error), _ptr_array(grad), d, rho,
                                                      _stream(stream)), "gs_accumulate_insert_staged")


def gs_sketch_merge_tree(sketch: int, P: int, stream=None) -> None:
    _check(load_library().gs_sketch_merge_tree(sketch, P, _stream(stream)), "gs_sketch_merge_tree")


def gs_sketch_merge_sketches(sketches, stream=None) -> None:
    """Tree merge of separately created sketches into the merged table of sketches[0]."""
    arr = (ctypes.c_void_p * len(sketches))(*sketches)
    _check(load_library().gs_sketch_merge_sketches(arr, len(sketches), _stream(stream)), "gs_sketch_merge_sketches")


def gs_query_topk_workspace_size(d: int, k: int) -> int:
    out = _sz()
    _check(load_library().gs_query_topk_workspace_size(d, k, ctypes.byref(out)),
           "gs_query_topk_workspace_size")
    return out.value


def gs_query_topk(sketch: int, d: int, k: int, idx_out, est_out, workspace, workspace_bytes=None,
                  stream=None) -> None:
    if workspace_bytes is None:
        workspace_bytes = workspace.numel() * workspace.element_size()
    _check(load_library().gs_query_topk(sketch, d, k, _ptr(idx_out), _ptr(est_out), _ptr(workspace),
                                        workspace_bytes, _stream(stream)), "gs_query_topk")


def gs_query_heavymix_workspace_size(d: int, k: int) -> int:
    out = _sz()
    _check(load_library().gs_query_heavymix_workspace_size(d, k, ctypes.byref(out)),
           "gs_query_heavymix_workspace_size")
    return out.value


def gs_query_heavymix(sketch: int, d: int, k: int, fill_seed: int, idx_out, est_out, l2sq_out, workspace,
                      workspace_bytes=None, stream=None) -> None:
    if workspace_bytes is None:
        workspace_bytes = workspace.numel() * workspace.element_size()
    _check(load_library().gs_query_heavymix(sketch, d, k, fill_seed, _ptr(idx_out), _ptr(est_out), _ptr(l2sq_out),
                                            _ptr(workspace), workspace_bytes, _stream(stream)), "gs_query_heavymix")


def gs_query_topk_noalloc(sketch: int, d: int, k: int, idx_out, est_out, stream=None) -> None:
    """gs_query_topk without a caller workspace: the library's fixed device scratch is used
    (for hosts that cannot allocate device memory; est_out is required)."""
    _check(load_library().gs_query_topk_noalloc(sketch, d, k, _ptr(idx_out), _ptr(est_out), _stream(stream)),
           "gs_query_topk_noalloc")


def gs_gather_and_zero(momentum, error, d: int, idx, k: int, vals_out, stream=None) -> None:
    P = len(momentum)
    _check(load_library().gs_gather_and_zero(_ptr_array(momentum), _ptr_array(error), P, d, _ptr(idx), k,
                                             _ptr(vals_out), _stream(stream)), "gs_gather_and_zero")


def gs_apply_update(weights, d: int, idx, vals, k: int, lr: float, stream=None) -> None:
    _check(load_library().gs_apply_update(_ptr(weights), d, _ptr(idx), _ptr(vals), k, lr, _stream(stream)),
           "gs_apply_update")


def gs_gather_zero_update(momentum, error, d: int, idx, k: int, vals_out, weights, lr: float,
                          stream=None) -> None:
    P = len(momentum)
    _check(load_library().gs_gather_zero_update(_ptr_array(momentum), _ptr_array(error), P, d, _ptr(idx), k,
                                                _ptr(vals_out), _ptr(weights), lr, _stream(stream)),
           "gs_gather_zero_update")


def gs_train_step(sketch: int, weights, lr: float, momentum, error, grad, d: int, rho: float, k: int,
                  idx_out, vals_out, est_out, workspace, workspace_bytes=None, stream=None) -> None:
    if workspace_bytes is None:
        workspace_bytes = workspace.numel() * workspace.element_size()
    _check(load_library().gs_train_step(sketch, _ptr(weights), lr, _ptr_array(momentum), _ptr_array(error),
                                        _ptr_array(grad), d, rho, k, _ptr(idx_out), _ptr(vals_out), _ptr(est_out),
                                        _ptr(workspace), workspace_bytes, _stream(stream)), "gs_train_step")


def gs_sketch_merged_table(sketch: int) -> int:
    out = _vp()
    _check(load_library().gs_sketch_merged_table(sketch, ctypes.byref(out)), "gs_sketch_merged_table")
    return out.value


def gs_sketch_query_at(sketch: int, idx, k: int, est_out, stream=None) -> None:
    _check(load_library().gs_sketch_query_at(sketch, _ptr(idx), k, _ptr(est_out), _stream(stream)),
           "gs_sketch_query_at")


def gs_sketch_add_sparse(sketch: int, idx, vals, k: int, scale: float, stream=None) -> None:
    _check(load_library().gs_sketch_add_sparse(sketch, _ptr(idx), _ptr(vals), k, scale, _stream(stream)),
           "gs_sketch_add_sparse")


def gs_sketched_state_step(workers: int, momentum: int, error: int, grad, d: int, rho: float, k: int, idx_out,
                           vals_out, weights, lr: float, workspace, workspace_bytes=None, stream=None) -> None:
    if workspace_bytes is None:
        workspace_bytes = workspace.numel() * workspace.element_size()
    _check(load_library().gs_sketched_state_step(workers, momentum, error, _ptr_array(grad), d, rho, k, _ptr(idx_out),
                                                 _ptr(vals_out), _ptr(weights), lr, _ptr(workspace), workspace_bytes,
                                                 _stream(stream)), "gs_sketched_state_step")


def gs_step_workspace_size(d: int, k: int) -> int:
    out = _sz()
    _check(load_library().gs_step_workspace_size(d, k, ctypes.byref(out)), "gs_step_workspace_size")
    return out.value


def gs_step(sketch: int, momentum, error, grad, d: int, rho: float, k: int, idx_out, vals_out,
            est_out, workspace, workspace_bytes=None, stream=None) -> None:
    if workspace_bytes is None:
        workspace_bytes = workspace.numel() * workspace.element_size()
    _check(load_library().gs_step(sketch, _ptr_array(momentum), _ptr_array(error), _ptr_array(grad), d, rho, k,
                                  _ptr(idx_out), _ptr(vals_out), _ptr(est_out), _ptr(workspace),
                                  workspace_bytes, _stream(stream)), "gs_step")


def gs_step_host(sketch: int, momentum, error, grad_host, grad_dev, d: int, rho: float, k: int,
                 idx_host, vals_host, workspace, workspace_bytes=None, stream=None) -> None:
    if workspace_bytes is None:
        workspace_bytes = workspace.numel() * workspace.element_size()
    _check(load_library().gs_step_host(sketch, _ptr_array(momentum), _ptr_array(error), _ptr_array(grad_host),
                                       _ptr_array(grad_dev), d, rho, k, _ptr(idx_host), _ptr(vals_host),
                                       _ptr(workspace), workspace_bytes, _stream(stream)), "gs_step_host")


GS_PLAN_TIME_INSERT = 1
GS_PLAN_TIME_QUERY = 2


def _nbytes(workspace, workspace_bytes):
    return workspace.numel() * workspace.element_size() if workspace_bytes is None else workspace_bytes


def gs_heavymix_step_workspace_size(d: int, k: int) -> int:
    out = _sz()
    _check(load_library().gs_heavymix_step_workspace_size(d, k, ctypes.byref(out)), "gs_heavymix_step_workspace_size")
    return out.value


def gs_heavymix_step(sketch: int, momentum, error, grad, d: int, rho: float, k: int, fill_seed: int, idx_out,
                     vals_out, l2sq_out, workspace, workspace_bytes=None, stream=None) -> None:
    _check(load_library().gs_heavymix_step(sketch, _ptr_array(momentum), _ptr_array(error), _ptr_array(grad), d, rho,
                                           k, fill_seed, _ptr(idx_out), _ptr(vals_out), _ptr(l2sq_out),
                                           _ptr(workspace), _nbytes(workspace, workspace_bytes), _stream(stream)),
           "gs_heavymix_step")


def gs_heavymix_step_plan_create(sketch: int, momentum, error, grad, d: int, rho: float, k: int, fill_seed: int,
                                 idx_out, vals_out, l2sq_out, workspace, workspace_bytes=None, flags: int = 0) -> int:
    out = _vp()
    _check(load_library().gs_heavymix_step_plan_create(sketch, _ptr_array(momentum), _ptr_array(error),
                                                       _ptr_array(grad), d, rho, k, fill_seed, _ptr(idx_out),
                                                       _ptr(vals_out), _ptr(l2sq_out), _ptr(workspace),
                                                       _nbytes(workspace, workspace_bytes), flags,
                                                       ctypes.byref(out)), "gs_heavymix_step_plan_create")
    return out.value


def gs_step_plan_create(sketch: int, momentum, error, grad, d: int, rho: float, k: int, idx_out, vals_out,
                        est_out=None, weights=None, lr: float = 0.0, workspace=None, workspace_bytes=None,
                        flags: int = 0) -> int:
    out = _vp()
    _check(load_library().gs_step_plan_create(sketch, _ptr_array(momentum), _ptr_array(error), _ptr_array(grad), d,
                                              rho, k, _ptr(idx_out), _ptr(vals_out), _ptr(est_out), _ptr(weights), lr,
                                              _ptr(workspace), _nbytes(workspace, workspace_bytes), flags,
                                              ctypes.byref(out)), "gs_step_plan_create")
    return out.value


def gs_step_host_plan_create(sketch: int, momentum, error, grad_host, grad_dev, d: int, rho: float, k: int,
                             idx_host, vals_host, workspace, workspace_bytes=None, flags: int = 0) -> int:
    out = _vp()
    _check(load_library().gs_step_host_plan_create(sketch, _ptr_array(momentum), _ptr_array(error),
                                                   _ptr_array(grad_host), _ptr_array(grad_dev), d, rho, k,
                                                   _ptr(idx_host), _ptr(vals_host), _ptr(workspace),
                                                   _nbytes(workspace, workspace_bytes), flags, ctypes.byref(out)),
           "gs_step_host_plan_create")
    return out.value


def gs_sketched_state_plan_create(workers: int, momentum: int, error: int, grad, d: int, rho: float, k: int,
                                  idx_out, vals_out, weights, lr: float, workspace, workspace_bytes=None,
                                  flags: int = 0) -> int:
    out = _vp()
    _check(load_library().gs_sketched_state_plan_create(workers, momentum, error, _ptr_array(grad), d, rho, k,
                                                        _ptr(idx_out), _ptr(vals_out), _ptr(weights), lr,
                                                        _ptr(workspace), _nbytes(workspace, workspace_bytes), flags,
                                                        ctypes.byref(out)), "gs_sketched_state_plan_create")
    return out.value


def gs_plan_launch(plan: int, stream=None) -> None:
    _check(load_library().gs_plan_launch(plan, _stream(stream)), "gs_plan_launch")


def gs_plan_insert_times(plan: int, n: int = 1024) -> list:
    buf = (ctypes.c_float * max(n, 1))()
    got = _i32()
    _check(load_library().gs_plan_insert_times(plan, ctypes.cast(buf, _vp), n, ctypes.byref(got)),
           "gs_plan_insert_times")
    return [float(buf[i]) for i in range(got.value)]


def gs_plan_query_times(plan: int, n: int = 1024) -> tuple:
    """(query_ms, select_ms): lists over the last launches, oldest first."""
    q = (ctypes.c_float * max(n, 1))()
    sel = (ctypes.c_float * max(n, 1))()
    got = _i32()
    _check(load_library().gs_plan_query_times(plan, ctypes.cast(q, _vp), ctypes.cast(sel, _vp), n,
                                              ctypes.byref(got)), "gs_plan_query_times")
    return [float(q[i]) for i in range(got.value)], [float(sel[i]) for i in range(got.value)]


def gs_plan_destroy(plan: int) -> None:
    _check(load_library().gs_plan_destroy(plan), "gs_plan_destroy")


def gs_insert_request_ceiling_window_size(sketch: int) -> int:
    out = _sz()
    _check(load_library().gs_insert_request_ceiling_window_size(sketch, ctypes.byref(out)),
           "gs_insert_request_ceiling_window_size")
    return out.value


def gs_insert_request_ceiling(sketch: int, d: int, window, window_bytes=None, stream=None) -> float:
    """Milliseconds of one insert phase's request mix with the vectors held in L2."""
    ms = _f32()
    _check(load_library().gs_insert_request_ceiling(sketch, d, _ptr(window), _nbytes(window, window_bytes),
                                                    ctypes.byref(ms), _stream(stream)), "gs_insert_request_ceiling")
    return float(ms.value)


def gs_query_request_ceiling(sketch: int, d: int, window, window_bytes=None, stream=None) -> float:
    """Milliseconds of the median query's loads alone (all r rows) for d coordinates."""
    ms = _f32()
    _check(load_library().gs_query_request_ceiling(sketch, d, _ptr(window), _nbytes(window, window_bytes),
                                                   ctypes.byref(ms), _stream(stream)), "gs_query_request_ceiling")
    return float(ms.value)


def gs_hash_eval(sketch: int, coords, n: int, bucket_out, sign_out, stream=None) -> None:
    _check(load_library().gs_hash_eval(sketch, _ptr(coords), n, _ptr(bucket_out), _ptr(sign_out),
                                       _stream(stream)), "gs_hash_eval")


def gs_sketch_copy_to_host(sketch: int, worker: int, host_out) -> None:
    """host_out: a contiguous host fp32 buffer of r*c values (numpy array or tensor)."""
    ptr = host_out.ctypes.data if hasattr(host_out, "ctypes") else _ptr(host_out)
    _check(load_library().gs_sketch_copy_to_host(sketch, worker, ptr), "gs_sketch_copy_to_host")


def gs_last_error() -> str:
    return load_library().gs_last_error().decode(errors="replace")
