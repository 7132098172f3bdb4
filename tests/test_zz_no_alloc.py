"""gs_query_topk_noalloc: the query for callers that cannot allocate device memory.

Some hosts give a library only the buffers it reads and writes (a framework that owns the
device memory pool, an operator interface without a workspace argument, a loop that must
not synchronise the device through cudaMalloc).  For them gs_query_topk_noalloc keeps its
scratch in a fixed array inside the library.  This test calls it through the C ABI twice in
a row, with different sizes, and checks that each call gives exactly what gs_query_topk with
a caller workspace gives on the same sketch; the tolerance is exact equality, since both
run the same arithmetic.  It also checks the size limit.  The file is named so that pytest
collects it last.
"""

import numpy as np
import pytest

torch = pytest.importorskip("torch")

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def gs():
    import paper_2108_06004_gb300 as lib
    lib.load_library()
    torch.cuda.set_device(0)
    return lib


def _sketch_with_data(gs, d, r, c, seed):
    rng = np.random.default_rng(seed)
    x = (rng.standard_normal(d) * 1e-3).astype(np.float32)
    x[rng.choice(d, max(1, d // 1000), replace=False)] *= 50
    sk = gs.gs_sketch_create(r, c, seed, 1)
    gs.gs_sketch_insert(sk, 0, torch.from_numpy(x).cuda(), d)
    gs.gs_sketch_merge_tree(sk, 1)
    return sk


def _with_workspace(gs, sk, d, k):
    ws = torch.empty(gs.gs_query_topk_workspace_size(d, k), dtype=torch.uint8, device="cuda")
    idx = torch.empty(k, dtype=torch.int64, device="cuda")
    est = torch.empty(d, dtype=torch.float32, device="cuda")
    gs.gs_query_topk(sk, d, k, idx, est, ws)
    torch.cuda.synchronize()
    return idx.cpu().numpy(), est.cpu().numpy()


def test_noalloc_matches_workspace_query_twice(gs):
    cases = [(1_000_003, 5, 1 << 14, 1000, 11), (250_001, 3, 3000, 4321, 12)]
    for d, r, c, k, seed in cases:
        sk = _sketch_with_data(gs, d, r, c, seed)
        try:
            idx_ref, est_ref = _with_workspace(gs, sk, d, k)
            idx = torch.full((k,), -1, dtype=torch.int64, device="cuda")
            est = torch.zeros(d, dtype=torch.float32, device="cuda")
            gs.gs_query_topk_noalloc(sk, d, k, idx, est)
            torch.cuda.synchronize()
            assert np.array_equal(idx.cpu().numpy(), idx_ref)
            assert np.array_equal(est.cpu().numpy().view(np.uint32), est_ref.view(np.uint32))
        finally:
            gs.gs_sketch_destroy(sk)


def test_noalloc_rejects_oversize_and_missing_est(gs):
    sk = gs.gs_sketch_create(3, 64, 1, 1)
    try:
        idx = torch.empty(4, dtype=torch.int64, device="cuda")
        est = torch.empty(8, dtype=torch.float32, device="cuda")
        with pytest.raises(gs.GsError) as ei:
            gs.gs_query_topk_noalloc(sk, gs.GS_NOALLOC_MAX_DIM + 1, 4, idx, est)
        assert ei.value.status == gs.GS_ERR_INVALID_ARG and "GS_NOALLOC_MAX_DIM" in str(ei.value)
        with pytest.raises(gs.GsError):
            gs.gs_query_topk_noalloc(sk, 8, 4, idx, None)
    finally:
        gs.gs_sketch_destroy(sk)


def test_noalloc_more_than_1024_segments(gs):
    """At d = 40,000,001 the fixed scratch serves 2,442 segments of 16,384 coordinates: its
    per-segment counting and writing passes run at a scale well beyond the small cases."""
    d, r, c, k, seed = 40_000_001, 5, 1 << 17, 40_000, 13
    sk = _sketch_with_data(gs, d, r, c, seed)
    try:
        idx_ref, est_ref = _with_workspace(gs, sk, d, k)
        for _ in range(2):
            idx = torch.full((k,), -1, dtype=torch.int64, device="cuda")
            est = torch.zeros(d, dtype=torch.float32, device="cuda")
            gs.gs_query_topk_noalloc(sk, d, k, idx, est)
            torch.cuda.synchronize()
            assert np.array_equal(idx.cpu().numpy(), idx_ref)
            assert np.array_equal(est.cpu().numpy().view(np.uint32), est_ref.view(np.uint32))
    finally:
        gs.gs_sketch_destroy(sk)


_RESET_CHILD = r'''
import ctypes, sys
import numpy as np
sys.path.insert(0, sys.argv[1])
import paper_2108_06004_gb300 as gs
gs.load_library()
rt = ctypes.CDLL("libcudart.so.13")
cu = ctypes.CDLL("libcuda.so.1")
vp, sz = ctypes.c_void_p, ctypes.c_size_t

def ctx_id():
    ctx = vp()
    if cu.cuCtxGetCurrent(ctypes.byref(ctx)) != 0 or not ctx.value:
        return 0
    i = ctypes.c_ulonglong()
    return i.value if cu.cuCtxGetId(ctx, ctypes.byref(i)) == 0 else 0

def malloc(n):
    p = vp()
    assert rt.cudaMalloc(ctypes.byref(p), sz(n)) == 0
    return p.value

def copy(dst, src, n, kind):
    assert rt.cudaMemcpy(vp(dst), vp(src), sz(n), kind) == 0

d, r, c, k = 300_007, 5, 1 << 12, 777
rng = np.random.default_rng(21)
ids = []
for rnd in range(2):
    x = (rng.standard_normal(d) * 1e-3).astype(np.float32)
    x[rng.choice(d, 300, replace=False)] *= 50
    sk = gs.gs_sketch_create(r, c, 21, 1)
    ids.append(ctx_id())
    bufs = []
    dx = malloc(4 * d); bufs.append(dx)
    copy(dx, x.ctypes.data, 4 * d, 1)
    gs.gs_sketch_insert(sk, 0, dx, d, 0)
    gs.gs_sketch_merge_tree(sk, 1, 0)
    wsb = gs.gs_query_topk_workspace_size(d, k)
    ws, i_ref, e_ref, i_na, e_na = malloc(wsb), malloc(8 * k), malloc(4 * d), malloc(8 * k), malloc(4 * d)
    bufs += [ws, i_ref, e_ref, i_na, e_na]
    gs.gs_query_topk(sk, d, k, i_ref, e_ref, ws, wsb, 0)
    gs.gs_query_topk_noalloc(sk, d, k, i_na, e_na, 0)
    assert rt.cudaDeviceSynchronize() == 0
    out = [np.empty(k, np.int64), np.empty(k, np.int64), np.empty(d, np.uint32), np.empty(d, np.uint32)]
    for a, src in zip(out, (i_ref, i_na, e_ref, e_na)):
        copy(a.ctypes.data, src, a.nbytes, 2)
    assert np.array_equal(out[0], out[1]) and np.array_equal(out[2], out[3]), "round %d differs" % rnd
    gs.gs_sketch_destroy(sk)
    for b in bufs:
        assert rt.cudaFree(vp(b)) == 0
    if rnd == 0:
        assert rt.cudaDeviceReset() == 0
        # what the library sees at its next call, before anything makes a context current
        seen = ctx_id()
        if seen and seen == ids[0]:
            print("STALE_ID", seen)
            sys.exit(3)
assert ids[0] and ids[1] and ids[0] != ids[1], ids
print("OK", ids)
'''


def test_noalloc_after_device_reset(tmp_path):
    """The scratch array's address is cached per device and context.  In a fresh process (no
    PyTorch, plain runtime allocations) a query, a cudaDeviceReset, and another query on a new
    sketch both match the workspace query: the reset gives the device a new context id, and the
    library looks the address up again.  The child stops before the second query if the
    context id could be mistaken for the old one, so a stale address is never used."""
    import os
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    script = tmp_path / "reset_child.py"
    script.write_text(_RESET_CHILD)
    res = subprocess.run([sys.executable, str(script), root], capture_output=True, text=True, timeout=300)
    assert res.returncode == 0 and "OK" in res.stdout, res.stdout[-2000:] + res.stderr[-2000:]
