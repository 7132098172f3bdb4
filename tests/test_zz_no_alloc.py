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
