"""GPU parity at the full sizes of the larger workloads (run on a GB300).

ResNet-50 size (d = 25,557,032, P = 8): one full step against the complete oracle.
VGG-16 size (d = 138,357,544, P = 16, r = 7, c = 2^20) and BERT-large size
(d = 333,244,416, P = 32 with 8 workers' gradients resident at a time, c = 2^21): one step in
the same launch configuration as the benchmark, checked where the oracle can be evaluated
piecewise or where a property holds at any size:
  * momentum and error at 20,000 sampled coordinates, bit-exact against the oracle's
    accumulate (or exactly zero where selected);
  * the merged table bit-equal to the fp32 tree of the GPU's worker tables;
  * one worker's first table row cell by cell against the oracle's sketch (VGG-16 size);
  * the estimate at the sampled coordinates, bit-exact against the oracle's median of the
    GPU's merged table (r odd);
  * the selected set equal to the exact top-k of the GPU's estimate (ties to the smaller
    index), checked in O(d);
  * gathered values against the exact fp64 sums of the pre-zeroing error vectors.
"""

import numpy as np
import pytest

torch = pytest.importorskip("torch")

import oracle  # noqa: E402
import workloads  # noqa: E402

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def gs():
    import paper_2108_06004_gb300 as lib
    lib.load_library()
    torch.cuda.set_device(0)
    return lib


@pytest.fixture(scope="module")
def H(gs):
    from tests import gpu_harness
    return gpu_harness


def test_step_resnet50_full_size(gs, H):
    from tests.test_gpu_parity import _run_steps
    w = workloads.get_config("resnet50")
    _run_steps(gs, H, w, w.d, 1)


def check_selection_linear(idx, est, k):
    """idx (ascending) is the top-k of |est| with ties to the smaller index, checked in O(d)."""
    key = est.view(np.uint32) & np.uint32(0x7FFFFFFF)
    assert idx.size == k and np.all(np.diff(idx) > 0)
    sel = np.zeros(key.size, dtype=bool)
    sel[idx] = True
    tau = key[idx].min()
    assert np.all(key[~sel] <= tau), "an unselected coordinate has a larger |est| than a selected one"
    assert np.all(sel[key > tau]), "a coordinate above the threshold is missing"
    eq = np.nonzero(key == tau)[0]
    n_eq_sel = int(sel[eq].sum())
    assert np.all(sel[eq[:n_eq_sel]]) and not np.any(sel[eq[n_eq_sel:]]), "ties not taken by smallest index"


@pytest.mark.parametrize("name,check_row", [("vgg16", True), ("bert-large", False)])
def test_step_large_sampled(gs, H, name, check_row):
    w = workloads.get_config(name)
    P, d, r, c, k, rho = w.P, w.d, w.r, w.c, w.k, w.rho
    batch = w.worker_batch or P
    seed = 77
    coeffs = oracle.derive_coefficients(r, seed)
    dev = torch.device("cuda")
    rng = np.random.default_rng(5)
    S = np.unique(np.concatenate([rng.integers(0, d, 20_000), [0, 1, 2, 3, d - 1, d - 2, d - 5]]))
    St = torch.from_numpy(S).to(dev)
    sk = gs.gs_sketch_create(r, c, seed, P, 0)
    info = gs.gs_sketch_info(sk)
    W = info["group_width"]
    assert batch % W == 0
    try:
        us = [torch.zeros(d, dtype=torch.float32, device=dev) for _ in range(P)]
        es = [torch.zeros(d, dtype=torch.float32, device=dev) for _ in range(P)]
        gbuf = [torch.empty(d, dtype=torch.float32, device=dev) for _ in range(batch)]
        g_at_S = []
        row_check = None
        gs.gs_sketch_zero(sk)
        for b0 in range(0, P, batch):
            for q in range(batch):
                workloads.make_gradient_torch(w, 0, b0 + q, gbuf[q])
                g_at_S.append(gbuf[q][St].cpu().numpy())
            gs.gs_accumulate_insert(sk, b0, us[b0:b0 + batch], es[b0:b0 + batch], gbuf, d, rho)
            if check_row and b0 == 0:
                torch.cuda.synchronize()
                row_check = es[0].cpu().numpy()
        del gbuf
        gs.gs_sketch_merge_tree(sk, P)
        ws = torch.empty(gs.gs_query_topk_workspace_size(d, k), dtype=torch.uint8, device=dev)
        idx = torch.empty(k, dtype=torch.int64, device=dev)
        est = torch.empty(d, dtype=torch.float32, device=dev)
        gs.gs_query_topk(sk, d, k, idx, est, ws)
        torch.cuda.synchronize()
        e_at_idx = np.stack([e[idx].cpu().numpy().astype(np.float64) for e in es])
        vals = torch.empty(k, dtype=torch.float32, device=dev)
        gs.gs_gather_and_zero(us, es, d, idx, k, vals)
        torch.cuda.synchronize()

        idx_h = idx.cpu().numpy()
        est_h = est.cpu().numpy()
        check_selection_linear(idx_h, est_h, k)

        # gathered values
        exact = e_at_idx.sum(axis=0)
        bound = (P - 1) * 2.0**-24 * np.abs(e_at_idx).sum(axis=0) * 1.000001
        assert np.all(np.abs(vals.cpu().numpy() - exact) <= bound)

        # momentum and error at the sampled coordinates
        selS = np.isin(S, idx_h)
        zero = np.zeros(S.size, np.float32)
        for p in range(P):
            u1, e1 = oracle.accumulate(zero, zero, g_at_S[p], rho)
            gu = us[p][St].cpu().numpy()
            ge = es[p][St].cpu().numpy()
            assert np.array_equal(gu[~selS].view(np.uint32), u1[~selS].view(np.uint32))
            assert np.array_equal(ge[~selS].view(np.uint32), e1[~selS].view(np.uint32))
            assert np.all(gu[selS] == 0) and np.all(ge[selS] == 0)

        # merge and estimate
        run = H.GpuRun(sk, [], [], d, k, rho, None, None, None, None)
        tabs = H.worker_tables(run, P, r, c)
        merged = H.merged_table(run, r, c)
        assert np.array_equal(merged, H.fp32_tree(tabs))
        est_o = oracle.query(merged.astype(np.float64), coeffs, S.size,
                             hashes=oracle.hash_rows(coeffs, c, S.astype(np.uint64)))
        assert np.array_equal(est_h[S].astype(np.float64), est_o)

        if row_check is not None:
            b, s = oracle.hash_rows((coeffs[0][:1], coeffs[1][:1], coeffs[2][:1], coeffs[3][:1]), c,
                                    np.arange(d, dtype=np.uint64))
            x64 = row_check.astype(np.float64)
            T0 = np.bincount(b[0], weights=s[0] * x64, minlength=c)
            A0 = np.bincount(b[0], weights=np.abs(x64), minlength=c)
            H.check_cells(tabs[0][0], T0, A0, "worker 0 row 0")
    finally:
        gs.gs_sketch_destroy(sk)
