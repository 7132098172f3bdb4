"""GPU parity: every call of the C ABI against the CPU oracle (run on a GB300).

Sizes span several CUDA tiles and ragged tails; the workload shapes are those of the
tiny (d = 2^20, P = 4) and ResNet-18-sized (d = 11,173,962, P = 8) configurations, plus
edge cases (d = 1, k = 1, k = d, c = 1, odd and even r, P not a power of two, every group
width, misaligned vectors).
"""

import numpy as np
import pytest

torch = pytest.importorskip("torch")

import oracle  # noqa: E402
import workloads  # noqa: E402

pytestmark = pytest.mark.gpu

P61 = (1 << 61) - 1


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


def _dev(x):
    return torch.from_numpy(np.ascontiguousarray(x)).cuda()


# ---- hash family ------------------------------------------------------------------------

@pytest.mark.parametrize("r,c,seed", [(5, 1 << 14, 20210813), (7, 1 << 20, 3), (3, 1000, 99), (16, 1, 0),
                                      (1, (1 << 26), 2**64 - 1)])
def test_coefficients_and_hashes_bit_exact(gs, r, c, seed):
    sk = gs.gs_sketch_create(r, c, seed, 1)
    try:
        coeffs = gs.gs_sketch_coefficients(sk)
        assert tuple(coeffs) == tuple(oracle.derive_coefficients(r, seed))
        rng = np.random.default_rng(seed % 1000)
        coords = np.concatenate([np.arange(1 << 16), [2**31 - 1, 2**31 - 2, 2**30, 11173961],
                                 rng.integers(0, 2**31, 200_000)]).astype(np.int64)
        n = coords.size
        bk = torch.empty(r * n, dtype=torch.int32, device="cuda")
        sg = torch.empty(r * n, dtype=torch.int8, device="cuda")
        gs.gs_hash_eval(sk, _dev(coords), n, bk, sg)
        want_b, want_s = oracle.hash_rows(coeffs, c, coords.astype(np.uint64))
        assert np.array_equal(bk.cpu().numpy().reshape(r, n), want_b)
        assert np.array_equal(sg.cpu().numpy().reshape(r, n), want_s)
        for t in (0, 1, n - 1, n - 2):
            for j in range(r):
                assert want_b[j, t] == oracle.bucket_exact(coeffs[0][j], coeffs[1][j], c, int(coords[t]))
        bad = _dev(np.array([-1, 2**31], dtype=np.int64))
        bk2 = torch.empty(r * 2, dtype=torch.int32, device="cuda")
        sg2 = torch.empty(r * 2, dtype=torch.int8, device="cuda")
        gs.gs_hash_eval(sk, bad, 2, bk2, sg2)
        assert np.all(bk2.cpu().numpy() == -1) and np.all(sg2.cpu().numpy() == 0)
    finally:
        gs.gs_sketch_destroy(sk)


# ---- step 1 ------------------------------------------------------------------------------

@pytest.mark.parametrize("d,offset", [(1, 0), (7, 0), (1_000_003, 0), (1_000_003, 1), (4096 * 152 * 3 + 2, 3)])
def test_accumulate_bit_exact(gs, d, offset):
    rng = np.random.default_rng(d + offset)
    mk = lambda: (rng.standard_normal(d) * 10.0 ** rng.integers(-30, 6, d)).astype(np.float32)
    u, e, g = mk(), mk(), mk()
    bufs = [torch.zeros(d + 4, dtype=torch.float32, device="cuda") for _ in range(3)]
    views = [b[offset:offset + d] for b in bufs]
    for v, x in zip(views, (u, e, g)):
        v.copy_(torch.from_numpy(x))
    for rho in (0.9, 0.0, 0.5):
        gs.gs_accumulate(views[0], views[1], views[2], d, rho)
        u, e = oracle.accumulate(u, e, g, rho)
        assert np.array_equal(views[0].cpu().numpy().view(np.uint32), u.view(np.uint32))
        assert np.array_equal(views[1].cpu().numpy().view(np.uint32), e.view(np.uint32))
    for b in bufs:  # guard cells outside the view untouched
        assert torch.all(b[:offset] == 0) and torch.all(b[offset + d:] == 0)


# ---- step 2 ------------------------------------------------------------------------------

@pytest.mark.parametrize("W,worker,P", [(1, 0, 1), (2, 1, 2), (4, 2, 3), (8, 5, 8), (8, 7, 13), (16, 11, 16)])
def test_single_vector_insert(gs, H, W, worker, P):
    d, r, c, seed = 300_001, 5, 1 << 12, 5
    rng = np.random.default_rng(W)
    x = (rng.standard_normal(d) * 1e-3).astype(np.float32)
    sk = gs.gs_sketch_create(r, c, seed, P, W)
    try:
        gs.gs_sketch_insert(sk, worker, _dev(x), d)
        run = H.GpuRun(sk, [], [], d, 1, 0.9, None, None, None, None)
        tabs = H.worker_tables(run, P, r, c)
        T, A = oracle.sketch(x, oracle.derive_coefficients(r, seed), c)
        H.check_cells(tabs[worker], T, A, "inserted table")
        for p in range(P):
            if p != worker:
                assert np.all(tabs[p] == 0)
    finally:
        gs.gs_sketch_destroy(sk)


@pytest.mark.parametrize("P,W,d,r,c,passes", [(1, 1, 70_001, 3, 1 << 10, 1), (3, 4, 123_457, 5, 1000, 1),
                                              (5, 8, 200_003, 4, 1 << 13, 1), (8, 2, 65_536, 5, 1 << 12, 1),
                                              (8, 8, 400_000, 7, 1 << 14, 1), (16, 8, 50_001, 5, 777, 1),
                                              (8, 0, 200_003, 3, 1 << 21, 3), (6, 0, 150_001, 5, 1 << 20, 5),
                                              (4, 0, 100_001, 7, 1 << 21, 7), (16, 16, 90_001, 5, 1 << 12, 1),
                                              (13, 0, 80_003, 3, 1 << 20, 3), (16, 0, 70_001, 5, 1 << 16, 1), (20, 16, 60_001, 4, 3001, 1),
                                              (8, 0, 90_001, 7, 1 << 19, 3)])
def test_accumulate_insert_merge(gs, H, P, W, d, r, c, passes):
    seed = P * 1000 + W
    rng = np.random.default_rng(seed)
    coeffs = oracle.derive_coefficients(r, seed)
    run = H.new_run(P, d, r, c, 1, seed, rho=0.9, group_width=W)
    try:
        info = gs.gs_sketch_info(run.sketch)
        if W:
            assert info["group_width"] == W
        W = info["group_width"]
        assert -(-r // info["rows_per_pass"]) == passes
        us = [(rng.standard_normal(d) * 1e-3).astype(np.float32) for _ in range(P)]
        es = [(rng.standard_normal(d) * 1e-3).astype(np.float32) for _ in range(P)]
        gr = [(rng.standard_normal(d) * 1e-3).astype(np.float32) for _ in range(P)]
        for p in range(P):
            run.us[p].copy_(torch.from_numpy(us[p]))
            run.es[p].copy_(torch.from_numpy(es[p]))
        gdev = [_dev(g) for g in gr]
        # two calls covering the workers in group-aligned pieces
        split = min(P, W) if P > W else P
        gs.gs_accumulate_insert(run.sketch, 0, run.us[:split], run.es[:split], gdev[:split], d, 0.9)
        if split < P:
            gs.gs_accumulate_insert(run.sketch, split, run.us[split:], run.es[split:], gdev[split:], d, 0.9)
        gs.gs_sketch_merge_tree(run.sketch, P)
        tabs = H.worker_tables(run, P, r, c)
        merged = H.merged_table(run, r, c)
        Ts, As = [], []
        for p in range(P):
            u1, e1 = oracle.accumulate(us[p], es[p], gr[p], 0.9)
            assert np.array_equal(H.host(run.us[p]).view(np.uint32), u1.view(np.uint32))
            assert np.array_equal(H.host(run.es[p]).view(np.uint32), e1.view(np.uint32))
            T, A = oracle.sketch(e1, coeffs, c)
            H.check_cells(tabs[p], T, A, f"worker {p}")
            Ts.append(T)
            As.append(A)
        assert np.array_equal(merged, H.fp32_tree(tabs)), "merge is not the fp32 tree of the worker tables"
        H.check_cells(merged, oracle.merge_tree(Ts), oracle.merge_tree(As), "merged")
        for Pm in range(1, P + 1):  # partial merges follow the same schedule
            gs.gs_sketch_merge_tree(run.sketch, Pm)
            assert np.array_equal(H.merged_table(run, r, c), H.fp32_tree(tabs[:Pm]))
    finally:
        run.close()


@pytest.mark.parametrize("P,W,d,r,c", [(4, 0, 1 << 20, 5, 1 << 14), (3, 4, 123_457, 5, 1000), (8, 8, 200_003, 3, 4096),
                                       (16, 16, 90_001, 5, 1 << 12), (2, 1, 70_001, 4, 50_000), (9, 0, 65_537, 7, 3001)])
def test_accumulate_insert_staged(gs, H, P, W, d, r, c):
    """The shared-memory-staged insert: momentum and error bit-exact against the oracle's
    accumulate, every worker-table cell within 1e-5 of its magnitude of the oracle's sketch, and
    the same rejection as documented where a row does not fit a shared-memory tile."""
    seed = P * 100 + r
    rng = np.random.default_rng(seed)
    coeffs = oracle.derive_coefficients(r, seed)
    run = H.new_run(P, d, r, c, 1, seed, rho=0.9, group_width=W)
    try:
        W = gs.gs_sketch_info(run.sketch)["group_width"]
        us = [(rng.standard_normal(d) * 1e-3).astype(np.float32) for _ in range(P)]
        es = [(rng.standard_normal(d) * 1e-3).astype(np.float32) for _ in range(P)]
        gr = [(rng.standard_normal(d) * 1e-3).astype(np.float32) for _ in range(P)]
        for p in range(P):
            run.us[p].copy_(torch.from_numpy(us[p]))
            run.es[p].copy_(torch.from_numpy(es[p]))
        gdev = [_dev(g) for g in gr]
        split = W if P > W else P
        gs.gs_accumulate_insert_staged(run.sketch, 0, run.us[:split], run.es[:split], gdev[:split], d, 0.9)
        if split < P:
            gs.gs_accumulate_insert_staged(run.sketch, split, run.us[split:], run.es[split:], gdev[split:], d, 0.9)
        tabs = H.worker_tables(run, P, r, c)
        for p in range(P):
            u1, e1 = oracle.accumulate(us[p], es[p], gr[p], 0.9)
            assert np.array_equal(H.host(run.us[p]).view(np.uint32), u1.view(np.uint32))
            assert np.array_equal(H.host(run.es[p]).view(np.uint32), e1.view(np.uint32))
            T, A = oracle.sketch(e1, coeffs, c)
            H.check_cells(tabs[p], T, A, f"worker {p}")
    finally:
        run.close()


def test_accumulate_insert_staged_rejects_large_rows(gs, H):
    run = H.new_run(2, 4096, 3, 1 << 16, 1, 3)
    try:
        with pytest.raises(gs.GsError) as ei:
            gs.gs_accumulate_insert_staged(run.sketch, 0, run.us, run.es, run.es, 4096, 0.9)
        assert ei.value.status == gs.GS_ERR_INVALID_ARG
    finally:
        run.close()


@pytest.mark.parametrize("P,d,r,c", [(1, 10_007, 3, 512), (5, 100_003, 5, 4096), (13, 50_001, 4, 1000), (64, 20_011, 3, 256)])
def test_merge_separate_sketches(gs, H, P, d, r, c):
    """P sketches created one per worker (the problem statement's form of the merge): the merged
    table of sketches[0] is bit-equal to the fp32 tree of their tables in the schedule's order and
    within 1e-5*A of the oracle's fp64 tree of the workers' sketches; mismatched families and a
    repeated sketch are rejected."""
    seed = 900 + P
    rng = np.random.default_rng(seed)
    coeffs = oracle.derive_coefficients(r, seed)
    sks = [gs.gs_sketch_create(r, c, seed, 1, 0) for _ in range(P)]
    other = gs.gs_sketch_create(r, c, seed + 1, 1, 0)
    try:
        xs = [(rng.standard_normal(d) * 1e-3).astype(np.float32) for _ in range(P)]
        for sk, x in zip(sks, xs):
            gs.gs_sketch_insert(sk, 0, _dev(x), d)
        gs.gs_sketch_merge_sketches(sks)
        tabs = []
        for sk in sks:
            buf = np.empty(r * c, np.float32)
            gs.gs_sketch_copy_to_host(sk, 0, buf)
            tabs.append(buf.reshape(r, c))
        merged = np.empty(r * c, np.float32)
        gs.gs_sketch_copy_to_host(sks[0], -1, merged)
        assert np.array_equal(merged.reshape(r, c), H.fp32_tree(tabs))
        ors = [oracle.sketch(x, coeffs, c) for x in xs]
        H.check_cells(merged.reshape(r, c), oracle.merge_tree([t for t, _ in ors]),
                      oracle.merge_tree([a for _, a in ors]), "merged")
        with pytest.raises(gs.GsError) as ei:
            gs.gs_sketch_merge_sketches(sks[:1] + [other])
        assert ei.value.status == gs.GS_ERR_MISMATCH
        with pytest.raises(gs.GsError) as ei:
            gs.gs_sketch_merge_sketches([sks[0], sks[0]])
        assert ei.value.status == gs.GS_ERR_INVALID_ARG
    finally:
        for sk in sks + [other]:
            gs.gs_sketch_destroy(sk)


def test_accumulate_insert_unaligned(gs, H):
    """Vectors that start 4 bytes past a 16-byte boundary take the scalar load path of the
    fused kernel; the state stays bit-exact and the tables agree with the oracle."""
    P, d, r, c, seed = 5, 100_003, 5, 4096, 77
    rng = np.random.default_rng(seed)
    coeffs = oracle.derive_coefficients(r, seed)
    sk = gs.gs_sketch_create(r, c, seed, P, 0)
    try:
        bufs = [[torch.zeros(d + 4, dtype=torch.float32, device="cuda") for _ in range(3)] for _ in range(P)]
        views = [[b[1:d + 1] for b in trio] for trio in bufs]
        host = []
        for p in range(P):
            u, e, g = [(rng.standard_normal(d) * 1e-2).astype(np.float32) for _ in range(3)]
            for v, x in zip(views[p], (u, e, g)):
                v.copy_(torch.from_numpy(x))
            host.append((u, e, g))
        gs.gs_sketch_zero(sk)
        gs.gs_accumulate_insert(sk, 0, [v[0] for v in views], [v[1] for v in views], [v[2] for v in views], d, 0.9)
        gs.gs_sketch_merge_tree(sk, P)
        torch.cuda.synchronize()
        Ts, As = [], []
        for p in range(P):
            u1, e1 = oracle.accumulate(*host[p], 0.9)
            assert np.array_equal(views[p][0].cpu().numpy().view(np.uint32), u1.view(np.uint32))
            assert np.array_equal(views[p][1].cpu().numpy().view(np.uint32), e1.view(np.uint32))
            T, A = oracle.sketch(e1, coeffs, c)
            buf = np.empty(r * c, dtype=np.float32)
            gs.gs_sketch_copy_to_host(sk, p, buf)
            H.check_cells(buf.reshape(r, c), T, A, f"worker {p}")
            Ts.append(T)
            As.append(A)
        buf = np.empty(r * c, dtype=np.float32)
        gs.gs_sketch_copy_to_host(sk, -1, buf)
        H.check_cells(buf.reshape(r, c), oracle.merge_tree(Ts), oracle.merge_tree(As), "merged")
        # the guard words around each view are untouched
        for trio in bufs:
            for b in trio[:2]:
                edge = b.cpu().numpy()
                assert edge[0] == 0 and np.all(edge[d + 1:] == 0)
    finally:
        gs.gs_sketch_destroy(sk)


# ---- steps 4-5 ---------------------------------------------------------------------------

@pytest.mark.parametrize("d,r,c,k", [(1, 5, 64, 1), (10, 3, 1, 4), (1000, 1, 1, 1000), (100_003, 5, 4096, 1),
                                     (100_003, 4, 4096, 333), (1 << 20, 5, 1 << 14, 1000),
                                     (500_000, 7, 3000, 500_000), (2_000_001, 15, 1 << 16, 2000)])
def test_query_topk(gs, H, d, r, c, k):
    seed = d + r + c + k
    rng = np.random.default_rng(seed % 2**32)
    coeffs = oracle.derive_coefficients(r, seed)
    x = (rng.standard_normal(d) * 1e-3).astype(np.float32)
    x[rng.choice(d, max(1, d // 500), replace=False)] *= 100
    run = H.new_run(1, d, r, c, k, seed)
    try:
        gs.gs_sketch_insert(run.sketch, 0, _dev(x), d)
        gs.gs_sketch_merge_tree(run.sketch, 1)
        ws = torch.empty(gs.gs_query_topk_workspace_size(d, k), dtype=torch.uint8, device="cuda")
        gs.gs_query_topk(run.sketch, d, k, run.idx, run.est, ws)
        est, idx = H.host(run.est), H.host(run.idx)
        T, A = oracle.sketch(x, coeffs, c)
        est_o = oracle.query(T, coeffs, d)
        band = oracle.cell_band(A, coeffs, np.arange(d))
        assert np.all(np.abs(est.astype(np.float64) - est_o) <= band)
        H.check_selection_exact(idx, est, k)
        H.check_topk_set(idx, oracle.topk(est_o, k), est_o, band, k, d)
        # without est_out the same indices come out
        idx2 = torch.empty(k, dtype=torch.int64, device="cuda")
        gs.gs_query_topk(run.sketch, d, k, idx2, None, ws)
        assert np.array_equal(H.host(idx2), idx)
    finally:
        run.close()


@pytest.mark.parametrize("d,k,nonzero", [(3_000_001, 5000, False), (2_500_003, 7777, True)])
def test_topk_large_plateau(gs, H, d, k, nonzero):
    """Millions of equal keys: every coordinate is a selection candidate, more than any
    block-local buffer holds.  With c = 1 and r = 1 every coordinate shares one cell, so
    |est| is the same nonzero value everywhere; the top-k is then the k smallest indices."""
    r, c = (1, 1) if nonzero else (5, 4096)
    run = H.new_run(1, d, r, c, k, 3)
    try:
        if nonzero:
            x = np.random.default_rng(9).standard_normal(d).astype(np.float32)
            gs.gs_sketch_insert(run.sketch, 0, _dev(x), d)
        gs.gs_sketch_merge_tree(run.sketch, 1)
        ws = torch.empty(gs.gs_query_topk_workspace_size(d, k), dtype=torch.uint8, device="cuda")
        gs.gs_query_topk(run.sketch, d, k, run.idx, run.est, ws)
        est = H.host(run.est)
        assert np.unique(np.abs(est)).size == 1 and ((est[0] != 0) == nonzero)
        assert np.array_equal(H.host(run.idx), np.arange(k))
    finally:
        run.close()


SAMPLE_PERIOD = 256   # the query's prune-key sample: the first four coordinates of every 256


def _prune_input(rng, d, k, adversarial):
    """A vector with k heavy coordinates over N(0, 1e-2^2) noise.  Natural: the heavy
    coordinates sit at random positions.  Adversarial: all of them sit on the query's sample
    (coordinates i with i mod 256 < 4), with magnitudes spread over two decades, so that the
    sample's rank puts the prune key far above the k-th largest |est| and the repair must run."""
    x = (rng.standard_normal(d) * 1e-2).astype(np.float32)
    if adversarial:
        pos = (np.arange(k) // 4) * SAMPLE_PERIOD + (np.arange(k) % 4)
        assert pos[-1] < d
    else:
        pos = rng.choice(d, k, replace=False)
    mag = np.exp(rng.uniform(0.0, np.log(100.0), k)).astype(np.float32)
    x[pos] = mag * rng.choice(np.array([-1.0, 1.0], np.float32), k)
    return x


def _check_pruned_against_full(H, got, e_int, want, e, k, r):
    assert np.array_equal(got, want), "selections differ"
    H.check_selection_exact(got, e, k)
    pruned, _ = H.pruned_rows(e_int, r)
    exact = e_int.view(np.uint32) == e.view(np.uint32)
    assert np.all(pruned | exact)
    tau = np.sort(np.abs(e))[-k]
    assert np.all(np.abs(e[pruned]) < tau) and not pruned[got].any()
    return pruned


@pytest.mark.parametrize("r,adversarial", [(5, False), (5, True), (4, False), (4, True), (7, False), (7, True),
                                           (3, False), (3, True)])
def test_pruned_query_matches_full_query(gs, H, r, adversarial):
    """Queries whose estimate stays in the workspace skip rows below a prune key that the query
    takes from a strided sample of its own estimate.  On natural input the key is safe and most
    coordinates stop after r/2 + 1 rows; on adversarial input (every heavy coordinate on the
    sample) the key lies above the k-th largest |est|, and the repair pass must restore every
    skipped estimate.  Either way the selection equals the full query's exactly, every selected
    estimate is exact, and every skipped one (a marker naming the rows it read) lies below the
    k-th largest |est|."""
    d, c, k, seed = 4_200_007, 1 << 16, 4000, 40 + r      # pruning applies from d = 2^22
    rng = np.random.default_rng(seed)
    sk = gs.gs_sketch_create(r, c, seed, 1, 0)
    try:
        ws = torch.empty(gs.gs_query_topk_workspace_size(d, k), dtype=torch.uint8, device="cuda")
        est_int = ws[: 4 * d].view(torch.float32)   # the query keeps its estimate at the workspace start
        idx = torch.empty(k, dtype=torch.int64, device="cuda")
        idx_full = torch.empty(k, dtype=torch.int64, device="cuda")
        est_full = torch.empty(d, dtype=torch.float32, device="cuda")
        x = _prune_input(rng, d, k, adversarial)
        gs.gs_sketch_zero(sk)
        gs.gs_sketch_insert(sk, 0, _dev(x), d)
        gs.gs_sketch_merge_tree(sk, 1)
        for t in range(2):   # the same query twice: nothing carries over from the first
            gs.gs_query_topk(sk, d, k, idx, None, ws)           # internal estimate: may prune
            torch.cuda.synchronize()
            got, e_int = H.host(idx).copy(), H.host(est_int).copy()
            gs.gs_query_topk(sk, d, k, idx_full, est_full, ws)  # caller's estimate: every row
            torch.cuda.synchronize()
            pruned = _check_pruned_against_full(H, got, e_int, H.host(idx_full), H.host(est_full), k, r)
            if adversarial:
                assert not pruned.any(), "the repair left skipped estimates"
            else:
                assert pruned.mean() > 0.5, f"only {pruned.mean():.3f} of the coordinates skipped rows"
    finally:
        gs.gs_sketch_destroy(sk)


@pytest.mark.parametrize("k,r,c", [(1, 5, 1 << 16), (7, 5, 1 << 16), (1_400_002, 5, 1 << 16), (1, 7, 1 << 18),
                                   (1_400_002, 7, 1 << 18)])
def test_pruned_query_extreme_k(gs, H, k, r, c):
    """Pruning queries at the extremes of k (one coordinate; a third of them), on the kernel that
    classifies the first rows in shared memory (c = 2^16) and on the one that reads them
    (r = 7, c = 2^18): the selection equals the full query's, every selected estimate is exact,
    and every marker lies below the k-th largest |est|."""
    d, seed = 4_200_007, 70 + k % 97 + r
    rng = np.random.default_rng(seed)
    sk = gs.gs_sketch_create(r, c, seed, 1, 0)
    try:
        ws = torch.empty(gs.gs_query_topk_workspace_size(d, k), dtype=torch.uint8, device="cuda")
        idx = torch.empty(k, dtype=torch.int64, device="cuda")
        idx_full = torch.empty(k, dtype=torch.int64, device="cuda")
        est_full = torch.empty(d, dtype=torch.float32, device="cuda")
        gs.gs_sketch_insert(sk, 0, _dev(_prune_input(rng, d, min(k, 4000), False)), d)
        gs.gs_sketch_merge_tree(sk, 1)
        gs.gs_query_topk(sk, d, k, idx, None, ws)
        torch.cuda.synchronize()
        got, e_int = H.host(idx).copy(), H.host(ws[: 4 * d].view(torch.float32)).copy()
        gs.gs_query_topk(sk, d, k, idx_full, est_full, ws)
        torch.cuda.synchronize()
        _check_pruned_against_full(H, got, e_int, H.host(idx_full), H.host(est_full), k, r)
    finally:
        gs.gs_sketch_destroy(sk)


def test_pruned_queries_on_two_streams(gs, H):
    """Queries of one sketch on two streams at once, each with its own workspace, one on natural
    and one on adversarial data (a second sketch), interleaved launch after launch: a query keeps
    its prune key in its own workspace, so every selection equals the full query's."""
    d, r, c, k = 4_200_007, 5, 1 << 16, 4000
    rng = np.random.default_rng(17)
    sks = [gs.gs_sketch_create(r, c, 17, 1, 0) for _ in range(2)]
    streams = [torch.cuda.Stream(), torch.cuda.Stream()]
    try:
        for sk, adv in zip(sks, (False, True)):
            gs.gs_sketch_insert(sk, 0, _dev(_prune_input(rng, d, k, adv)), d)
            gs.gs_sketch_merge_tree(sk, 1)
        wss = [torch.empty(gs.gs_query_topk_workspace_size(d, k), dtype=torch.uint8, device="cuda") for _ in range(4)]
        want = []
        for sk in sks:
            idx_full = torch.empty(k, dtype=torch.int64, device="cuda")
            gs.gs_query_topk(sk, d, k, idx_full, torch.empty(d, dtype=torch.float32, device="cuda"), wss[0])
            torch.cuda.synchronize()
            want.append(H.host(idx_full).copy())
        torch.cuda.synchronize()
        idxs = [[torch.empty(k, dtype=torch.int64, device="cuda") for _ in range(12)] for _ in range(2)]
        for n in range(12):
            for q in range(2):
                # stream q alternates between the two sketches; each stream uses its own workspaces
                gs.gs_query_topk(sks[(n + q) % 2], d, k, idxs[q][n], None, wss[2 * q + (n % 2)], None,
                                 streams[q])
        torch.cuda.synchronize()
        for q in range(2):
            for n in range(12):
                assert np.array_equal(H.host(idxs[q][n]), want[(n + q) % 2]), f"stream {q}, query {n}"
    finally:
        for sk in sks:
            gs.gs_sketch_destroy(sk)


def _settle_threshold(v, f):
    """Per column of v (rows x coordinates, the signed cells in the order the query reads them):
    the least t0 such that every t > t0 has at least f values < t and at least f values > -t,
    i.e. the larger of the f-th smallest value and minus the f-th largest."""
    srt = np.sort(v, axis=0)
    return np.maximum(srt[f - 1], -srt[v.shape[0] - f])


@pytest.mark.parametrize("r,c", [(3, 1 << 16), (4, 1 << 16), (5, 1 << 16), (7, 1 << 16), (16, 1 << 16),
                                 (5, 1 << 19), (7, 1 << 18)])
def test_pruned_rows_follow_the_rule(gs, H, r, c):
    """The rows each coordinate examined, from its marker, against the rule, with the signed cells
    recomputed on the host from the merged table and the hash values: one prune key t must
    exist such that every coordinate that stopped after n rows was settled by its first n cells
    (t above their settle threshold) and unsettled by its first n - 1 when n > r/2 + 1, and
    every coordinate that examined all r rows was unsettled by its first r - 1.  The cells read
    are those the header states: all n examined ones, or, where the classes of the first
    f = r/2 + 1 rows fit in 192 KiB of shared memory (the first five cases), n - f."""
    d, k, seed = 4_200_007, 4000, 60 + r
    f = r // 2 + 1
    rng = np.random.default_rng(seed)
    sk = gs.gs_sketch_create(r, c, seed, 1, 0)
    try:
        ws = torch.empty(gs.gs_query_topk_workspace_size(d, k), dtype=torch.uint8, device="cuda")
        idx = torch.empty(k, dtype=torch.int64, device="cuda")
        gs.gs_sketch_insert(sk, 0, _dev(_prune_input(rng, d, k, False)), d)
        gs.gs_sketch_merge_tree(sk, 1)
        gs.gs_query_topk(sk, d, k, idx, None, ws)
        torch.cuda.synchronize()
        e_int = H.host(ws[: 4 * d].view(torch.float32)).copy()
        pruned, n = H.pruned_rows(e_int, r)
        g = ((e_int.view(np.uint32)[pruned] >> np.uint32(5)) & np.uint32(31)).astype(np.int64)
        assert np.array_equal(g, n - f if f * c // 4 <= 192 << 10 else n), "cells read differ from the header"
        # markers name f <= n < r rows, so for r = 4 every one names 3
        assert pruned.mean() > 0.5 and (r - 1 == f or np.any(n > f)), "coordinates should stop at several row counts"
        T = np.empty(r * c, np.float32)
        gs.gs_sketch_copy_to_host(sk, -1, T)
        T = T.reshape(r, c)
        bk = torch.empty(r * d, dtype=torch.int32, device="cuda")
        sg = torch.empty(r * d, dtype=torch.int8, device="cuda")
        gs.gs_hash_eval(sk, _dev(np.arange(d, dtype=np.int64)), d, bk, sg)
        bk, sg = H.host(bk).reshape(r, d), H.host(sg).reshape(r, d)
        v = T[np.arange(r)[:, None], bk] * sg.astype(np.float32)   # exact: a sign flip
        lo, hi = 0.0, np.inf            # the prune key must satisfy lo < t <= hi
        for rows in range(f, r + 1):
            at = np.nonzero(pruned)[0][n == rows] if rows < r else np.nonzero(~pruned)[0]
            if at.size == 0:
                continue
            if rows < r:
                lo = max(lo, float(_settle_threshold(v[:rows, at], f).max()))
            if rows > f:
                hi = min(hi, float(_settle_threshold(v[:rows - 1, at], f).min()))
        assert lo < hi, f"no prune key explains the rows read: settled below {lo}, unsettled from {hi}"
    finally:
        gs.gs_sketch_destroy(sk)


def test_no_pruning_below_4m_coordinates(gs, H):
    """Under 2^22 coordinates a query reads every row: its internal estimate equals the full one."""
    d, r, c, k = (1 << 22) - 1, 5, 1 << 14, 500
    rng = np.random.default_rng(8)
    sk = gs.gs_sketch_create(r, c, 8, 1, 0)
    try:
        gs.gs_sketch_insert(sk, 0, _dev((rng.standard_normal(d) * 1e-2).astype(np.float32)), d)
        gs.gs_sketch_merge_tree(sk, 1)
        ws = torch.empty(gs.gs_query_topk_workspace_size(d, k), dtype=torch.uint8, device="cuda")
        idx = torch.empty(k, dtype=torch.int64, device="cuda")
        est = torch.empty(d, dtype=torch.float32, device="cuda")
        for _ in range(2):
            gs.gs_query_topk(sk, d, k, idx, None, ws)
        torch.cuda.synchronize()
        e_int = H.host(ws[: 4 * d].view(torch.float32)).copy()
        gs.gs_query_topk(sk, d, k, idx, est, ws)
        torch.cuda.synchronize()
        assert np.array_equal(e_int.view(np.uint32), H.host(est).view(np.uint32))
    finally:
        gs.gs_sketch_destroy(sk)


def test_topk_all_ties_and_zeros(gs, H):
    d, r, c, k = 50_000, 5, 256, 1234
    run = H.new_run(1, d, r, c, k, 1)
    try:
        ws = torch.empty(gs.gs_query_topk_workspace_size(d, k), dtype=torch.uint8, device="cuda")
        gs.gs_sketch_merge_tree(run.sketch, 1)           # all-zero sketch: est = 0 everywhere
        gs.gs_query_topk(run.sketch, d, k, run.idx, run.est, ws)
        assert np.array_equal(H.host(run.idx), np.arange(k))
    finally:
        run.close()


# ---- step 6 ------------------------------------------------------------------------------

@pytest.mark.parametrize("P,d,k", [(1, 10, 10), (2, 1001, 57), (3, 5003, 100), (4, 1_000_003, 1000),
                                   (9, 20_001, 333), (17, 10_007, 99), (33, 12_345, 500), (64, 20_000, 777)])
def test_gather_and_zero(gs, P, d, k):
    rng = np.random.default_rng(P)
    us = [(rng.standard_normal(d)).astype(np.float32) for _ in range(P)]
    es = [(rng.standard_normal(d)).astype(np.float32) for _ in range(P)]
    idx = np.sort(rng.choice(d, k, replace=False)).astype(np.int64)
    ud, ed = [_dev(u) for u in us], [_dev(e) for e in es]
    vals = torch.empty(k, dtype=torch.float32, device="cuda")
    gs.gs_gather_and_zero(ud, ed, d, _dev(idx), k, vals)
    v, us2, es2 = oracle.gather_and_zero(us, es, idx)
    stack = np.stack([e[idx].astype(np.float64) for e in es])
    assert np.all(np.abs(vals.cpu().numpy() - v) <= (P - 1) * 2.0**-24 * np.abs(stack).sum(0) * 1.000001)
    # the fp32 sum in worker order, exactly
    ref = np.zeros(k, np.float32)
    for e in es:
        ref = (ref + e[idx]).astype(np.float32)
    assert np.array_equal(vals.cpu().numpy(), ref)
    for p in range(P):
        assert np.array_equal(ud[p].cpu().numpy(), us2[p]) and np.array_equal(ed[p].cpu().numpy(), es2[p])


def test_gather_skips_out_of_range(gs):
    d = 100
    u = [torch.ones(d, device="cuda")]
    e = [torch.ones(d, device="cuda")]
    idx = _dev(np.array([-5, 3, 100, 2**40], dtype=np.int64))
    vals = torch.empty(4, device="cuda")
    gs.gs_gather_and_zero(u, e, d, idx, 4, vals)
    v = vals.cpu().numpy()
    assert np.isnan(v[0]) and v[1] == 1.0 and np.isnan(v[2]) and np.isnan(v[3])
    assert float(u[0].sum()) == d - 1 and float(e[0][3]) == 0.0


# ---- whole steps -------------------------------------------------------------------------

def _run_steps(gs, H, w, d, steps, c=None, k=None, r=None, P=None, group_width=0, seed=2021):
    P = P or w.P
    r = r or w.r
    c = c or w.c
    k = k or w.k
    coeffs = oracle.derive_coefficients(r, seed)
    run = H.new_run(P, d, r, c, k, seed, rho=w.rho, group_width=group_width)
    nsym = 0
    try:
        for t in range(steps):
            grads = workloads.make_gradients(w, t, range(P), d=d)
            gdev = [_dev(g) for g in grads]
            us0 = [H.host(u) for u in run.us]
            es0 = [H.host(e) for e in run.es]
            H.gpu_step(run, gdev)
            torch.cuda.synchronize()
            res = oracle.step(us0, es0, grads, w.rho, coeffs, c, k)
            nsym += H.compare_step(res, coeffs, [H.host(u) for u in run.us], [H.host(e) for e in run.es],
                                   H.host(run.idx), H.host(run.vals), H.host(run.est), k,
                                   H.worker_tables(run, P, r, c), H.merged_table(run, r, c))
    finally:
        run.close()
    return nsym


def test_steps_tiny_config(gs, H):
    w = workloads.get_config("tiny-2^20")
    _run_steps(gs, H, w, w.d, w.steps)


@pytest.mark.parametrize("P,r,c,k,W", [(5, 4, 1000, 777, 0), (6, 3, 4099, 50, 2), (3, 5, 1 << 12, 1, 1),
                                       (9, 5, 2048, 100, 0)])
def test_steps_ragged(gs, H, P, r, c, k, W):
    w = workloads.get_config("resnet18")
    _run_steps(gs, H, w, 100_003, 2, c=c, k=k, r=r, P=P, group_width=W)


def test_steps_resnet18_full_size(gs, H):
    w = workloads.get_config("resnet18")
    _run_steps(gs, H, w, w.d, 2)


@pytest.mark.parametrize("kind", ["pinned", "pageable", "device"])
def test_step_host_buffers(gs, H, kind):
    """gs_step_host with gradients in pinned host memory, in plain (pageable) numpy arrays and
    in device memory; results returned to host buffers."""
    w = workloads.get_config("resnet18")
    P, d, r, c, k, seed = 5, 300_001, 5, 4096, 300, 41
    coeffs = oracle.derive_coefficients(r, seed)
    run = H.new_run(P, d, r, c, k, seed, rho=w.rho)
    try:
        gdev_buf = [torch.empty(d, dtype=torch.float32, device="cuda") for _ in range(P)]
        idx_h = torch.empty(k, dtype=torch.int64).pin_memory()
        vals_h = torch.empty(k, dtype=torch.float32).pin_memory()
        for t in range(2):
            grads = workloads.make_gradients(w, t, range(P), d=d)
            if kind == "pinned":
                src = [torch.from_numpy(g).pin_memory() for g in grads]
            elif kind == "pageable":
                src = [np.ascontiguousarray(g) for g in grads]
            else:
                src = [_dev(g) for g in grads]
            ptrs = [s.ctypes.data if isinstance(s, np.ndarray) else s for s in src]
            us0 = [H.host(u) for u in run.us]
            es0 = [H.host(e) for e in run.es]
            gs.gs_step_host(run.sketch, run.us, run.es, ptrs, gdev_buf, d, w.rho, k, idx_h, vals_h, run.ws)
            res = oracle.step(us0, es0, grads, w.rho, coeffs, c, k)
            idx = idx_h.numpy().copy()
            band = oracle.cell_band(res.merged_abs, coeffs, np.arange(d))
            H.check_topk_set(idx, res.idx, res.est, band, k, d)
            H.check_state([H.host(u) for u in run.us], [H.host(e) for e in run.es], res, idx)
            H.check_vals(vals_h.numpy().copy(), idx, res.es_pre)
    finally:
        run.close()


@pytest.mark.parametrize("r", [5, 4, 7])
def test_internal_estimate_query_matches(gs, H, r):
    """Steps whose estimate stays in the workspace (est_out = NULL) select exactly what a
    query returning the estimate selects on the same merged table, and agree with the oracle,
    also across a step where the state is cleared and the threshold collapses."""
    w = workloads.get_config("resnet18")
    P, d, c, k, seed = 4, 400_003, 1 << 13, 500, 91
    coeffs = oracle.derive_coefficients(r, seed)
    run = H.new_run(P, d, r, c, k, seed, rho=w.rho)
    try:
        ws_q = torch.empty(gs.gs_query_topk_workspace_size(d, k), dtype=torch.uint8, device="cuda")
        idx_exact = torch.empty(k, dtype=torch.int64, device="cuda")
        for t in range(5):
            grads = workloads.make_gradients(w, t, range(P), d=d)
            if t == 3:  # collapse the state and the gradients: the threshold falls far below the hint
                for u, e in zip(run.us, run.es):
                    u.zero_()
                    e.zero_()
                grads = [(g * np.float32(1e-3)).astype(np.float32) for g in grads]
            us0 = [H.host(u) for u in run.us]
            es0 = [H.host(e) for e in run.es]
            gs.gs_step(run.sketch, run.us, run.es, [_dev(g) for g in grads], d, w.rho, k, run.idx, run.vals,
                       None, run.ws)
            gs.gs_query_topk(run.sketch, d, k, idx_exact, run.est, ws_q)   # same merged table, est returned
            torch.cuda.synchronize()
            idx = H.host(run.idx)
            assert np.array_equal(idx, H.host(idx_exact)), f"step {t}: selections differ"
            H.check_selection_exact(idx, H.host(run.est), k)
            res = oracle.step(us0, es0, grads, w.rho, coeffs, c, k)
            band = oracle.cell_band(res.merged_abs, coeffs, np.arange(d))
            H.check_topk_set(idx, res.idx, res.est, band, k, d)
            H.check_state([H.host(u) for u in run.us], [H.host(e) for e in run.es], res, idx)
            H.check_vals(H.host(run.vals), idx, res.es_pre)
    finally:
        run.close()


# ---- step 7: weight update (Alg. 1 step 26) ------------------------------------------------

def test_apply_update_bit_exact(gs):
    rng = np.random.default_rng(77)
    d, k = 1_000_003, 5000
    w = (rng.standard_normal(d) * 10.0 ** rng.integers(-5, 3, d)).astype(np.float32)
    idx = np.sort(rng.choice(d, k, replace=False)).astype(np.int64)
    vals = (rng.standard_normal(k) * 10.0 ** rng.integers(-8, 2, k)).astype(np.float32)
    wd = _dev(w)
    gs.gs_apply_update(wd, d, _dev(idx), _dev(vals), k, 0.03)
    want = oracle.apply_update(w, idx, vals, 0.03)
    assert np.array_equal(wd.cpu().numpy().view(np.uint32), want.view(np.uint32))
    # indices outside [0, d) are skipped
    w2 = _dev(np.ones(10, np.float32))
    gs.gs_apply_update(w2, 10, _dev(np.array([-1, 3, 10], np.int64)), _dev(np.ones(3, np.float32)), 3, 1.0)
    assert w2.cpu().numpy().tolist() == [1, 1, 1, 0, 1, 1, 1, 1, 1, 1]


def test_gather_zero_update_fused(gs):
    rng = np.random.default_rng(78)
    P, d, k, lr = 6, 200_001, 777, 0.1
    us = [(rng.standard_normal(d)).astype(np.float32) for _ in range(P)]
    es = [(rng.standard_normal(d)).astype(np.float32) for _ in range(P)]
    w = rng.standard_normal(d).astype(np.float32)
    idx = np.sort(rng.choice(d, k, replace=False)).astype(np.int64)
    ud, ed, wd = [_dev(u) for u in us], [_dev(e) for e in es], _dev(w)
    vals = torch.empty(k, dtype=torch.float32, device="cuda")
    gs.gs_gather_zero_update(ud, ed, d, _dev(idx), k, vals, wd, lr)
    ref = np.zeros(k, np.float32)
    for e in es:
        ref = (ref + e[idx]).astype(np.float32)
    assert np.array_equal(vals.cpu().numpy(), ref)
    want = oracle.apply_update(w, idx, ref, lr)
    assert np.array_equal(wd.cpu().numpy().view(np.uint32), want.view(np.uint32))
    _, us2, es2 = oracle.gather_and_zero(us, es, idx)
    for p in range(P):
        assert np.array_equal(ud[p].cpu().numpy(), us2[p]) and np.array_equal(ed[p].cpu().numpy(), es2[p])


def test_train_steps(gs, H):
    """Alg. 1 end to end for the simulated workers: compression step plus weight update."""
    w_cfg = workloads.get_config("resnet18")
    P, d, r, c, k, seed, lr = 8, 250_001, 5, 1 << 12, 250, 17, 0.05
    coeffs = oracle.derive_coefficients(r, seed)
    run = H.new_run(P, d, r, c, k, seed, rho=w_cfg.rho)
    try:
        w = _dev(np.random.default_rng(3).standard_normal(d).astype(np.float32))
        for t in range(3):
            grads = workloads.make_gradients(w_cfg, t, range(P), d=d)
            us0 = [H.host(u) for u in run.us]
            es0 = [H.host(e) for e in run.es]
            w0 = H.host(w)
            gs.gs_train_step(run.sketch, w, lr, run.us, run.es, [_dev(g) for g in grads], d, w_cfg.rho, k, run.idx,
                             run.vals, run.est, run.ws)
            torch.cuda.synchronize()
            res = oracle.step(us0, es0, grads, w_cfg.rho, coeffs, c, k)
            idx, vals = H.host(run.idx), H.host(run.vals)
            H.compare_step(res, coeffs, [H.host(u) for u in run.us], [H.host(e) for e in run.es], idx, vals,
                           H.host(run.est), k)
            want = oracle.apply_update(w0, idx, vals, lr)
            assert np.array_equal(H.host(w).view(np.uint32), want.view(np.uint32))
    finally:
        run.close()


# ---- HEAVYMIX (Alg. 2 as printed) ----------------------------------------------------------

@pytest.mark.parametrize("r,k,spikes", [(5, 4000, 800), (4, 3000, 5000), (7, 20000, 300)])
def test_heavymix_pruned_matches_full(gs, H, r, k, spikes):
    """From 2^22 coordinates a HEAVYMIX query with an internal estimate skips the rows of
    coordinates whose first r/2 + 1 cells bound est^2 below l2sq / k: they lie outside H and
    enter the selection only through the random fill.  The selection equals the query that
    returns every estimate, and rows were in fact skipped."""
    d, c, seed, fill_seed = 4_200_007, 1 << 16, 17 + r, 2**62 + 3
    rng = np.random.default_rng(seed)
    x = (rng.standard_normal(d) * 1e-3).astype(np.float32)
    x[rng.choice(d, spikes, replace=False)] *= np.float32(60.0)
    sk = gs.gs_sketch_create(r, c, seed, 1, 0)
    try:
        gs.gs_sketch_insert(sk, 0, _dev(x), d)
        gs.gs_sketch_merge_tree(sk, 1)
        ws = torch.empty(gs.gs_query_heavymix_workspace_size(d, k), dtype=torch.uint8, device="cuda")
        l2 = torch.empty(2, dtype=torch.float64, device="cuda")
        idx_full = torch.empty(k, dtype=torch.int64, device="cuda")
        idx = torch.empty(k, dtype=torch.int64, device="cuda")
        est = torch.empty(d, dtype=torch.float32, device="cuda")
        gs.gs_query_heavymix(sk, d, k, fill_seed, idx_full, est, l2[0:1], ws)
        gs.gs_query_heavymix(sk, d, k, fill_seed, idx, None, l2[1:2], ws)
        torch.cuda.synchronize()
        e_int = H.host(ws[: 4 * d].view(torch.float32))
        assert np.array_equal(H.host(idx), H.host(idx_full))
        l2h = H.host(l2)
        assert abs(l2h[0] - l2h[1]) <= 1e-12 * l2h[0]   # fp64 atomic sums: order varies
        assert np.array_equal(H.host(idx_full), oracle.heavymix_select(H.host(est), float(l2h[0]), k, fill_seed))
        pruned, _ = H.pruned_rows(e_int, r)
        assert pruned.mean() > 0.2, "rows were not skipped"
        e = H.host(est).astype(np.float64)
        assert np.all(e[pruned] ** 2 < l2h[0] / k)
    finally:
        gs.gs_sketch_destroy(sk)


@pytest.mark.parametrize("d,r,c,k,spikes,scale", [(400_003, 5, 1 << 12, 300, 40, 50.0),
                                                  (400_003, 5, 1 << 12, 5, 40, 50.0),
                                                  (250_001, 4, 3001, 2000, 10, 20.0),
                                                  (1 << 20, 7, 1 << 14, 1000, 5243, 100.0)])
def test_heavymix(gs, H, d, r, c, k, spikes, scale):
    seed, fill_seed = d % 1000 + r, 2**63 + 12345
    rng = np.random.default_rng(seed)
    x = (rng.standard_normal(d) * 1e-3).astype(np.float32)
    x[rng.choice(d, spikes, replace=False)] *= np.float32(scale)
    coeffs = oracle.derive_coefficients(r, seed)
    run = H.new_run(1, d, r, c, k, seed)
    try:
        gs.gs_sketch_insert(run.sketch, 0, _dev(x), d)
        gs.gs_sketch_merge_tree(run.sketch, 1)
        ws = torch.empty(gs.gs_query_heavymix_workspace_size(d, k), dtype=torch.uint8, device="cuda")
        l2 = torch.empty(1, dtype=torch.float64, device="cuda")
        gs.gs_query_heavymix(run.sketch, d, k, fill_seed, run.idx, run.est, l2, ws)
        torch.cuda.synchronize()
        idx, est, l2sq = H.host(run.idx), H.host(run.est), float(l2.item())
        merged = H.merged_table(run, r, c).astype(np.float64)
        rows = np.sort((merged ** 2).sum(axis=1))
        want_l2 = rows[r // 2] if r % 2 else 0.5 * (rows[r // 2 - 1] + rows[r // 2])
        assert abs(l2sq - want_l2) <= 1e-12 * want_l2
        # exact: the selection rule applied to the GPU's own estimate and l2sq
        assert np.array_equal(idx, oracle.heavymix_select(est, l2sq, k, fill_seed))
        # against the fp64 oracle: the same l2sq within the cell tolerance, est within its band
        T, A = oracle.sketch(x, coeffs, c)
        _, est_o, l2_o = oracle.heavymix(T, coeffs, d, k, fill_seed)
        assert abs(l2sq - l2_o) <= 1e-4 * l2_o
        band = oracle.cell_band(A, coeffs, np.arange(d))
        assert np.all(np.abs(est.astype(np.float64) - est_o) <= band)
        _check_heavymix_against_oracle(H, idx, est, l2sq, est_o, l2_o, band, k, fill_seed)
    finally:
        run.close()


def _check_heavymix_against_oracle(H, idx, est, l2sq, est_o, l2_o, band, k, fill_seed):
    """The GPU's HEAVYMIX selection against the fp64 oracle's.  H may differ only at the
    threshold band (|est_o| within the cell band of sqrt(l2sq / k), widened by the l2sq
    difference).  With |H| < k the selection is H plus the fill, and the fill order (xi_i, i)
    is fixed by the indices alone: the expected set is the oracle's rule applied to the
    oracle's H with only the band coordinates taken as the GPU placed them, so the fill must
    match exactly (with no flip this is the oracle's own selection).  With |H| >= k it is the
    top-k of H by |est|, equal to the oracle's except within the tie band."""
    h_gpu = oracle.heavymix_members(est, l2sq, k)
    h_o = oracle.heavymix_members(est_o, l2_o, k)
    thr = np.sqrt(l2_o / k)
    slack = abs(np.sqrt(l2sq / k) - thr)
    flip = np.nonzero(h_gpu != h_o)[0]
    edge = np.abs(np.abs(est_o[flip]) - thr) <= band[flip] + slack
    assert np.all(edge), f"H differs away from the threshold at {flip[~edge][:5]}"
    if h_gpu.sum() < k:
        h_exp = h_o.copy()
        h_exp[flip] = h_gpu[flip]          # the band coordinates are the only free choices
        want = oracle.heavymix_select_from(h_exp, est_o, k, fill_seed)
        assert np.array_equal(idx, want), "the fill differs from the oracle's fill order"
    else:
        masked_o = np.where(h_o, est_o, 0.0)
        H.check_topk_set(idx, oracle.topk(masked_o, k), masked_o, band + slack, k, est_o.size)


def _random_step_configs(n, seed=2108):
    """Seeded draws of small step shapes: P in 1..20, d up to 300,000 (often ragged), r in 1..9,
    c a power of two or not, k from 1 to d, and every group width the library accepts."""
    rng = np.random.default_rng(seed)
    out = []
    for _ in range(n):
        P = int(rng.integers(1, 21))
        d = int(rng.choice([rng.integers(1, 100), rng.integers(100, 300_001)]))
        r = int(rng.integers(1, 10))
        c = int(2 ** rng.integers(0, 16)) if rng.random() < 0.6 else int(rng.integers(1, 40_000))
        k = int(rng.integers(1, d + 1)) if rng.random() < 0.3 else int(min(d, rng.integers(1, 2000)))
        W = int(rng.choice([0, 0, 1, 2, 4, 8, 16]))
        out.append((P, d, r, c, k, W))
    return out


@pytest.mark.parametrize("P,d,r,c,k,W", _random_step_configs(16))
def test_random_step_shapes(gs, H, P, d, r, c, k, W):
    """Two steps of randomly drawn shapes against the oracle, with every agreement check of the
    step tests (tables, merged table, estimate band, selection, state, gathered values)."""
    w = workloads.get_config("tiny-2^20")
    _run_steps(gs, H, w, d, 2, c=c, k=k, r=r, P=P, group_width=W, seed=d % 997 + r)
