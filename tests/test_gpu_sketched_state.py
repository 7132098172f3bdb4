"""GPU parity for the variant that keeps momentum and error as r x c sketches (Sec. II: a
linear sketch can carry momentum and error accumulation itself).

Agreement:
  * per-index query of a table: the same median of the same fp32 cells as the oracle (odd r
    exactly; even r within the rounding of the fp32 mean), and equal to the full query's
    estimate at those coordinates;
  * sparse signed insert: cells within rel * A of the oracle's fp64 sketch (fp32 atomics in
    any order);
  * one step: the workers' merged sketch S within rel * A_S; the selection within the tie
    band of the oracle's estimate from E; the extracted values within the estimate band;
    U and E after the removal within rel * (A + the removed magnitude), plus, for U, the
    band of its own estimate at each removed coordinate (that estimate is an fp32 median);
    the weights exactly fl(w - fl(lr * delta)).
The oracle is fed the GPU's state before every step, so each step is checked on its own.
"""

from __future__ import annotations

import numpy as np
import pytest
import torch

import oracle

pytestmark = pytest.mark.gpu

REL = 1e-5


@pytest.fixture(scope="module")
def gs():
    import paper_2108_06004_gb300 as lib
    lib.load_library()
    return lib


def _dev(x):
    return torch.from_numpy(np.ascontiguousarray(x)).to("cuda")


def _table(gs, sk, r, c):
    buf = np.empty(r * c, dtype=np.float32)
    gs.gs_sketch_copy_to_host(sk, -1, buf)
    return buf.reshape(r, c)


@pytest.mark.parametrize("r,c", [(5, 4096), (4, 1000), (1, 64), (7, 3001)])
def test_query_at(gs, r, c):
    d, seed = 50_000, 11 + r
    rng = np.random.default_rng(seed)
    x = rng.standard_normal(d).astype(np.float32)
    sk = gs.gs_sketch_create(r, c, seed, 1, 0)
    try:
        gs.gs_sketch_insert(sk, 0, _dev(x), d)
        gs.gs_sketch_merge_tree(sk, 1)
        coords = np.concatenate([[0, d - 1, 2**31 - 1], rng.integers(0, d, 997)]).astype(np.int64)
        out = torch.empty(coords.size, dtype=torch.float32, device="cuda")
        gs.gs_sketch_query_at(sk, _dev(coords), coords.size, out)
        k = 10
        ws = torch.empty(gs.gs_query_topk_workspace_size(d, k), dtype=torch.uint8, device="cuda")
        idx = torch.empty(k, dtype=torch.int64, device="cuda")
        est = torch.empty(d, dtype=torch.float32, device="cuda")
        gs.gs_query_topk(sk, d, k, idx, est, ws)
        bad = torch.empty(2, dtype=torch.float32, device="cuda")
        gs.gs_sketch_query_at(sk, _dev(np.array([-1, 2**31], dtype=np.int64)), 2, bad)
        torch.cuda.synchronize()
        got = out.cpu().numpy()
        T = _table(gs, sk, r, c)
        co = oracle.derive_coefficients(r, seed)
        want = oracle.query_at(T.astype(np.float64), co, coords)
        if r % 2:
            assert np.array_equal(got.astype(np.float64), want)
        else:
            assert np.all(np.abs(got - want) <= 2.0 ** -24 * np.abs(want))
        # the per-index query and the full query agree at every in-range coordinate
        inr = coords < d
        assert np.array_equal(got[inr], est.cpu().numpy()[coords[inr]])
        assert np.all(np.isnan(bad.cpu().numpy()))
    finally:
        gs.gs_sketch_destroy(sk)


@pytest.mark.parametrize("r,c,k,scale", [(5, 4096, 3000, -1.0), (3, 257, 20000, 0.75), (6, 64, 1, 2.0)])
def test_add_sparse(gs, r, c, k, scale):
    seed = 7 * r + k
    rng = np.random.default_rng(seed)
    d = 4 * k + 5
    idx = np.sort(rng.choice(d, k, replace=False)).astype(np.int64)
    vals = rng.standard_normal(k).astype(np.float32)
    sk = gs.gs_sketch_create(r, c, seed, 1, 0)
    try:
        gs.gs_sketch_zero(sk)
        gs.gs_sketch_add_sparse(sk, _dev(idx), _dev(vals), k, scale)
        # out-of-range coordinates touch nothing
        gs.gs_sketch_add_sparse(sk, _dev(np.array([-3, 2**31 + 5], dtype=np.int64)),
                                _dev(np.ones(2, np.float32)), 2, 1.0)
        torch.cuda.synchronize()
        co = oracle.derive_coefficients(r, seed)
        T, A = oracle.sketch_sparse(idx, np.float64(np.float32(scale)) * vals.astype(np.float64), co, c)
        err = np.abs(_table(gs, sk, r, c).astype(np.float64) - T)
        assert np.all(err <= REL * A), float((err - REL * A).max())
    finally:
        gs.gs_sketch_destroy(sk)


def test_sketched_state_rejects_mismatch(gs):
    a = gs.gs_sketch_create(5, 1024, 1, 2, 0)
    b = gs.gs_sketch_create(5, 1024, 1, 1, 0)
    e = gs.gs_sketch_create(5, 1024, 2, 1, 0)
    try:
        d, k = 1000, 10
        g = [torch.zeros(d, device="cuda") for _ in range(2)]
        ws = torch.empty(gs.gs_step_workspace_size(d, k), dtype=torch.uint8, device="cuda")
        idx = torch.empty(k, dtype=torch.int64, device="cuda")
        vals = torch.empty(k, device="cuda")
        with pytest.raises(gs.GsError):
            gs.gs_sketched_state_step(a, b, e, g, d, 0.9, k, idx, vals, None, 0.0, ws)
        with pytest.raises(gs.GsError):
            gs.gs_sketched_state_step(a, b, b, g, d, 0.9, k, idx, vals, None, 0.0, ws)
    finally:
        for s in (a, b, e):
            gs.gs_sketch_destroy(s)


def _run_steps(gs, P, d, r, c, k, steps, rho, lr, seed, group_width=0):
    rng = np.random.default_rng(seed)
    co = oracle.derive_coefficients(r, seed)
    wk = gs.gs_sketch_create(r, c, seed, P, group_width)
    U = gs.gs_sketch_create(r, c, seed, 1, 0)
    E = gs.gs_sketch_create(r, c, seed, 1, 0)
    try:
        gs.gs_sketch_zero(U)
        gs.gs_sketch_zero(E)
        ws = torch.empty(gs.gs_step_workspace_size(d, k), dtype=torch.uint8, device="cuda")
        idx = torch.empty(k, dtype=torch.int64, device="cuda")
        vals = torch.empty(k, dtype=torch.float32, device="cuda")
        w0 = rng.standard_normal(d).astype(np.float32)
        w = _dev(w0)
        AU = np.zeros((r, c))
        AE = np.zeros((r, c))
        ties = 0
        for _ in range(steps):
            gsn = [(rng.standard_normal(d) * rng.uniform(0.5, 2.0)).astype(np.float32) for _ in range(P)]
            for p in range(P):  # a few large coordinates per worker, shared across workers
                gsn[p][rng.integers(0, d, 8)] += np.float32(30.0)
            U_prev = _table(gs, U, r, c).astype(np.float64)
            E_prev = _table(gs, E, r, c).astype(np.float64)
            w_prev = w.cpu().numpy()
            gs.gs_sketched_state_step(wk, U, E, [_dev(g) for g in gsn], d, rho, k, idx, vals, w, lr, ws)
            torch.cuda.synchronize()
            res = oracle.sketched_state_step(U_prev, E_prev, AU, AE, gsn, rho, co, c, k, REL)
            gi, gv = idx.cpu().numpy(), vals.cpu().numpy()
            # S: the tree-merged sketch of the raw gradients
            S = _table(gs, wk, r, c).astype(np.float64)
            assert np.all(np.abs(S - res.S) <= REL * res.AS)
            # selection and extracted values
            ties += oracle_tie_check(gi, res, k, d)
            assert np.all(np.abs(gv.astype(np.float64) - res.est[gi]) <= res.band[gi])
            # E after the removal of S(delta) at the GPU's selection with the GPU's values
            SD, AD = oracle.sketch_sparse(gi, gv.astype(np.float64), co, c)
            E_gpu = _table(gs, E, r, c).astype(np.float64)
            assert np.all(np.abs(E_gpu - (res.E_pre - SD)) <= REL * (res.AE_pre + AD))
            # U after the removal of S(delta_u), delta_u its own estimate at the selection
            du = oracle.query_at(res.U_pre, co, gi)
            SDu, ADu = oracle.sketch_sparse(gi, du, co, c)
            bu = oracle.cell_band(res.AU_pre, co, gi, REL)
            _, Abu = oracle.sketch_sparse(gi, bu, co, c)
            U_gpu = _table(gs, U, r, c).astype(np.float64)
            assert np.all(np.abs(U_gpu - (res.U_pre - SDu)) <= REL * (res.AU_pre + ADu) + Abu)
            # weights: exactly fl(w - fl(lr * delta)) at the selection
            want = w_prev.copy()
            want[gi] = (w_prev[gi] - np.float32(lr) * gv).astype(np.float32)
            assert np.array_equal(w.cpu().numpy().view(np.uint32), want.view(np.uint32))
            AU, AE = res.AU_pre + ADu, res.AE_pre + AD
        return ties
    finally:
        for s in (wk, U, E):
            gs.gs_sketch_destroy(s)


def oracle_tie_check(gi, res, k, d):
    assert gi.size == k and np.all(np.diff(gi) > 0) and gi[0] >= 0 and gi[-1] < d
    sym = np.setxor1d(gi, res.idx)
    if sym.size == 0:
        return 0
    a = np.abs(res.est)
    kth = res.idx[np.argmin(a[res.idx])]
    off = np.abs(a[sym] - a[kth]) > res.band[sym] + res.band[kth]
    assert not off.any(), f"selection differs outside the tie band at {sym[off][:8]}"
    return int(sym.size)


@pytest.mark.parametrize("P,d,r,c,k,steps,gw", [
    (4, 20_000, 5, 2048, 50, 4, 0),
    (3, 100_003, 5, 8192, 400, 3, 0),
    (8, 65_536, 4, 4096, 200, 3, 8),
    (6, 31_337, 3, 1500, 100, 3, 2),
    (1, 4_099, 7, 256, 1, 2, 0),
    (4, 4_200_001, 5, 1 << 16, 4000, 3, 0),   # from 2^22 coordinates the query skips rows
])
def test_sketched_state_steps(gs, P, d, r, c, k, steps, gw):
    _run_steps(gs, P, d, r, c, k, steps, rho=0.9, lr=0.05, seed=d % 977 + P, group_width=gw)


def test_sketched_state_resnet18_size(gs):
    """Full ResNet-18 length (11,173,962 coordinates) for P = 4 workers, one step, with the
    sketch and k of the main workload."""
    _run_steps(gs, 4, 11_173_962, 5, 1 << 20, 111_739, 1, rho=0.9, lr=0.01, seed=5)
