"""Plans: a whole step captured into a CUDA graph and launched many times.

A plan launch must give what the direct call gives: the same agreement with the oracle,
step after step, with the gradients refilled in place between launches (the plan holds
pointers, not data).  Also checked: the timed insert phase yields one positive duration per
launch, the host-buffer plan returns its results to host memory after a stream
synchronisation, and the sketched-state plan follows the oracle like the direct call.
"""

from __future__ import annotations

import numpy as np
import pytest
import torch

import oracle
import workloads

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def gs():
    import paper_2108_06004_gb300 as lib
    lib.load_library()
    return lib


@pytest.fixture(scope="module")
def H(gs):
    from tests import gpu_harness
    return gpu_harness


def _dev(x):
    return torch.from_numpy(np.ascontiguousarray(x)).to("cuda")


@pytest.mark.parametrize("P,d,r,c,k,W,train", [
    (4, 100_003, 5, 8192, 300, 0, False),
    (6, 65_537, 3, 4099, 50, 2, True),
    (8, 1 << 20, 5, 1 << 14, 1000, 0, False),
])
def test_step_plan(gs, H, P, d, r, c, k, W, train):
    w = workloads.get_config("resnet18")
    seed, lr = 29 + P, 0.05
    coeffs = oracle.derive_coefficients(r, seed)
    run = H.new_run(P, d, r, c, k, seed, rho=w.rho, group_width=W)
    gbuf = [torch.empty(d, dtype=torch.float32, device="cuda") for _ in range(P)]
    weights = _dev(np.random.default_rng(5).standard_normal(d).astype(np.float32)) if train else None
    plan = gs.gs_step_plan_create(run.sketch, run.us, run.es, gbuf, d, w.rho, k, run.idx, run.vals, run.est,
                                  weights, lr, run.ws, flags=gs.GS_PLAN_TIME_INSERT)
    try:
        steps = 3
        for t in range(steps):
            grads = workloads.make_gradients(w, t, range(P), d=d)
            for b, g in zip(gbuf, grads):
                b.copy_(torch.from_numpy(g))
            us0 = [H.host(u) for u in run.us]
            es0 = [H.host(e) for e in run.es]
            w0 = H.host(weights) if train else None
            gs.gs_plan_launch(plan)
            torch.cuda.synchronize()
            res = oracle.step(us0, es0, grads, w.rho, coeffs, c, k)
            gi, gv = H.host(run.idx), H.host(run.vals)
            H.compare_step(res, coeffs, [H.host(u) for u in run.us], [H.host(e) for e in run.es], gi, gv,
                           H.host(run.est), k, H.worker_tables(run, P, r, c), H.merged_table(run, r, c))
            if train:
                want = w0.copy()
                want[gi] = (w0[gi] - np.float32(lr) * gv).astype(np.float32)
                assert np.array_equal(H.host(weights).view(np.uint32), want.view(np.uint32))
        times = gs.gs_plan_insert_times(plan, 100)
        assert len(times) == steps and all(t > 0 for t in times)
    finally:
        gs.gs_plan_destroy(plan)
        run.close()


def test_step_plan_untimed_rejects_times(gs, H):
    run = H.new_run(2, 4096, 3, 256, 8, 3)
    g = [torch.zeros(4096, device="cuda") for _ in range(2)]
    plan = gs.gs_step_plan_create(run.sketch, run.us, run.es, g, 4096, 0.9, 8, run.idx, run.vals, None, None, 0.0,
                                  run.ws)
    try:
        gs.gs_plan_launch(plan)
        with pytest.raises(gs.GsError):
            gs.gs_plan_insert_times(plan, 4)
    finally:
        gs.gs_plan_destroy(plan)
        run.close()


def test_step_plan_ring_keeps_last_launches(gs, H):
    """More launches than the ring holds: the times of the last 1024 are returned."""
    run = H.new_run(2, 8192, 3, 512, 16, 4)
    g = [torch.randn(8192, device="cuda") for _ in range(2)]
    plan = gs.gs_step_plan_create(run.sketch, run.us, run.es, g, 8192, 0.9, 16, run.idx, run.vals, None, None, 0.0,
                                  run.ws, flags=gs.GS_PLAN_TIME_INSERT)
    try:
        for _ in range(1100):
            gs.gs_plan_launch(plan)
        times = gs.gs_plan_insert_times(plan, 2000)
        assert len(times) == 1024 and all(t > 0 for t in times)
    finally:
        gs.gs_plan_destroy(plan)
        run.close()


def test_step_host_plan(gs, H):
    w = workloads.get_config("resnet18")
    P, d, r, c, k, seed = 5, 300_001, 5, 4096, 300, 43
    coeffs = oracle.derive_coefficients(r, seed)
    run = H.new_run(P, d, r, c, k, seed, rho=w.rho)
    host = [torch.empty(d, dtype=torch.float32).pin_memory() for _ in range(P)]
    gdev = [torch.empty(d, dtype=torch.float32, device="cuda") for _ in range(P)]
    idx_h = torch.empty(k, dtype=torch.int64).pin_memory()
    vals_h = torch.empty(k, dtype=torch.float32).pin_memory()
    plan = gs.gs_step_host_plan_create(run.sketch, run.us, run.es, host, gdev, d, w.rho, k, idx_h, vals_h, run.ws,
                                       flags=gs.GS_PLAN_TIME_INSERT)
    try:
        for t in range(3):
            grads = workloads.make_gradients(w, t, range(P), d=d)
            for hb, g in zip(host, grads):
                hb.copy_(torch.from_numpy(g))
            us0 = [H.host(u) for u in run.us]
            es0 = [H.host(e) for e in run.es]
            gs.gs_plan_launch(plan)
            torch.cuda.current_stream().synchronize()
            res = oracle.step(us0, es0, grads, w.rho, coeffs, c, k)
            idx, vals = idx_h.numpy().copy(), vals_h.numpy().copy()
            band = oracle.cell_band(res.merged_abs, coeffs, np.arange(d))
            H.check_topk_set(idx, res.idx, res.est, band, k, d)
            H.check_state([H.host(u) for u in run.us], [H.host(e) for e in run.es], res, idx)
            H.check_vals(vals, idx, res.es_pre)
    finally:
        gs.gs_plan_destroy(plan)
        run.close()


def test_sketched_state_plan(gs):
    P, d, r, c, k, seed, rho, lr, rel = 4, 50_000, 5, 2048, 100, 77, 0.9, 0.05, 1e-5
    rng = np.random.default_rng(seed)
    co = oracle.derive_coefficients(r, seed)
    wk = gs.gs_sketch_create(r, c, seed, P, 0)
    U = gs.gs_sketch_create(r, c, seed, 1, 0)
    E = gs.gs_sketch_create(r, c, seed, 1, 0)
    gs.gs_sketch_zero(U)
    gs.gs_sketch_zero(E)
    gbuf = [torch.empty(d, dtype=torch.float32, device="cuda") for _ in range(P)]
    ws = torch.empty(gs.gs_step_workspace_size(d, k), dtype=torch.uint8, device="cuda")
    idx = torch.empty(k, dtype=torch.int64, device="cuda")
    vals = torch.empty(k, dtype=torch.float32, device="cuda")
    weights = _dev(rng.standard_normal(d).astype(np.float32))
    plan = gs.gs_sketched_state_plan_create(wk, U, E, gbuf, d, rho, k, idx, vals, weights, lr, ws,
                                            flags=gs.GS_PLAN_TIME_INSERT)

    def table(sk):
        buf = np.empty(r * c, dtype=np.float32)
        gs.gs_sketch_copy_to_host(sk, -1, buf)
        return buf.reshape(r, c).astype(np.float64)

    try:
        AU = np.zeros((r, c))
        AE = np.zeros((r, c))
        for t in range(3):
            grads = [rng.standard_normal(d).astype(np.float32) for _ in range(P)]
            for p in range(P):
                grads[p][rng.integers(0, d, 5)] += np.float32(25.0)
            for b, g in zip(gbuf, grads):
                b.copy_(torch.from_numpy(g))
            U0, E0, w0 = table(U), table(E), weights.cpu().numpy()
            gs.gs_plan_launch(plan)
            torch.cuda.synchronize()
            res = oracle.sketched_state_step(U0, E0, AU, AE, grads, rho, co, c, k, rel)
            gi, gv = idx.cpu().numpy(), vals.cpu().numpy()
            assert np.all(np.diff(gi) > 0) and gi.size == k
            sym = np.setxor1d(gi, res.idx)
            if sym.size:
                a = np.abs(res.est)
                kth = res.idx[np.argmin(a[res.idx])]
                assert np.all(np.abs(a[sym] - a[kth]) <= res.band[sym] + res.band[kth])
            assert np.all(np.abs(gv.astype(np.float64) - res.est[gi]) <= res.band[gi])
            SD, AD = oracle.sketch_sparse(gi, gv.astype(np.float64), co, c)
            assert np.all(np.abs(table(E) - (res.E_pre - SD)) <= rel * (res.AE_pre + AD))
            want = w0.copy()
            want[gi] = (w0[gi] - np.float32(lr) * gv).astype(np.float32)
            assert np.array_equal(weights.cpu().numpy().view(np.uint32), want.view(np.uint32))
            du = oracle.query_at(res.U_pre, co, gi)
            _, ADu = oracle.sketch_sparse(gi, du, co, c)
            AU, AE = res.AU_pre + ADu, res.AE_pre + AD
        assert len(gs.gs_plan_insert_times(plan, 10)) == 3
    finally:
        gs.gs_plan_destroy(plan)
        for s in (wk, U, E):
            gs.gs_sketch_destroy(s)


def test_step_plan_resnet18_full_size(gs, H):
    """The launch configuration bench.py times: the ResNet-18-sized workload (d = 11,173,962,
    P = 8, r = 5, c = 2^17, k = 11,200) stepped through a plan, two steps, every output
    compared with the oracle."""
    w = workloads.get_config("resnet18")
    P, d, r, c, k, seed = w.P, w.d, w.r, w.c, w.k, 20210813
    coeffs = oracle.derive_coefficients(r, seed)
    run = H.new_run(P, d, r, c, k, seed, rho=w.rho)
    gbuf = [torch.empty(d, dtype=torch.float32, device="cuda") for _ in range(P)]
    plan = gs.gs_step_plan_create(run.sketch, run.us, run.es, gbuf, d, w.rho, k, run.idx, run.vals, run.est,
                                  flags=gs.GS_PLAN_TIME_INSERT, workspace=run.ws)
    try:
        for t in range(2):
            grads = workloads.make_gradients(w, t, range(P))
            for b, g in zip(gbuf, grads):
                b.copy_(torch.from_numpy(g))
            us0 = [H.host(u) for u in run.us]
            es0 = [H.host(e) for e in run.es]
            gs.gs_plan_launch(plan)
            torch.cuda.synchronize()
            res = oracle.step(us0, es0, grads, w.rho, coeffs, c, k)
            H.compare_step(res, coeffs, [H.host(u) for u in run.us], [H.host(e) for e in run.es], H.host(run.idx),
                           H.host(run.vals), H.host(run.est), k, H.worker_tables(run, P, r, c),
                           H.merged_table(run, r, c))
    finally:
        gs.gs_plan_destroy(plan)
        run.close()


def test_step_plan_with_row_pruning(gs, H):
    """A plan whose estimate stays internal, at a size where the query skips rows (d >= 2^22):
    after every launch the selection equals a full query of the same merged table, and the
    gathered values are the exact fp32 sums of the accumulated error vectors."""
    w = workloads.get_config("resnet18")
    P, d, r, c, k, seed = 4, 4_500_001, 5, 1 << 16, 4000, 91
    run = H.new_run(P, d, r, c, k, seed, rho=w.rho)
    gbuf = [torch.empty(d, dtype=torch.float32, device="cuda") for _ in range(P)]
    plan = gs.gs_step_plan_create(run.sketch, run.us, run.es, gbuf, d, w.rho, k, run.idx, run.vals, None,
                                  workspace=run.ws)
    ws2 = torch.empty(gs.gs_query_topk_workspace_size(d, k), dtype=torch.uint8, device="cuda")
    idx_full = torch.empty(k, dtype=torch.int64, device="cuda")
    est_full = torch.empty(d, dtype=torch.float32, device="cuda")
    try:
        for t in range(4):
            grads = workloads.make_gradients(w, t, range(P), d=d)
            for b, g in zip(gbuf, grads):
                b.copy_(torch.from_numpy(g))
            us0 = [H.host(u) for u in run.us]
            es0 = [H.host(e) for e in run.es]
            gs.gs_plan_launch(plan)
            gs.gs_query_topk(run.sketch, d, k, idx_full, est_full, ws2)
            torch.cuda.synchronize()
            gi = H.host(run.idx)
            assert np.array_equal(gi, H.host(idx_full)), f"launch {t}: selection differs from the full query"
            H.check_selection_exact(gi, H.host(est_full), k)
            e_int = H.host(run.ws[: 4 * d].view(torch.float32))   # the plan's internal estimate
            pruned, _ = H.pruned_rows(e_int, r)
            assert pruned.mean() > 0.3, f"launch {t}: rows were not skipped"
            es_pre = [oracle.accumulate(u0, e0, g, w.rho)[1] for u0, e0, g in zip(us0, es0, grads)]
            ref = np.zeros(k, np.float32)
            for e in es_pre:
                ref = (ref + e[gi]).astype(np.float32)
            assert np.array_equal(H.host(run.vals).view(np.uint32), ref.view(np.uint32))
    finally:
        gs.gs_plan_destroy(plan)
        run.close()


def test_step_plan_repairs_a_prune_key_above_the_threshold(gs, H):
    """Inside a plan the repair of a too-high prune key runs as a graph node.  The first launch
    gets ordinary gradients (the key is safe); the second, from cleared state, gets gradients
    whose heavy coordinates all lie on the query's prune-key sample (coordinates i with
    i mod 256 < 4), so the sampled key lies above the k-th largest |est| and every skipped
    estimate must be recomputed."""
    w = workloads.get_config("resnet18")
    P, d, r, c, k, seed = 2, 4_300_001, 5, 1 << 16, 3000, 93
    run = H.new_run(P, d, r, c, k, seed, rho=w.rho)
    gbuf = [torch.empty(d, dtype=torch.float32, device="cuda") for _ in range(P)]
    plan = gs.gs_step_plan_create(run.sketch, run.us, run.es, gbuf, d, w.rho, k, run.idx, run.vals, None,
                                  workspace=run.ws)
    ws2 = torch.empty(gs.gs_query_topk_workspace_size(d, k), dtype=torch.uint8, device="cuda")
    idx_full = torch.empty(k, dtype=torch.int64, device="cuda")
    est_full = torch.empty(d, dtype=torch.float32, device="cuda")
    rng = np.random.default_rng(93)
    try:
        for t in range(2):
            grads = workloads.make_gradients(w, t, range(P), d=d)
            if t == 1:
                pos = (np.arange(k) // 4) * 256 + (np.arange(k) % 4)
                grads[0][pos] = np.exp(rng.uniform(0.0, np.log(100.0), k)).astype(np.float32)
            for b, g in zip(gbuf, grads):
                b.copy_(torch.from_numpy(g))
            for u, e in zip(run.us, run.es):
                u.zero_()
                e.zero_()
            gs.gs_plan_launch(plan)
            torch.cuda.synchronize()
            gi = H.host(run.idx).copy()
            e_int = H.host(run.ws[: 4 * d].view(torch.float32))
            gs.gs_query_topk(run.sketch, d, k, idx_full, est_full, ws2)
            torch.cuda.synchronize()
            assert np.array_equal(gi, H.host(idx_full)), f"launch {t}: selection differs from the full query"
            pruned, _ = H.pruned_rows(e_int, r)
            if t == 0:
                assert pruned.mean() > 0.3, "rows were not skipped"
            else:        # repaired: every estimate is the full one
                assert np.array_equal(e_int.view(np.uint32), H.host(est_full).view(np.uint32))
            ref = np.zeros(k, np.float32)
            for g in grads:   # from cleared state, e = u = g
                ref = (ref + g[gi]).astype(np.float32)
            assert np.array_equal(H.host(run.vals).view(np.uint32), ref.view(np.uint32))
    finally:
        gs.gs_plan_destroy(plan)
        run.close()


def test_step_plan_query_times(gs, H):
    """GS_PLAN_TIME_QUERY: one positive median-query and selection duration per launch; a plan
    created without the flag rejects the request."""
    run = H.new_run(2, 8192, 3, 512, 16, 4)
    g = [torch.randn(8192, device="cuda") for _ in range(2)]
    flags = gs.GS_PLAN_TIME_INSERT | gs.GS_PLAN_TIME_QUERY
    plan = gs.gs_step_plan_create(run.sketch, run.us, run.es, g, 8192, 0.9, 16, run.idx, run.vals, None, None, 0.0,
                                  run.ws, flags=flags)
    plain = gs.gs_step_plan_create(run.sketch, run.us, run.es, g, 8192, 0.9, 16, run.idx, run.vals, None, None, 0.0,
                                   run.ws, flags=gs.GS_PLAN_TIME_INSERT)
    try:
        for _ in range(5):
            gs.gs_plan_launch(plan)
        q, s = gs.gs_plan_query_times(plan, 10)
        assert len(q) == len(s) == 5 and all(x > 0 for x in q + s)
        assert len(gs.gs_plan_insert_times(plan, 10)) == 5
        gs.gs_plan_launch(plain)
        with pytest.raises(gs.GsError):
            gs.gs_plan_query_times(plain, 4)
    finally:
        gs.gs_plan_destroy(plan)
        gs.gs_plan_destroy(plain)
        run.close()


def test_heavymix_step_and_plan(gs, H):
    """A step with the HEAVYMIX selection, first through gs_heavymix_step and then twice through
    its plan (gradients refilled in place), each against the fp64 oracle: momentum and error
    bit-exact off the selection and zero on it, the estimate (kept in the workspace) within its
    band, the selection exactly the rule applied to the GPU's own estimate and l2sq, and equal
    to the oracle's wherever H agrees (band coordinates are the only free choices)."""
    from tests.test_gpu_parity import _check_heavymix_against_oracle
    w = workloads.get_config("tiny-2^20")
    P, d, r, c, k, seed, fill_seed = 4, 300_007, 5, 4096, 300, 51, 2**40 + 7
    coeffs = oracle.derive_coefficients(r, seed)
    run = H.new_run(P, d, r, c, k, seed, rho=w.rho)
    ws = torch.empty(gs.gs_heavymix_step_workspace_size(d, k), dtype=torch.uint8, device="cuda")
    l2 = torch.empty(1, dtype=torch.float64, device="cuda")
    gbuf = [torch.empty(d, dtype=torch.float32, device="cuda") for _ in range(P)]
    plan = gs.gs_heavymix_step_plan_create(run.sketch, run.us, run.es, gbuf, d, w.rho, k, fill_seed, run.idx,
                                           run.vals, l2, ws, flags=gs.GS_PLAN_TIME_INSERT | gs.GS_PLAN_TIME_QUERY)
    try:
        hashes = oracle.hash_rows(coeffs, c, np.arange(d, dtype=np.uint64))
        for t in range(3):
            grads = workloads.make_gradients(w, t, range(P), d=d)
            for b, g in zip(gbuf, grads):
                b.copy_(torch.from_numpy(g))
            us0 = [H.host(u) for u in run.us]
            es0 = [H.host(e) for e in run.es]
            if t == 0:
                gs.gs_heavymix_step(run.sketch, run.us, run.es, gbuf, d, w.rho, k, fill_seed, run.idx, run.vals, l2, ws)
            else:
                gs.gs_plan_launch(plan)
            torch.cuda.synchronize()
            idx, vals, l2sq = H.host(run.idx), H.host(run.vals), float(l2.item())
            est = H.host(ws[: 4 * d].view(torch.float32)).copy()      # d < 2^22: every row read
            assert np.array_equal(idx, oracle.heavymix_select(est, l2sq, k, fill_seed))
            pre = [oracle.accumulate(u0, e0, g, w.rho) for u0, e0, g in zip(us0, es0, grads)]
            tabs = [oracle.sketch(e1, coeffs, c, hashes) for _, e1 in pre]
            T = oracle.merge_tree([a for a, _ in tabs])
            A = oracle.merge_tree([b for _, b in tabs])
            _, est_o, l2_o = oracle.heavymix(T, coeffs, d, k, fill_seed, hashes)
            band = oracle.cell_band(A, coeffs, np.arange(d))
            assert np.all(np.abs(est.astype(np.float64) - est_o) <= band)
            assert abs(l2sq - l2_o) <= 1e-4 * l2_o
            _check_heavymix_against_oracle(H, idx, est, l2sq, est_o, l2_o, band, k, fill_seed)
            sel = np.zeros(d, bool)
            sel[idx] = True
            for p, (u1, e1) in enumerate(pre):
                gu, ge = H.host(run.us[p]), H.host(run.es[p])
                assert np.array_equal(gu[~sel].view(np.uint32), u1[~sel].view(np.uint32))
                assert np.array_equal(ge[~sel].view(np.uint32), e1[~sel].view(np.uint32))
                assert np.all(gu[sel] == 0) and np.all(ge[sel] == 0)
            H.check_vals(vals, idx, [e1 for _, e1 in pre])
        q, s = gs.gs_plan_query_times(plan, 10)
        assert len(q) == 2 and all(x > 0 for x in q + s)
    finally:
        gs.gs_plan_destroy(plan)
        run.close()
