"""GPU parity at the full size of every workload, over several steps, against the oracle.

Each workload runs in the launch configuration the benchmark times: a captured plan per step
with the estimate kept in the workspace (so the query skips rows), and for BERT-large the 32
workers streamed 8 at a time with fresh gradients per batch.  Before every step the GPU's
momentum and error are copied on the device; after it, the oracle (evaluated in pieces by a
process pool, ``tests/full_size.py``) recomputes the step from that state and the step's
gradients, and the agreement is checked everywhere:

  * momentum and error of every worker: bit-identical on every coordinate the GPU did not
    select, exactly zero on those it did (full vectors);
  * every cell of the merged table within 1e-5 of its magnitude, and of every worker table at
    P <= 8 (the first and the last worker's at P = 16 and 32, where the oracle's merged table is
    computed as the sketch of the summed error vectors, equal to the tree by linearity);
  * the full estimate of every coordinate (a second query of the same merged table that
    returns it) within its band of the oracle's estimate; every coordinate the step's query
    skipped has an oracle estimate below the GPU's k-th largest |est| plus its band;
  * the step's selection equals that full query's, is exactly the top-k of its estimate, and
    equals the oracle's top-k except within the tie band;
  * the gathered values within the fp32 bound of the exact sums.

Steps: 5 at the ResNet-18 and ResNet-50 sizes, 2 at the VGG-16 and BERT-large sizes.
"""

from __future__ import annotations

import numpy as np
import pytest

torch = pytest.importorskip("torch")

import oracle  # noqa: E402
import workloads  # noqa: E402

pytestmark = pytest.mark.gpu

SEED = 2108


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


def _fill(gs, w, t, workers, bufs):
    for q, b in zip(workers, bufs):
        workloads.make_gradient_torch(w, t, q, b)


class _Clock:
    """Wall time per phase of a step, printed at the end (shown with pytest -s)."""

    def __init__(self):
        import time
        self.time = time.perf_counter
        self.t = self.time()
        self.parts = {}

    def lap(self, name):
        now = self.time()
        self.parts[name] = self.parts.get(name, 0.0) + now - self.t
        self.t = now


def run_full_size(gs, H, name, steps):
    from tests import full_size
    clock = _Clock()
    w = workloads.get_config(name)
    P, d, r, c, k, rho = w.P, w.d, w.r, w.c, w.k, w.rho
    streamed = bool(w.worker_batch) and w.worker_batch < P
    batch = w.worker_batch if streamed else P
    coeffs = oracle.derive_coefficients(r, SEED)
    dev = torch.device("cuda")
    slots = min(full_size.host_cores(), 8, P)
    with full_size.ParallelOracle(coeffs, c, d, slots) as po:
        clock.lap("oracle hashes")
        sk = gs.gs_sketch_create(r, c, SEED, P, 0)
        plan = None
        try:
            us = [torch.zeros(d, dtype=torch.float32, device=dev) for _ in range(P)]
            es = [torch.zeros(d, dtype=torch.float32, device=dev) for _ in range(P)]
            u0 = [torch.empty_like(u) for u in us]
            e0 = [torch.empty_like(e) for e in es]
            gbuf = [torch.empty(d, dtype=torch.float32, device=dev) for _ in range(batch)]
            ws = torch.empty(gs.gs_step_workspace_size(d, k), dtype=torch.uint8, device=dev)
            ws2 = torch.empty(gs.gs_query_topk_workspace_size(d, k), dtype=torch.uint8, device=dev)
            idx = torch.empty(k, dtype=torch.int64, device=dev)
            vals = torch.empty(k, dtype=torch.float32, device=dev)
            idx_full = torch.empty(k, dtype=torch.int64, device=dev)
            est_full = torch.empty(d, dtype=torch.float32, device=dev)
            if not streamed:
                plan = gs.gs_step_plan_create(sk, us, es, gbuf, d, rho, k, idx, vals, None, None, 0.0, ws)
            for t in range(steps):
                for a, b in zip(u0 + e0, us + es):
                    a.copy_(b)
                # the step, as the benchmark launches it
                if streamed:
                    gs.gs_sketch_zero(sk)
                    for b0 in range(0, P, batch):
                        _fill(gs, w, t, range(b0, b0 + batch), gbuf)
                        gs.gs_accumulate_insert(sk, b0, us[b0:b0 + batch], es[b0:b0 + batch], gbuf, d, rho)
                    gs.gs_sketch_merge_tree(sk, P)
                    gs.gs_query_topk(sk, d, k, idx, None, ws)
                    gs.gs_gather_and_zero(us, es, d, idx, k, vals)
                else:
                    _fill(gs, w, t, range(P), gbuf)
                    gs.gs_plan_launch(plan)
                # the full estimate of the same merged table
                gs.gs_query_topk(sk, d, k, idx_full, est_full, ws2)
                torch.cuda.synchronize()
                gi = H.host(idx).copy()
                assert np.array_equal(gi, H.host(idx_full)), f"step {t}: pruned and full selections differ"
                e_int = H.host(ws[: 4 * d].view(torch.float32)).copy()
                est_g = H.host(est_full).copy()
                check_selection_linear(gi, est_g, k)
                clock.lap("GPU step and selection checks")

                # the oracle, worker by worker from the GPU's pre-step state, slots-many at a time
                tabled = set(range(P)) if P <= 8 else {0, P - 1}
                T_sum = A_sum = 0.0
                own_tables, e_rows = {}, [None] * P
                for p0 in range(0, P, slots):
                    group = list(range(p0, min(P, p0 + slots)))
                    for s, p in enumerate(group):
                        if streamed:
                            _fill(gs, w, t, [p], gbuf[:1])
                            g = gbuf[0]
                        else:
                            g = gbuf[p]
                        for nm, src in (("u0", u0[p]), ("e0", e0[p]), ("g", g), ("ug", us[p]), ("eg", es[p])):
                            torch.from_numpy(po.slot(s, nm)).copy_(src)   # device -> the mapped slot
                    clock.lap("copies to the oracle")
                    Ts, As, own, e_sel, counts = po.workers(range(len(group)), rho, gi,
                                                           tabled=[s for s, p in enumerate(group) if p in tabled])
                    clock.lap("oracle workers")
                    T_sum = T_sum + Ts
                    A_sum = A_sum + As
                    for s, p in enumerate(group):
                        bu, be, nz = counts[s]
                        assert bu == 0 and be == 0, f"step {t}, worker {p}: {bu} momentum, {be} error values differ"
                        assert nz == 0, f"step {t}, worker {p}: selected coordinates not zeroed"
                        e_rows[p] = e_sel[s]
                        if s in own:
                            own_tables[p] = own[s]
                for p, (Tp, Ap) in own_tables.items():
                    tab = np.empty(r * c, np.float32)
                    gs.gs_sketch_copy_to_host(sk, p, tab)
                    H.check_cells(tab.reshape(r, c), Tp, Ap, f"step {t}, worker {p} table")
                if len(own_tables) == P:   # every worker's table: the oracle's tree
                    T = oracle.merge_tree([own_tables[p][0] for p in range(P)])
                    A = oracle.merge_tree([own_tables[p][1] for p in range(P)])
                else:                      # else its equal by linearity, the sketch of the sum
                    T, A = T_sum, A_sum
                merged = np.empty(r * c, np.float32)
                gs.gs_sketch_copy_to_host(sk, -1, merged)
                H.check_cells(merged.reshape(r, c), T, A, f"step {t}, merged table")
                e_sel = np.stack(e_rows).astype(np.float64)
                del own_tables
                clock.lap("tables: merge and cell checks")

                est_o, band = po.query(T, A)
                clock.lap("oracle query")
                err = np.abs(est_g.astype(np.float64) - est_o)
                assert np.all(err <= band), f"step {t}: estimate outside its band at {np.nonzero(err > band)[0][:10]}"
                pruned, _ = H.pruned_rows(e_int, r)
                tau_g = np.abs(est_g[gi]).min()
                assert np.all(np.abs(est_o[pruned]) <= tau_g + band[pruned]), f"step {t}: a skipped row mattered"
                idx_o = oracle.topk_by_threshold(est_o, k)
                H.check_topk_set(gi, idx_o, est_o, band, k, d)

                # gathered values: the exact sums of the oracle's accumulated error at the selection
                exact = e_sel.sum(axis=0)
                bound = (P - 1) * 2.0**-24 * np.abs(e_sel).sum(axis=0) * (1 + 1e-6)
                assert np.all(np.abs(H.host(vals).astype(np.float64) - exact) <= bound), f"step {t}: gathered values"
                del est_o, band, err
                clock.lap("estimate, top-k and value checks")
        finally:
            if plan:
                gs.gs_plan_destroy(plan)
            gs.gs_sketch_destroy(sk)
            print(f"{name}: " + ", ".join(f"{k} {v:.1f} s" for k, v in clock.parts.items()))


@pytest.mark.parametrize("name,steps", [("resnet18", 5), ("resnet50", 5), ("vgg16", 2), ("bert-large", 2)])
def test_full_size_steps(gs, H, name, steps):
    try:
        run_full_size(gs, H, name, steps)
    finally:
        torch.cuda.empty_cache()   # return the workload's device memory to the driver for later tests
