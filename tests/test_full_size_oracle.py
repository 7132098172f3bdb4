"""The piecewise, multi-process evaluation of the oracle used by the full-size GPU tests
(tests/full_size.py) gives exactly what the plain ``oracle.step`` gives on a small case: the
same worker tables and merged table (up to fp64 summation order), the merged table also as the
sketch of the workers' summed error vectors, bit-identical accumulated state at the selected
coordinates and everywhere else, the same estimate, band and top-k."""

import numpy as np

import oracle
from tests import full_size


def test_parallel_oracle_equals_plain_step(monkeypatch):
    monkeypatch.setattr(full_size, "PIECE", 1 << 15)
    rng = np.random.default_rng(3)
    d, r, c, k, P, rho = 200_003, 5, 2048, 300, 3, 0.9
    co = oracle.derive_coefficients(r, 9)
    us = [(rng.standard_normal(d) * 1e-2).astype(np.float32) for _ in range(P)]
    es = [(rng.standard_normal(d) * 1e-2).astype(np.float32) for _ in range(P)]
    gs = [(rng.standard_normal(d) * 1e-2).astype(np.float32) for _ in range(P)]
    res = oracle.step(us, es, gs, rho, co, c, k)
    with full_size.ParallelOracle(co, c, d, slots=P, procs=2) as po:
        for p in range(P):
            for name, v in (("u0", us[p]), ("e0", es[p]), ("g", gs[p]), ("ug", res.us[p]), ("eg", res.es[p])):
                po.slot(p, name)[:] = v
        T_sum, A_sum, own, e_sel, counts = po.workers(range(P), rho, res.idx, tabled=range(P))
        for p in range(P):
            assert counts[p] == [0, 0, 0]
            assert np.allclose(own[p][0], res.tables[p], rtol=0, atol=1e-12 * res.abs_tables[p].max())
            assert np.allclose(own[p][1], res.abs_tables[p], rtol=1e-14, atol=0)
            assert np.array_equal(e_sel[p], res.es_pre[p][res.idx])
        # the merged table by linearity: the sketch of the sum of the workers' error vectors
        assert np.allclose(T_sum, res.merged, rtol=0, atol=1e-12 * res.merged_abs.max())
        assert np.allclose(A_sum, res.merged_abs, rtol=1e-13, atol=0)
        M = oracle.merge_tree([own[p][0] for p in range(P)])
        MA = oracle.merge_tree([own[p][1] for p in range(P)])
        est, band = po.query(M, MA)
        assert np.allclose(est, res.est, rtol=0, atol=1e-12)
        assert np.allclose(band, oracle.cell_band(res.merged_abs, co, np.arange(d)), rtol=1e-13, atol=0)
        assert np.array_equal(oracle.topk_by_threshold(est, k), res.idx)
        # one slot alone, its pieces split over both processes: the same result
        T0, _, own0, e0, c0 = po.workers([0], rho, res.idx, tabled=[0])
        assert np.allclose(own0[0][0], own[0][0], rtol=0, atol=1e-12 * res.abs_tables[0].max())
        assert np.allclose(T0, own[0][0], rtol=0, atol=1e-12 * res.abs_tables[0].max())
        assert np.array_equal(e0[0], e_sel[0]) and c0[0] == [0, 0, 0]
        # a planted mistake in the GPU-side state is counted
        po.slot(0, "eg")[5] = np.float32(1.0)
        assert po.workers([0], rho, res.idx)[4][0] == [0, 1, 0]
