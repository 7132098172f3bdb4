"""The piecewise, multi-process evaluation of the oracle used by the full-size GPU tests
(tests/full_size.py) gives exactly what the plain ``oracle.step`` gives on a small case: the
same worker tables (up to fp64 summation order over the pieces), bit-identical accumulated
state at the selected coordinates and everywhere else, the same estimate, band and top-k."""

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
        out = po.workers(range(P), rho, res.idx)
        for p, (T, A, e_sel, bad_u, bad_e, nonzero) in enumerate(out):
            assert bad_u == 0 and bad_e == 0 and nonzero == 0
            assert np.allclose(T, res.tables[p], rtol=0, atol=1e-12 * res.abs_tables[p].max())
            assert np.allclose(A, res.abs_tables[p], rtol=1e-14, atol=0)
            assert np.array_equal(e_sel, res.es_pre[p][res.idx])
        M = oracle.merge_tree([o[0] for o in out])
        MA = oracle.merge_tree([o[1] for o in out])
        est, band = po.query(M, MA)
        assert np.allclose(est, res.est, rtol=0, atol=1e-12)
        assert np.allclose(band, oracle.cell_band(res.merged_abs, co, np.arange(d)), rtol=1e-13, atol=0)
        assert np.array_equal(oracle.topk_by_threshold(est, k), res.idx)
        # one slot alone is split over both processes: the same result
        T0, A0, e0, bu0, be0, nz0 = po.workers([0], rho, res.idx)[0]
        assert np.allclose(T0, out[0][0], rtol=0, atol=1e-12 * res.abs_tables[0].max())
        assert np.array_equal(e0, out[0][2]) and bu0 == be0 == nz0 == 0
        # a planted mistake in the GPU-side state is counted
        po.slot(0, "eg")[5] = np.float32(1.0)
        assert po.workers([0], rho, res.idx)[0][4] == 1
