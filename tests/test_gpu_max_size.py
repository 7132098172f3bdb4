"""The largest dimension the library accepts: d = 2^31 - 1 coordinates (ragged: d mod 4 = 3).

One worker's gradient is zero except at seven spikes, among them the first and the last
coordinates and coordinates past 2^30.  The expected step is then exact and needs no pass
of the oracle over 2^31 coordinates:
  * the sketch holds only the spikes: the merged table equals the oracle's sparse sketch of
    them (oracle.sketch_sparse);
  * every other estimate is 0 unless a coordinate shares a cell with a spike in three of the
    five rows, which for c = 2^20 has probability below 2^-30 over all coordinates; so the
    top-k is the spikes plus the k - 7 smallest other indices (ties of the zero key go to the
    smaller index), and every coordinate is a selection candidate, which drives the
    candidate buffers far past their block-local capacity;
  * the gathered values are the spikes (u = e = g after one step from zero), zeros elsewhere;
  * after the step momentum and error are zero everywhere.
About 52 GB stay on the device (three d-vectors and the query workspace).
"""

from __future__ import annotations

import numpy as np
import pytest
import torch

import oracle

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def gs():
    import paper_2108_06004_gb300 as lib
    lib.load_library()
    return lib


def test_step_at_max_dimension(gs):
    d = gs.GS_MAX_DIM
    assert d == 2**31 - 1
    torch.cuda.empty_cache()   # blocks cached by earlier tests count as used
    free, _ = torch.cuda.mem_get_info()
    if free < (64 << 30):
        pytest.skip("needs 64 GB of free device memory")
    P, r, c, k, seed = 1, 5, 1 << 20, 1000, 31
    spikes = np.array([0, 1, 12_345, 2**30, 2**31 - 4, 2**31 - 3, d - 1], dtype=np.int64)
    vals = np.array([3.0, -2.5, 7.25, -9.0, 4.5, 1.75, -6.0], dtype=np.float32)
    dev = "cuda"
    sk = gs.gs_sketch_create(r, c, seed, P, 0)
    try:
        g = torch.zeros(d, dtype=torch.float32, device=dev)
        g[torch.from_numpy(spikes).to(dev)] = torch.from_numpy(vals).to(dev)
        u = torch.zeros(d, dtype=torch.float32, device=dev)
        e = torch.zeros(d, dtype=torch.float32, device=dev)
        ws = torch.empty(gs.gs_step_workspace_size(d, k), dtype=torch.uint8, device=dev)
        idx = torch.empty(k, dtype=torch.int64, device=dev)
        out = torch.empty(k, dtype=torch.float32, device=dev)
        gs.gs_step(sk, [u], [e], [g], d, 0.9, k, idx, out, None, ws)
        torch.cuda.synchronize()

        table = np.empty(r * c, dtype=np.float32)
        gs.gs_sketch_copy_to_host(sk, -1, table)
        coeffs = oracle.derive_coefficients(r, seed)
        T, _ = oracle.sketch_sparse(spikes, vals.astype(np.float64), coeffs, c)
        assert np.array_equal(table.reshape(r, c).astype(np.float64), T)  # a few exact fp32 sums

        rest = np.setdiff1d(np.arange(k, dtype=np.int64), spikes)[: k - spikes.size]
        want = np.sort(np.concatenate([spikes, rest]))
        got = idx.cpu().numpy()
        assert np.array_equal(got, want)
        want_vals = np.zeros(k, dtype=np.float32)
        want_vals[np.searchsorted(want, spikes)] = vals
        assert np.array_equal(out.cpu().numpy(), want_vals)
        assert int(torch.count_nonzero(u)) == 0 and int(torch.count_nonzero(e)) == 0
    finally:
        gs.gs_sketch_destroy(sk)
