"""Run the CUDA library through its binding and compare it with the CPU oracle.

Agreement, as the parity tests state it:
  * hash buckets and signs: bit-exact;
  * sketch cells: |T_gpu - T_oracle| <= rel * A_oracle, with A the cell's sum of
    |contributions| and rel = 1e-5;
  * estimates: |est_gpu - est_oracle| <= beta_i = rel * max_j A[j][h_j(i)] (a median moves
    by at most the largest perturbation of its inputs);
  * top-k: index sets equal except for coordinates whose oracle |est| lies within
    beta_i + beta_tau of the oracle's k-th largest |est| tau;
  * momentum and error: bit-identical on every coordinate the GPU did not select (equal to
    the oracle's accumulated values), exactly zero on the ones it did;
  * gathered values: within (P - 1) * 2^-24 * sum_p |e_p[i]| of the exact fp64 sum, the
    error bound of P - 1 sequential fp32 additions.
"""

from __future__ import annotations

import dataclasses

import numpy as np
import torch

import oracle
import paper_2108_06004_gb300 as gs

REL = 1e-5
U32 = 2.0 ** -24


@dataclasses.dataclass
class GpuRun:
    sketch: int
    us: list
    es: list
    d: int
    k: int
    rho: float
    ws: torch.Tensor
    idx: torch.Tensor
    vals: torch.Tensor
    est: torch.Tensor

    def close(self):
        if self.sketch:
            gs.gs_sketch_destroy(self.sketch)
            self.sketch = 0


def new_run(P, d, r, c, k, seed, rho=0.9, group_width=0, dev="cuda:0") -> GpuRun:
    sk = gs.gs_sketch_create(r, c, seed, P, group_width)
    us = [torch.zeros(d, dtype=torch.float32, device=dev) for _ in range(P)]
    es = [torch.zeros(d, dtype=torch.float32, device=dev) for _ in range(P)]
    ws = torch.empty(gs.gs_step_workspace_size(d, k), dtype=torch.uint8, device=dev)
    idx = torch.empty(k, dtype=torch.int64, device=dev)
    vals = torch.empty(k, dtype=torch.float32, device=dev)
    est = torch.empty(d, dtype=torch.float32, device=dev)
    return GpuRun(sk, us, es, d, k, rho, ws, idx, vals, est)


def gpu_step(run: GpuRun, grads_dev) -> None:
    gs.gs_step(run.sketch, run.us, run.es, grads_dev, run.d, run.rho, run.k, run.idx, run.vals,
               run.est, run.ws)


def host(t: torch.Tensor) -> np.ndarray:
    return t.detach().cpu().numpy()


def pruned_rows(e_int: np.ndarray, r: int):
    """(mask, rows): the coordinates whose workspace estimate is a pruning marker,
    -((32 g + n) * 2^-149) with n the rows whose cells were examined and g how many of those
    cells were read from the table, and n for each of them.  Every marker must name
    f <= n < r (f = r/2 + 1) and n - f <= g <= n."""
    bits = e_int.view(np.uint32)
    mask = (bits > np.uint32(0x80000000)) & (bits < np.uint32(0x80000400))
    n = (bits[mask] & np.uint32(31)).astype(np.int64)
    g = ((bits[mask] >> np.uint32(5)) & np.uint32(31)).astype(np.int64)
    f = r // 2 + 1
    assert np.all((n >= f) & (n < r)), "a marker names an impossible row count"
    assert np.all((g <= n) & (g >= n - f)), "a marker names an impossible count of cells read"
    return mask, n


def worker_tables(run: GpuRun, P: int, r: int, c: int):
    out = []
    for p in range(P):
        buf = np.empty(r * c, dtype=np.float32)
        gs.gs_sketch_copy_to_host(run.sketch, p, buf)
        out.append(buf.reshape(r, c))
    return out


def merged_table(run: GpuRun, r: int, c: int) -> np.ndarray:
    buf = np.empty(r * c, dtype=np.float32)
    gs.gs_sketch_copy_to_host(run.sketch, -1, buf)
    return buf.reshape(r, c)


def check_cells(T_gpu, T_orc, A_orc, what: str, rel: float = REL):
    T_gpu = np.asarray(T_gpu, dtype=np.float64)
    err = np.abs(T_gpu - T_orc)
    bad = err > rel * A_orc
    assert not bad.any(), (f"{what}: {int(bad.sum())} cells outside rel*A, worst "
                           f"{float((err - rel * A_orc).max()):.3e}")


def check_topk_set(gpu_idx, orc_idx, est_orc, band, k: int, d: int):
    gpu_idx = np.asarray(gpu_idx)
    assert gpu_idx.size == k
    assert np.all(np.diff(gpu_idx) > 0), "indices not strictly ascending"
    assert gpu_idx[0] >= 0 and gpu_idx[-1] < d
    sym = np.setxor1d(gpu_idx, orc_idx)
    if sym.size == 0:
        return 0
    a = np.abs(est_orc)
    sel = np.asarray(orc_idx)
    kth = sel[np.argmin(a[sel])]
    tau, btau = a[kth], band[kth]
    off = np.abs(a[sym] - tau) > band[sym] + btau
    assert not off.any(), (f"top-k differs outside the tie band at {sym[off][:10]} "
                           f"(|est|={a[sym][off][:5]}, tau={tau})")
    return int(sym.size)


def check_selection_exact(gpu_idx, est_gpu, k: int):
    """The GPU's index set is exactly the top-k of the GPU's own fp32 estimate (keys = bits
    of |est|, ties toward the smaller index)."""
    key = (np.asarray(est_gpu, dtype=np.float32).view(np.uint32) & np.uint32(0x7FFFFFFF))
    order = np.lexsort((np.arange(key.size), -key.astype(np.int64)))
    want = np.sort(order[:k])
    assert np.array_equal(np.asarray(gpu_idx), want), "selection differs from the exact top-k of est"


def check_state(gpu_us, gpu_es, res: oracle.StepResult, gpu_idx):
    sel = np.zeros(res.us[0].size, dtype=bool)
    sel[np.asarray(gpu_idx)] = True
    for p, (gu, ge) in enumerate(zip(gpu_us, gpu_es)):
        gu = np.asarray(gu, dtype=np.float32)
        ge = np.asarray(ge, dtype=np.float32)
        assert np.array_equal(gu[~sel].view(np.uint32), res.us_pre[p][~sel].view(np.uint32)), f"momentum[{p}] differs"
        assert np.array_equal(ge[~sel].view(np.uint32), res.es_pre[p][~sel].view(np.uint32)), f"error[{p}] differs"
        assert np.all(gu[sel] == 0) and np.all(ge[sel] == 0), f"selected coordinates of worker {p} not zeroed"


def check_vals(gpu_vals, gpu_idx, es_pre):
    P = len(es_pre)
    stack = np.stack([np.asarray(e, dtype=np.float32)[np.asarray(gpu_idx)].astype(np.float64) for e in es_pre])
    exact = stack.sum(axis=0)
    bound = (P - 1) * U32 * np.abs(stack).sum(axis=0) * (1 + 1e-6)
    err = np.abs(np.asarray(gpu_vals, dtype=np.float64) - exact)
    assert np.all(err <= bound), f"gathered values off by {float((err - bound).max()):.3e} beyond the fp32 bound"


def compare_step(res: oracle.StepResult, coeffs, gpu_us, gpu_es, gpu_idx, gpu_vals, gpu_est, k,
                 gpu_tables=None, gpu_merged=None, rel: float = REL):
    """All agreement checks for one step; returns the size of the tie-band difference."""
    d = res.us[0].size
    if gpu_tables is not None:
        for p, T in enumerate(gpu_tables):
            check_cells(T, res.tables[p], res.abs_tables[p], f"worker {p} table", rel)
    if gpu_merged is not None:
        check_cells(gpu_merged, res.merged, res.merged_abs, "merged table", rel)
    band = oracle.cell_band(res.merged_abs, coeffs, np.arange(d), rel)
    err = np.abs(np.asarray(gpu_est, dtype=np.float64) - res.est)
    assert np.all(err <= band), f"estimate outside band at {np.nonzero(err > band)[0][:10]}"
    check_selection_exact(gpu_idx, gpu_est, k)
    nsym = check_topk_set(gpu_idx, res.idx, res.est, band, k, d)
    check_state(gpu_us, gpu_es, res, gpu_idx)
    check_vals(gpu_vals, gpu_idx, res.es_pre)
    return nsym


def fp32_tree(tables):
    """The merge schedule applied with fp32 additions, for a bit-exact check of the kernel."""
    work = [np.array(t, dtype=np.float32, copy=True) for t in tables]
    for pairs in oracle.merge_schedule(len(work)):
        for recv, send in pairs:
            work[recv] = (work[send] + work[recv]).astype(np.float32)
    return work[0]
