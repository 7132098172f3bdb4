"""The oracle at the full sizes of the workloads: the same oracle functions, evaluated on pieces
of the coordinate range by a pool of processes (test infrastructure only).

At d = 138M or 333M with 16 or 32 workers, ``oracle.step`` would hold every worker's vectors,
every hash value and the fp64 intermediates at once.  The Count Sketch is linear (Sec. III-A):
the sketch of a vector is the sum of the sketches of its pieces, each piece hashed at its own
global coordinates (``oracle.sketch(..., idx=...)``, pinned against the whole-vector sketch).
Accumulation and the median query are elementwise.  So every quantity of a step is computed
here exactly as ``oracle.step`` computes it, piece by piece:

  * the hash buckets and signs of all d coordinates, once per test, into files that every
    process maps (``hash_rows`` per piece);
  * per worker, tasks over parts of its pieces (so that every process is busy): ``accumulate``
    piece by piece from the GPU's pre-step state and the step's gradient, the bit-exact
    comparison with the GPU's post-step momentum and error (zero at the selected coordinates),
    and the worker's fp64 sketch and magnitude table summed over the pieces; also the
    accumulated error at the selected coordinates;
  * ``merge_tree`` of the worker tables (in the calling process);
  * the median query and its tolerance band, piece by piece into mapped files.

The pool is started with the "spawn" method, so that no child inherits a CUDA context.
"""

from __future__ import annotations

import multiprocessing as mp
import os
import shutil
import tempfile

import numpy as np

import oracle

PIECE = 1 << 22   # coordinates per piece


def _mapped(path, dtype, shape, mode):
    return np.lib.format.open_memmap(path, mode=mode, dtype=dtype, shape=shape)


def _pieces(d):
    return [(a, min(a + PIECE, d)) for a in range(0, d, PIECE)]


# ---- tasks (run in the pool's processes) --------------------------------------------------

def _hash_task(args):
    dirpath, coeffs, c, a, b = args
    bk = _mapped(os.path.join(dirpath, "buckets.npy"), None, None, "r+")
    sg = _mapped(os.path.join(dirpath, "signs.npy"), None, None, "r+")
    buckets, signs = oracle.hash_rows(coeffs, c, np.arange(a, b, dtype=np.uint64))
    bk[:, a:b] = buckets.astype(np.int32)
    sg[:, a:b] = signs
    bk.flush()
    sg.flush()
    return b - a


def _worker_task(args):
    """One worker's step, over the pieces [p0, p1) of its coordinate range, from its slot of
    mapped vectors (u0, e0, g: the GPU's state before the step and the step's gradient; ug, eg:
    the GPU's state after it).  Returns the fp64 sketch and magnitude table of those pieces, the
    accumulated error at the selected coordinates inside them (zero elsewhere), and the counts of
    momentum / error values that differ from the GPU's and of selected values not zeroed."""
    dirpath, slot, coeffs, c, d, rho, sel, p0, p1 = args
    bk = _mapped(os.path.join(dirpath, "buckets.npy"), None, None, "r")
    sg = _mapped(os.path.join(dirpath, "signs.npy"), None, None, "r")
    vec = {n: _mapped(os.path.join(dirpath, f"slot{slot}_{n}.npy"), None, None, "r")
           for n in ("u0", "e0", "g", "ug", "eg")}
    r = bk.shape[0]
    T = np.zeros((r, c))
    A = np.zeros((r, c))
    e_sel = np.zeros(sel.size, np.float32)
    bad_u = bad_e = nonzero_sel = 0
    for a, b in _pieces(d)[p0:p1]:
        u1, e1 = oracle.accumulate(vec["u0"][a:b], vec["e0"][a:b], vec["g"][a:b], rho)
        lo, hi = np.searchsorted(sel, [a, b])
        loc = sel[lo:hi] - a
        e_sel[lo:hi] = e1[loc]
        keep = np.ones(b - a, bool)
        keep[loc] = False
        ug, eg = np.asarray(vec["ug"][a:b]), np.asarray(vec["eg"][a:b])
        bad_u += int(np.count_nonzero(ug[keep].view(np.uint32) != u1[keep].view(np.uint32)))
        bad_e += int(np.count_nonzero(eg[keep].view(np.uint32) != e1[keep].view(np.uint32)))
        nonzero_sel += int(np.count_nonzero(ug[loc]) + np.count_nonzero(eg[loc]))
        t, m = oracle.sketch(e1, coeffs, c, hashes=(np.asarray(bk[:, a:b]), np.asarray(sg[:, a:b])))
        T += t
        A += m
    return T, A, e_sel, bad_u, bad_e, nonzero_sel


def _query_task(args):
    dirpath, coeffs, a, b, rel = args
    bk = _mapped(os.path.join(dirpath, "buckets.npy"), None, None, "r")
    sg = _mapped(os.path.join(dirpath, "signs.npy"), None, None, "r")
    T = np.load(os.path.join(dirpath, "merged.npy"))
    Aab = np.load(os.path.join(dirpath, "merged_abs.npy"))
    est = _mapped(os.path.join(dirpath, "est.npy"), None, None, "r+")
    band = _mapped(os.path.join(dirpath, "band.npy"), None, None, "r+")
    hb, hs = np.asarray(bk[:, a:b]).astype(np.int64), np.asarray(sg[:, a:b])
    est[a:b] = oracle.query(T, coeffs, b - a, hashes=(hb, hs))
    band[a:b] = oracle.cell_band(Aab, coeffs, None, rel, hashes=(hb, hs))
    est.flush()
    band.flush()
    return b - a


# ---- the driver ------------------------------------------------------------------------------

def storage_dir(need_bytes: int) -> str:
    """A directory with room for the mapped files: /dev/shm when it has the space, else the
    temporary directory."""
    for base in ("/dev/shm", tempfile.gettempdir()):
        try:
            if shutil.disk_usage(base).free > need_bytes * 1.2:
                return tempfile.mkdtemp(prefix="gs_full_", dir=base)
        except OSError:
            continue
    return tempfile.mkdtemp(prefix="gs_full_")


def host_cores() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except (AttributeError, OSError):
        return os.cpu_count() or 1


class ParallelOracle:
    """The oracle of one workload at full size, in pieces (see the module docstring)."""

    def __init__(self, coeffs, c: int, d: int, slots: int, procs: int | None = None):
        self.coeffs, self.c, self.d = coeffs, c, d
        self.r = len(coeffs[0])
        self.slots = slots
        need = d * (5 * self.r + 5 * 4 * slots + 16)
        self.dir = storage_dir(need)
        self.procs = procs or max(1, min(host_cores(), 16))
        self.pool = mp.get_context("spawn").Pool(self.procs)
        _mapped(os.path.join(self.dir, "buckets.npy"), np.int32, (self.r, d), "w+").flush()
        _mapped(os.path.join(self.dir, "signs.npy"), np.int8, (self.r, d), "w+").flush()
        self.pool.map(_hash_task, [(self.dir, coeffs, c, a, b) for a, b in _pieces(d)])
        for s in range(slots):
            for n in ("u0", "e0", "g", "ug", "eg"):
                _mapped(self.slot_path(s, n), np.float32, (d,), "w+").flush()

    def slot_path(self, slot: int, name: str) -> str:
        return os.path.join(self.dir, f"slot{slot}_{name}.npy")

    def slot(self, slot: int, name: str) -> np.ndarray:
        return _mapped(self.slot_path(slot, name), None, None, "r+")

    def workers(self, slot_ids, rho: float, sel):
        """Run the worker tasks of the filled slots, each slot's pieces split over enough tasks
        to keep every process busy; returns one combined result per slot, in slot order."""
        sel = np.ascontiguousarray(np.sort(np.asarray(sel, np.int64)))
        slot_ids = list(slot_ids)
        npieces = len(_pieces(self.d))
        split = max(1, min(npieces, -(-self.procs // max(1, len(slot_ids)))))
        bounds = [(npieces * q // split, npieces * (q + 1) // split) for q in range(split)]
        tasks = [(self.dir, s, self.coeffs, self.c, self.d, rho, sel, p0, p1) for s in slot_ids for p0, p1 in bounds]
        parts = self.pool.map(_worker_task, tasks, chunksize=1)
        out = []
        for n in range(len(slot_ids)):
            mine = parts[n * split:(n + 1) * split]
            T = sum(m[0] for m in mine)
            A = sum(m[1] for m in mine)
            e_sel = sum(m[2] for m in mine)
            out.append((T, A, e_sel, sum(m[3] for m in mine), sum(m[4] for m in mine), sum(m[5] for m in mine)))
        return out

    def query(self, merged, merged_abs, rel: float = 1e-5):
        """(est, band): the fp64 median estimate of every coordinate and its tolerance band."""
        np.save(os.path.join(self.dir, "merged.npy"), np.asarray(merged, np.float64))
        np.save(os.path.join(self.dir, "merged_abs.npy"), np.asarray(merged_abs, np.float64))
        est = _mapped(os.path.join(self.dir, "est.npy"), np.float64, (self.d,), "w+")
        band = _mapped(os.path.join(self.dir, "band.npy"), np.float64, (self.d,), "w+")
        est.flush()
        band.flush()
        self.pool.map(_query_task, [(self.dir, self.coeffs, a, b, rel) for a, b in _pieces(self.d)])
        est = _mapped(os.path.join(self.dir, "est.npy"), None, None, "r")
        band = _mapped(os.path.join(self.dir, "band.npy"), None, None, "r")
        return np.array(est), np.array(band)

    def close(self):
        if self.pool is not None:
            self.pool.close()
            self.pool.join()
            self.pool = None
        shutil.rmtree(self.dir, ignore_errors=True)

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()
