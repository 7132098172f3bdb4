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
  * for each group of workers held in the slots, tasks over parts of the pieces (so that every
    process is busy): per worker ``accumulate`` piece by piece from the GPU's pre-step state and
    the step's gradient, the bit-exact comparison with the GPU's post-step momentum and error
    (zero at the selected coordinates), the accumulated error at the selected coordinates, and,
    for the workers asked for, their own fp64 sketch and magnitude table;
  * the merged table: ``merge_tree`` of the worker tables where every worker has one, else, by
    the same linearity (pinned: the merge of sketches is the sketch of the sum, and likewise for
    the magnitude tables), the sketch of the fp64 sum of the workers' accumulated error vectors
    and the magnitude table of the sum of their absolute values;
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


def _group_task(args):
    """A group of workers' step over the pieces [p0, p1) of the coordinate range, from their
    slots of mapped vectors (u0, e0, g: the GPU's state before the step and the step's gradient;
    ug, eg: the GPU's state after it).  Per worker: the accumulated error at the selected
    coordinates inside those pieces (zero elsewhere) and the counts of momentum / error values
    that differ from the GPU's and of selected values not zeroed; for the workers in `tabled`,
    their own fp64 sketch and magnitude table.  For the group: the sketch of the sum of its
    accumulated error vectors and the magnitude table of the sum of their absolute values (by
    linearity, their merge)."""
    dirpath, slots, tabled, coeffs, c, d, rho, sel, p0, p1 = args
    bk = _mapped(os.path.join(dirpath, "buckets.npy"), None, None, "r")
    sg = _mapped(os.path.join(dirpath, "signs.npy"), None, None, "r")
    r = bk.shape[0]
    vecs = {s: {n: _mapped(os.path.join(dirpath, f"slot{s}_{n}.npy"), None, None, "r")
                for n in ("u0", "e0", "g", "ug", "eg")} for s in slots}
    own = {s: (np.zeros((r, c)), np.zeros((r, c))) for s in tabled}
    T_sum, A_sum = np.zeros((r, c)), np.zeros((r, c))
    e_sel = {s: np.zeros(sel.size, np.float32) for s in slots}
    counts = {s: [0, 0, 0] for s in slots}
    for a, b in _pieces(d)[p0:p1]:
        hashes = (np.asarray(bk[:, a:b]), np.asarray(sg[:, a:b]))
        lo, hi = np.searchsorted(sel, [a, b])
        loc = sel[lo:hi] - a
        keep = np.ones(b - a, bool)
        keep[loc] = False
        x_sum = np.zeros(b - a)
        a_sum = np.zeros(b - a)
        for s in slots:
            v = vecs[s]
            u1, e1 = oracle.accumulate(v["u0"][a:b], v["e0"][a:b], v["g"][a:b], rho)
            e_sel[s][lo:hi] = e1[loc]
            ug, eg = np.asarray(v["ug"][a:b]), np.asarray(v["eg"][a:b])
            counts[s][0] += int(np.count_nonzero(ug[keep].view(np.uint32) != u1[keep].view(np.uint32)))
            counts[s][1] += int(np.count_nonzero(eg[keep].view(np.uint32) != e1[keep].view(np.uint32)))
            counts[s][2] += int(np.count_nonzero(ug[loc]) + np.count_nonzero(eg[loc]))
            x_sum += e1
            a_sum += np.abs(e1.astype(np.float64))
            if s in own:
                t, m = oracle.sketch(e1, coeffs, c, hashes=hashes)
                own[s][0][:] += t
                own[s][1][:] += m
        T_sum += oracle.sketch(x_sum, coeffs, c, hashes=hashes)[0]
        A_sum += oracle.sketch(a_sum, coeffs, c, hashes=hashes)[1]
    return T_sum, A_sum, own, e_sel, counts


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

    def workers(self, slot_ids, rho: float, sel, tabled=()):
        """The step of the workers in the filled slots, their pieces split over every process.
        Returns (T_sum, A_sum, own, e_sel, counts): the sketch of the sum of their accumulated
        error vectors and the magnitude table of the sum of their absolute values; own[slot] =
        (T, A) for the slots in `tabled`; e_sel[slot], the accumulated error at the selected
        coordinates; counts[slot] = (momentum values differing from the GPU's, error values
        differing, selected values not zeroed)."""
        sel = np.ascontiguousarray(np.sort(np.asarray(sel, np.int64)))
        slot_ids = list(slot_ids)
        tabled = [s for s in slot_ids if s in set(tabled)]
        npieces = len(_pieces(self.d))
        split = max(1, min(npieces, self.procs))
        bounds = [(npieces * q // split, npieces * (q + 1) // split) for q in range(split)]
        parts = self.pool.map(_group_task, [(self.dir, slot_ids, tabled, self.coeffs, self.c, self.d, rho, sel, p0, p1)
                                            for p0, p1 in bounds], chunksize=1)
        T_sum = sum(m[0] for m in parts)
        A_sum = sum(m[1] for m in parts)
        own = {s: (sum(m[2][s][0] for m in parts), sum(m[2][s][1] for m in parts)) for s in tabled}
        e_sel = {s: sum(m[3][s] for m in parts) for s in slot_ids}
        counts = {s: [sum(m[4][s][q] for m in parts) for q in range(3)] for s in slot_ids}
        return T_sum, A_sum, own, e_sel, counts

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
