"""gs-SGD compression step, restated plainly on the CPU (test infrastructure only).

One step for P data-parallel workers, in the order of Alg. 1 (Global Sketching SGD) and
Alg. 2 (HEAVYMIX) of the paper:

  1. accumulate   u_p <- rho*u_p + g_p ;  e_p <- e_p + u_p            (fp32 semantics)
     Momentum and error feedback are named in Sec. II (1-bit SGD error feedback, DGC
     momentum correction, and their being carried through a linear sketch); Alg. 1 itself
     sketches the stochastic gradient directly.  The reading taken here keeps both
     accumulators per worker and sketches the error accumulator e_p.
  2. sketch       S_p = S(e_p), an r x c Count Sketch (Alg. 1 step 5, Sec. III-A)
  3. tree merge   recursive halving over the P sketches (Alg. 1 steps 8-23; Sec. III-A for
                  P not a power of two: with an odd number of participants the one with the
                  largest id sits the round out)
  4. query        est_i = median_j s_j(i) * S[j][h_j(i)]  (Alg. 2 step 1)
  5. top-k        the k coordinates of largest |est|, ties to the smaller index
                  (Alg. 2 steps 2-3 read as a deterministic top-k, see the design notes)
  6. second round the exact values v_t = sum_p e_p[I_t] of the selected coordinates
                  (Alg. 2 step 4), after which u_p and e_p are zeroed at I_t.
  7. update       w <- w - lr * G~, G~ = v at I and 0 elsewhere (Alg. 1 step 26)

Sketch cells, merge, median and gathered values are computed in fp64; alongside each table
the oracle keeps the table of absolute contributions (sum of |s*x| per cell), which sets
the tolerance bands used by the parity tests.
"""

from __future__ import annotations

import dataclasses

import numpy as np

from .countsketch import hash_rows, splitmix64_at


# ---- 1. accumulate ---------------------------------------------------------------------

def _f32(x: np.ndarray) -> np.ndarray:
    return np.asarray(x, dtype=np.float64).astype(np.float32)


def accumulate(u: np.ndarray, e: np.ndarray, g: np.ndarray, rho: float):
    """Return (u', e') with u' = fl(fl(rho*u) + g) and e' = fl(e + u'), fl = fp32 RN.

    Each single operation is carried out in fp64 and rounded once to fp32; for one
    +, - or * of fp32 operands this is exactly the IEEE fp32 round-to-nearest result.
    No fused multiply-add is involved.  ``rho`` is taken as the fp32 value nearest to it.
    """
    rho32 = np.float64(np.float32(rho))
    u64 = np.asarray(u, dtype=np.float32).astype(np.float64)
    e64 = np.asarray(e, dtype=np.float32).astype(np.float64)
    g64 = np.asarray(g, dtype=np.float32).astype(np.float64)
    prod = _f32(rho32 * u64).astype(np.float64)
    u_new = _f32(prod + g64)
    e_new = _f32(e64 + u_new.astype(np.float64))
    return u_new, e_new


# ---- 2. sketch -------------------------------------------------------------------------

def sketch(x: np.ndarray, coeffs, c: int, hashes=None, idx=None):
    """Count Sketch of vector x (fp32, or an fp64 sum of fp32 vectors): (T, A), both [r, c] fp64.

    T[j][b] = sum over i with h_j(i) = b of s_j(i) * x_i
    A[j][b] = sum over the same i of |x_i|       (the magnitude carried by the cell)
    ``idx`` gives the global coordinate of each entry of x (default 0 .. len(x) - 1), so that
    a long vector can be sketched piece by piece: by the linearity of the Count Sketch
    (Sec. III-A), the sketch of x is the sum of the sketches of its pieces, each piece hashed
    at its own global coordinates.  ``hashes`` may pass ``hash_rows(coeffs, c, idx)`` computed
    once for many vectors.
    """
    x64 = np.asarray(x, dtype=np.float64)     # fp32 vectors widen exactly; fp64 sums stay as they are
    d = x64.size
    if hashes is None:
        gi = np.arange(d, dtype=np.uint64) if idx is None else np.asarray(idx, dtype=np.uint64)
        hashes = hash_rows(coeffs, c, gi)
    buckets, signs = hashes
    r = buckets.shape[0]
    T = np.zeros((r, c), dtype=np.float64)
    A = np.zeros((r, c), dtype=np.float64)
    ax = np.abs(x64)
    for j in range(r):
        T[j] = np.bincount(buckets[j], weights=signs[j] * x64, minlength=c)
        A[j] = np.bincount(buckets[j], weights=ax, minlength=c)
    return T, A


# ---- 3. tree merge ---------------------------------------------------------------------

def merge_schedule(P: int):
    """Rounds of the recursive-halving reduce for P workers.

    Round l (l = 0, 1, ...) involves the workers whose rank is a multiple of 2^l, listed
    in rank order.  The participant at an even position receives from the next one and
    adds; with an odd count the last (largest id) participant sits the round out.  The
    result ends on worker 0 after ceil(log2 P) rounds.  Returns a list of rounds, each a
    list of (receiver, sender) pairs.
    """
    rounds = []
    step = 1
    while step < P:
        ranks = list(range(0, P, step))
        pairs = [(ranks[m], ranks[m + 1]) for m in range(0, len(ranks) - 1, 2)]
        rounds.append(pairs)
        step *= 2
    return rounds


def merge_tree(tables):
    """Sum the P tables along ``merge_schedule(P)``; returns the table left on worker 0.

    ``tables`` is a list of arrays of equal shape; the inputs are not modified.
    Each receive is 'sends = recvs + sends' (Alg. 1), done in fp64.
    """
    work = [np.array(t, dtype=np.float64, copy=True) for t in tables]
    for pairs in merge_schedule(len(work)):
        for recv, send in pairs:
            work[recv] = work[send] + work[recv]
    return work[0]


# ---- 4. query --------------------------------------------------------------------------

def query(T: np.ndarray, coeffs, d: int, hashes=None, idx=None):
    """est_i = median over rows j of s_j(i) * T[j][h_j(i)] for i < d (fp64), or for the global
    coordinates ``idx`` when given (then d = len(idx)).

    With an odd number of rows the median is the middle order statistic; with an even
    number it is the mean of the two middle ones.
    """
    c = T.shape[1]
    if hashes is None:
        gi = np.arange(d, dtype=np.uint64) if idx is None else np.asarray(idx, dtype=np.uint64)
        hashes = hash_rows(coeffs, c, gi)
    buckets, signs = hashes
    r = buckets.shape[0]
    d = buckets.shape[1]
    vals = np.empty((r, d), dtype=np.float64)
    for j in range(r):
        vals[j] = signs[j] * T[j][buckets[j]]
    vals.sort(axis=0)
    if r % 2 == 1:
        return vals[r // 2].copy()
    return 0.5 * (vals[r // 2 - 1] + vals[r // 2])


def cell_band(A: np.ndarray, coeffs, idx, rel: float = 1e-5, hashes=None):
    """Per-coordinate tolerance band rel * max_j A[j][h_j(i)] for the median estimate, at the
    coordinates idx (or at those whose ``hash_rows`` are passed as ``hashes``)."""
    c = A.shape[1]
    buckets, _ = hashes if hashes is not None else hash_rows(coeffs, c, np.asarray(idx, dtype=np.uint64))
    r = buckets.shape[0]
    mags = np.stack([A[j][buckets[j]] for j in range(r)])
    return rel * mags.max(axis=0)


# ---- 5. top-k --------------------------------------------------------------------------

def topk(est: np.ndarray, k: int) -> np.ndarray:
    """The k indices of largest |est|, ties broken toward the smaller index, ascending."""
    est = np.asarray(est, dtype=np.float64)
    order = np.lexsort((np.arange(est.size), -np.abs(est)))
    return np.sort(order[:k]).astype(np.int64)


def topk_by_threshold(est: np.ndarray, k: int) -> np.ndarray:
    """The same set as ``topk``, found without a full sort (for vectors of hundreds of millions
    of entries): tau = the k-th largest |est|; every index with |est| > tau, then the
    k - #{|est| > tau} smallest indices with |est| == tau; ascending."""
    a = np.abs(np.asarray(est, dtype=np.float64))
    tau = np.partition(a, a.size - k)[a.size - k]
    gt = np.nonzero(a > tau)[0]
    eq = np.nonzero(a == tau)[0]
    return np.sort(np.concatenate([gt, eq[: k - gt.size]])).astype(np.int64)


# ---- 5'. HEAVYMIX ----------------------------------------------------------------------

def heavymix_select(est: np.ndarray, l2sq: float, k: int, fill_seed: int) -> np.ndarray:
    """Alg. 2 steps 2-3 from given estimates and ||g||^2 estimate (indices ascending):
    H = {i : est_i^2 >= l2sq / k}, evaluated in fp64 on the estimates as given; if
    |H| >= k the k members of H with largest |est| (ties to the smaller index), else H plus the
    l = k - |H| members of NH with the smallest xi_i = splitmix64_at(fill_seed, i) >> 33,
    ties to the smaller index (a uniformly random l-subset of NH)."""
    est = np.asarray(est, dtype=np.float64)
    in_h = heavymix_members(est, l2sq, k)
    return heavymix_select_from(in_h, est, k, fill_seed)


def heavymix_members(est: np.ndarray, l2sq: float, k: int) -> np.ndarray:
    """The membership mask of H = {i : est_i^2 >= l2sq / k} (Alg. 2 step 2), in fp64."""
    est = np.asarray(est, dtype=np.float64)
    return est * est >= l2sq / k


def heavymix_select_from(in_h: np.ndarray, est: np.ndarray, k: int, fill_seed: int) -> np.ndarray:
    """Alg. 2 step 3 for a given membership mask of H: the top-k of H by |est| when |H| >= k,
    else H plus the first k - |H| members of NH in the fill order (xi_i, i)."""
    est = np.asarray(est, dtype=np.float64)
    in_h = np.asarray(in_h, dtype=bool)
    nh = int(in_h.sum())
    if nh >= k:
        return topk(np.where(in_h, est, 0.0), k)
    NH = np.nonzero(~in_h)[0]
    xi = (splitmix64_at(fill_seed, NH) >> np.uint64(33)).astype(np.int64)
    fill = NH[np.lexsort((NH, xi))[: k - nh]]
    return np.sort(np.concatenate([np.nonzero(in_h)[0], fill])).astype(np.int64)


def heavymix(T: np.ndarray, coeffs, d: int, k: int, fill_seed: int, hashes=None):
    """Alg. 2 steps 1-3 as printed (returns idx ascending, est, l2sq): est is the median query
    (step 1); l2sq, the median over rows j of sum_b T[j][b]^2, estimates ||g||_2^2; the
    selection is ``heavymix_select`` (steps 2-3)."""
    est = query(T, coeffs, d, hashes)
    rows = np.sort(np.sum(np.asarray(T, dtype=np.float64) ** 2, axis=1))
    r = rows.size
    l2sq = rows[r // 2] if r % 2 == 1 else 0.5 * (rows[r // 2 - 1] + rows[r // 2])
    return heavymix_select(est, l2sq, k, fill_seed), est, l2sq


# ---- 6. second round: gather exact values and zero the accumulators ---------------------

def gather_and_zero(us, es, idx):
    """Return (vals, us', es'): vals[t] = sum_p e_p[idx[t]] (fp64), accumulators zeroed.

    The inputs are not modified.
    """
    idx = np.asarray(idx, dtype=np.int64)
    vals = np.zeros(idx.size, dtype=np.float64)
    for e in es:
        vals += np.asarray(e, dtype=np.float32)[idx].astype(np.float64)
    us_out, es_out = [], []
    for u, e in zip(us, es):
        u2 = np.array(u, dtype=np.float32, copy=True)
        e2 = np.array(e, dtype=np.float32, copy=True)
        u2[idx] = 0.0
        e2[idx] = 0.0
        us_out.append(u2)
        es_out.append(e2)
    return vals, us_out, es_out


# ---- 7. weight update ------------------------------------------------------------------

def apply_update(w: np.ndarray, idx, vals, lr: float) -> np.ndarray:
    """Alg. 1 step 26, w <- w - lr * G~ with G~ = vals at idx and 0 elsewhere, in fp32
    semantics: w'[i] = fl(w[i] - fl(lr * v)) with lr taken as the nearest fp32 value.  The
    input is not modified; idx must hold distinct indices."""
    w2 = np.array(w, dtype=np.float32, copy=True)
    idx = np.asarray(idx, dtype=np.int64)
    lr64 = np.float64(np.float32(lr))
    v64 = np.asarray(vals, dtype=np.float32).astype(np.float64)
    step = (lr64 * v64).astype(np.float32).astype(np.float64)
    w2[idx] = (w2[idx].astype(np.float64) - step).astype(np.float32)
    return w2


# ---- 8. momentum and error kept as sketches ----------------------------------------------

def query_at(T: np.ndarray, coeffs, idx) -> np.ndarray:
    """The median estimate of ``query`` at the coordinates ``idx`` only (fp64)."""
    idx = np.asarray(idx, dtype=np.uint64)
    c = T.shape[1]
    buckets, signs = hash_rows(coeffs, c, idx)
    r = buckets.shape[0]
    vals = np.stack([signs[j] * T[j][buckets[j]] for j in range(r)]).astype(np.float64)
    vals.sort(axis=0)
    if r % 2 == 1:
        return vals[r // 2].copy()
    return 0.5 * (vals[r // 2 - 1] + vals[r // 2])


def sketch_sparse(idx, vals, coeffs, c: int):
    """(T, A): the Count Sketch of the sparse vector with vals at idx (fp64), and its
    magnitude table."""
    idx = np.asarray(idx, dtype=np.uint64)
    v = np.asarray(vals, dtype=np.float64)
    buckets, signs = hash_rows(coeffs, c, idx)
    r = buckets.shape[0]
    T = np.zeros((r, c))
    A = np.zeros((r, c))
    for j in range(r):
        T[j] = np.bincount(buckets[j], weights=signs[j] * v, minlength=c)
        A[j] = np.bincount(buckets[j], weights=np.abs(v), minlength=c)
    return T, A


@dataclasses.dataclass
class SketchedStateResult:
    S: np.ndarray       # merged sketch of the step's gradients
    U: np.ndarray       # momentum sketch after the step
    E: np.ndarray       # error sketch after the step
    AU: np.ndarray      # magnitude tables of U and E (tolerance bands)
    AE: np.ndarray
    est: np.ndarray     # estimate from the accumulated error sketch (before removal)
    band: np.ndarray    # per-coordinate band of est
    idx: np.ndarray     # selected coordinates, ascending
    delta: np.ndarray   # values sent for the update: the error sketch's estimate at idx
    delta_u: np.ndarray # the momentum sketch's estimate at idx (removed from U)
    U_pre: np.ndarray   # U and E after accumulation, before the removal
    E_pre: np.ndarray
    AU_pre: np.ndarray
    AE_pre: np.ndarray
    AS: np.ndarray      # magnitude table of S


def sketched_state_step(U, E, AU, AE, gs, rho: float, coeffs, c: int, k: int, rel: float = 1e-5):
    """One step with momentum and error carried as r x c sketches (the linear-sketch variant
    named in Sec. II): S = tree merge of S(g_p); U <- rho U + S; E <- E + U; I = top-k of the
    estimate from E; delta = that estimate at I; then the extracted mass leaves both sketches,
    E <- E - S(delta), U <- U - S(delta_u) with delta_u the estimate of U at I.  fp64; AU, AE
    carry the magnitude tables for the tolerance bands."""
    d = np.asarray(gs[0]).size
    hashes = hash_rows(coeffs, c, np.arange(d, dtype=np.uint64))
    sk = [sketch(g, coeffs, c, hashes) for g in gs]
    S = merge_tree([t for t, _ in sk])
    AS = merge_tree([a for _, a in sk])
    r64 = np.float64(np.float32(rho))
    U1 = r64 * np.asarray(U, np.float64) + S
    AU1 = r64 * np.asarray(AU, np.float64) + AS
    E1 = np.asarray(E, np.float64) + U1
    AE1 = np.asarray(AE, np.float64) + AU1
    est = query(E1, coeffs, d, hashes)
    band = cell_band(AE1, coeffs, np.arange(d), rel)
    idx = topk(est, k)
    delta = est[idx]
    delta_u = query_at(U1, coeffs, idx)
    SD, AD = sketch_sparse(idx, delta, coeffs, c)
    SDu, ADu = sketch_sparse(idx, delta_u, coeffs, c)
    return SketchedStateResult(S, U1 - SDu, E1 - SD, AU1 + ADu, AE1 + AD, est, band, idx, delta, delta_u,
                               U1, E1, AU1, AE1, AS)


# ---- one full step ---------------------------------------------------------------------

@dataclasses.dataclass
class StepResult:
    us: list            # per-worker momentum after the step (fp32)
    es: list            # per-worker error accumulator after the step (fp32)
    us_pre: list        # per-worker momentum after accumulate, before zeroing
    es_pre: list        # per-worker error accumulator after accumulate, before zeroing
    tables: list        # per-worker sketch T_p (fp64 [r, c])
    abs_tables: list    # per-worker magnitude tables A_p (fp64 [r, c])
    merged: np.ndarray  # merged sketch (fp64 [r, c])
    merged_abs: np.ndarray
    est: np.ndarray     # fp64 [d]
    idx: np.ndarray     # int64 [k], ascending
    vals: np.ndarray    # fp64 [k]


def step(us, es, gs, rho: float, coeffs, c: int, k: int) -> StepResult:
    """One gs-SGD compression step over P workers (lists of fp32 vectors of length d)."""
    P = len(gs)
    d = np.asarray(gs[0]).size
    hashes = hash_rows(coeffs, c, np.arange(d, dtype=np.uint64))  # shared by all workers
    us1, es1, tables, abs_tables = [], [], [], []
    for p in range(P):
        u1, e1 = accumulate(us[p], es[p], gs[p], rho)
        T, A = sketch(e1, coeffs, c, hashes)
        us1.append(u1)
        es1.append(e1)
        tables.append(T)
        abs_tables.append(A)
    merged = merge_tree(tables)
    merged_abs = merge_tree(abs_tables)
    est = query(merged, coeffs, d, hashes)
    idx = topk(est, k)
    vals, us2, es2 = gather_and_zero(us1, es1, idx)
    return StepResult(us2, es2, us1, es1, tables, abs_tables, merged, merged_abs, est, idx, vals)
