"""Pins of the CPU oracle against facts fixed outside the oracle itself.

Each test checks the oracle against a published value, a closed form, an invariant of the
Count Sketch (Sec. III-A: S(a) = C a is linear, so S(a + b) = S(a) + S(b)), the structure
of the recursive-halving merge (Alg. 1 and the non-power-of-two rule of Sec. III-A), the
output contract of Alg. 2 (exact values on the selected set, zero elsewhere), brute force
on tiny inputs, or fp32 arithmetic as numpy performs it.  ``test_oracle_mutations`` plants
plausible mistakes in copies of the oracle and checks that these pins catch them.
"""

import math
import os

import numpy as np
import pytest

import oracle

P61 = (1 << 61) - 1
GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ---- coefficients ------------------------------------------------------------------------

def test_splitmix64_published_vector():
    lines = [l.strip() for l in open(os.path.join(GOLDEN, "splitmix64_seed1234567.txt"))
             if l.strip() and not l.startswith("#")]
    seed = int(lines[0].split()[1])
    want = [int(x) for x in lines[1:]]
    gen = oracle.splitmix64(seed)
    assert [next(gen) for _ in want] == want


def test_coefficients_ranges_and_order():
    for seed in (0, 1, 42, 2**64 - 1):
        a, b, a2, b2 = oracle.derive_coefficients(16, seed)
        assert all(1 <= v <= P61 - 1 for v in a + a2)
        assert all(0 <= v <= P61 - 1 for v in b + b2)
    # four draws per row in the order a, b, a', b'
    gen = oracle.splitmix64(7)
    draws = [next(gen) for _ in range(8)]
    a, b, a2, b2 = oracle.derive_coefficients(2, 7)
    for j in range(2):
        assert a[j] == 1 + draws[4 * j] % (P61 - 1)
        assert b[j] == draws[4 * j + 1] % P61
        assert a2[j] == 1 + draws[4 * j + 2] % (P61 - 1)
        assert b2[j] == draws[4 * j + 3] % P61
    assert oracle.derive_coefficients(3, 5) != oracle.derive_coefficients(3, 6)


# ---- hash family -------------------------------------------------------------------------

EXTREME_COEFFS = [
    ([1], [0], [1], [0]),
    ([P61 - 1], [P61 - 1], [P61 - 1], [P61 - 1]),
    ([2**60 + 12345], [2**61 - 2], [3], [2**31 - 1]),
    ([2**31 - 1], [2**31], [2**61 - 3], [1]),
    ([(1 << 61) - (1 << 30)], [12345678901234567], [987654321987654], [P61 - 2]),
]


@pytest.mark.parametrize("c", [1, 2, 7, 1 << 14, 1000003, 1 << 26])
def test_hash_numpy_matches_bigint(c):
    rng = np.random.default_rng(c)
    idx = np.concatenate([np.array([0, 1, 2, 3, 2**31 - 1, 2**31 - 2, 2**30, 11173961]),
                          rng.integers(0, 2**31, 4000)]).astype(np.uint64)
    coef_sets = EXTREME_COEFFS + [tuple(oracle.derive_coefficients(3, c))]
    for co in coef_sets:
        buckets, signs = oracle.hash_rows(co, c, idx)
        for j in range(len(co[0])):
            for t, i in enumerate(idx.tolist()):
                assert buckets[j, t] == oracle.bucket_exact(co[0][j], co[1][j], c, i)
                assert signs[j, t] == oracle.sign_exact(co[2][j], co[3][j], i)


def test_hash_identity_and_negation_closed_forms():
    i = np.arange(0, 2**31, 9973, dtype=np.uint64)
    c = 1 << 20
    # a = 1, b = 0: h(i) = i mod c; sign = parity of i
    b1, s1 = oracle.hash_rows(([1], [0], [1], [0]), c, i)
    assert np.array_equal(b1[0], (i % c).astype(np.int64))
    assert np.array_equal(s1[0], np.where(i % 2 == 0, 1, -1))
    # a = p - 1 = -1 (mod p), b = 0: h(i) = (p - i) mod c for i > 0
    b2, _ = oracle.hash_rows(([P61 - 1], [0], [1], [0]), c, i[1:])
    want = np.array([(P61 - int(v)) % c for v in i[1:]], dtype=np.int64)
    assert np.array_equal(b2[0], want)


def test_hash_rejects_large_coordinates():
    with pytest.raises(ValueError):
        oracle.hash_rows(([1], [0], [1], [0]), 8, np.array([2**31], dtype=np.uint64))


# ---- accumulate --------------------------------------------------------------------------

def test_accumulate_equals_numpy_fp32_arithmetic():
    rng = np.random.default_rng(0)
    n = 200_000
    u = (rng.standard_normal(n) * 10.0 ** rng.integers(-30, 5, n)).astype(np.float32)
    e = (rng.standard_normal(n) * 10.0 ** rng.integers(-30, 5, n)).astype(np.float32)
    g = (rng.standard_normal(n) * 10.0 ** rng.integers(-30, 5, n)).astype(np.float32)
    for rho in (0.9, 0.5, 0.0, 0.999):
        u1, e1 = oracle.accumulate(u, e, g, rho)
        r32 = np.float32(rho)
        uw = (r32 * u) + g          # numpy float32 ops: one rounding each, never fused
        ew = e + uw
        assert uw.dtype == np.float32
        assert np.array_equal(u1.view(np.uint32), uw.view(np.uint32))
        assert np.array_equal(e1.view(np.uint32), ew.view(np.uint32))


def test_accumulate_closed_form_dyadic():
    # rho = 1/2, g = 1 every step, u_0 = e_0 = 0:
    #   u_t = 2 - 2^(1-t),  e_t = 2t - 2 + 2^(1-t)   (exact in fp32 for small t)
    u = np.zeros(3, np.float32)
    e = np.zeros(3, np.float32)
    g = np.ones(3, np.float32)
    for t in range(1, 20):
        u, e = oracle.accumulate(u, e, g, 0.5)
        assert np.all(u == 2.0 - 2.0 ** (1 - t))
        assert np.all(e == 2.0 * t - 2.0 + 2.0 ** (1 - t))


# ---- sketch ------------------------------------------------------------------------------

def _dyadic(rng, n, lo=-512, hi=512, scale=2.0**-10):
    return (rng.integers(lo, hi, n) * scale).astype(np.float32)


@pytest.mark.parametrize("r,c", [(1, 1), (3, 17), (5, 1 << 10), (7, 4096)])
def test_sketch_linearity_exact(r, c):
    rng = np.random.default_rng(r * c)
    co = oracle.derive_coefficients(r, 99 + c)
    x1, x2 = _dyadic(rng, 5000), _dyadic(rng, 5000)
    T1, _ = oracle.sketch(x1, co, c)
    T2, _ = oracle.sketch(x2, co, c)
    T12, _ = oracle.sketch(x1 + x2, co, c)   # x1 + x2 exact in fp32 for these values
    assert np.array_equal(T1 + T2, T12)
    Tm, _ = oracle.sketch(-3.0 * x1, co, c)  # homogeneity, exact for a power-of-two-ish 3
    assert np.array_equal(Tm, -3.0 * T1)


def test_sketch_row_sums_and_magnitudes():
    rng = np.random.default_rng(3)
    d, r, c = 3000, 5, 64
    co = oracle.derive_coefficients(r, 3)
    x = _dyadic(rng, d)
    T, A = oracle.sketch(x, co, c)
    for j in range(r):
        want = sum(oracle.sign_exact(co[2][j], co[3][j], i) * float(x[i]) for i in range(d))
        assert T[j].sum() == want
        assert A[j].sum() == np.abs(x.astype(np.float64)).sum()
        assert np.all(np.abs(T[j]) <= A[j])


def test_single_spike_recovery():
    d, r, c = 5000, 5, 1024
    co = oracle.derive_coefficients(r, 11)
    for i, v in ((0, 0.75), (1234, -3.5), (d - 1, 2.0**-20)):
        x = np.zeros(d, np.float32)
        x[i] = v
        T, _ = oracle.sketch(x, co, c)
        est = oracle.query(T, co, d)
        assert est[i] == v
        assert list(oracle.topk(est, 1)) == [i]
        # every other coordinate sees v in at most some rows, so |est| <= |v|
        assert np.all(np.abs(est) <= abs(v))


def _injective_coeffs(r, seed):
    """Rows with a = 1 and distinct offsets: h_j(i) = (i + b_j) mod c, injective for c >= d."""
    rng = np.random.default_rng(seed)
    a = [1] * r
    b = [int(v) for v in rng.integers(0, 2**40, r)]
    a2 = [int(v) for v in rng.integers(1, 2**60, r)]
    b2 = [int(v) for v in rng.integers(0, 2**60, r)]
    return a, b, a2, b2


@pytest.mark.parametrize("r", [1, 3, 4, 5])
def test_collision_free_sketch_is_exact(r):
    rng = np.random.default_rng(r)
    d = 700
    co = _injective_coeffs(r, r)
    x = rng.standard_normal(d).astype(np.float32)
    x[::7] = x[1::7][: x[::7].size]            # plant exact ties of |x|
    T, _ = oracle.sketch(x, co, c=d)
    est = oracle.query(T, co, d)
    assert np.array_equal(est, x.astype(np.float64))
    for k in (1, 5, 100, d):
        brute = sorted(range(d), key=lambda i: (-abs(float(x[i])), i))[:k]
        assert list(oracle.topk(est, k)) == sorted(brute)


@pytest.mark.parametrize("r", [3, 4, 5, 7])
def test_median_ignores_one_contaminated_row(r):
    # row 0: h(i) = 2i mod d, so i and i + d/2 share a bucket; other rows injective.
    rng = np.random.default_rng(10 + r)
    d = 512
    a, b, a2, b2 = _injective_coeffs(r, 20 + r)
    a[0], b[0] = 2, 0
    co = (a, b, a2, b2)
    x = rng.standard_normal(d).astype(np.float32)
    T, _ = oracle.sketch(x, co, c=d)
    est = oracle.query(T, co, d)
    assert np.array_equal(est, x.astype(np.float64))


def test_sketch_bruteforce_tiny():
    rng = np.random.default_rng(5)
    d, r, c = 40, 3, 7
    co = oracle.derive_coefficients(r, 5)
    x = rng.standard_normal(d).astype(np.float32)
    T, A = oracle.sketch(x, co, c)
    for j in range(r):
        cells = [[] for _ in range(c)]
        for i in range(d):
            cells[oracle.bucket_exact(co[0][j], co[1][j], c, i)].append(
                oracle.sign_exact(co[2][j], co[3][j], i) * float(x[i]))
        for bkt in range(c):
            assert math.isclose(T[j][bkt], math.fsum(cells[bkt]), rel_tol=1e-14, abs_tol=1e-14)
            assert math.isclose(A[j][bkt], math.fsum(abs(v) for v in cells[bkt]),
                                rel_tol=1e-14, abs_tol=1e-14)


def test_count_sketch_error_bound():
    """Accuracy sanity (not parity): with c buckets each row errs by about ||x||_2/sqrt(c);
    by Chebyshev a row exceeds 3||x||_2/sqrt(c) with probability <= 1/9, and the median of
    5 rows only when 3 rows do: probability <= 10/729 < 1.4 %."""
    rng = np.random.default_rng(8)
    d, r, c = 200_000, 5, 4096
    co = oracle.derive_coefficients(r, 8)
    x = (rng.standard_normal(d) * 1e-3).astype(np.float32)
    heavy = rng.choice(d, 20, replace=False)
    x[heavy] = np.float32(0.5)
    T, _ = oracle.sketch(x, co, c)
    est = oracle.query(T, co, d)
    eps = 3.0 / math.sqrt(c)
    err = np.abs(est - x.astype(np.float64))
    assert np.mean(err > eps * np.linalg.norm(x.astype(np.float64))) < 10 / 729
    assert set(oracle.topk(est, 20).tolist()) == set(heavy.tolist())


# ---- merge -------------------------------------------------------------------------------

def test_merge_schedule_structure():
    S = oracle.merge_schedule
    assert S(1) == []
    assert S(2) == [[(0, 1)]]
    assert S(4) == [[(0, 1), (2, 3)], [(0, 2)]]
    assert S(5) == [[(0, 1), (2, 3)], [(0, 2)], [(0, 4)]]
    assert S(6) == [[(0, 1), (2, 3), (4, 5)], [(0, 2)], [(0, 4)]]
    for P in range(1, 70):
        rounds = S(P)
        assert len(rounds) == (0 if P == 1 else math.ceil(math.log2(P)))
        sent, alive = set(), set(range(P))
        for pairs in rounds:
            involved = [q for pr in pairs for q in pr]
            assert len(involved) == len(set(involved))          # one message per worker
            for recv, send in pairs:
                assert recv < send and recv in alive and send in alive
                sent.add(send)
                alive.discard(send)
            # with an odd number of participants only the largest id sits out
            step = 2 ** rounds.index(pairs)
            parts = list(range(0, P, step))
            idle = [q for q in parts if q not in involved]
            assert idle == ([parts[-1]] if len(parts) % 2 else [])
        assert alive == {0} and sent == set(range(1, P))


@pytest.mark.parametrize("P", [1, 2, 3, 4, 5, 6, 7, 8, 9, 16, 32])
def test_merge_equals_flat_sum_and_is_order_invariant(P):
    rng = np.random.default_rng(P)
    tabs = [(rng.integers(-2**20, 2**20, (3, 50)) * 2.0**-12) for _ in range(P)]
    flat = np.sum(tabs, axis=0)
    assert np.array_equal(oracle.merge_tree(tabs), flat)
    perm = rng.permutation(P)
    assert np.array_equal(oracle.merge_tree([tabs[q] for q in perm]), flat)


def test_merge_of_sketches_is_sketch_of_sum():
    rng = np.random.default_rng(12)
    r, c, d, P = 5, 256, 4000, 6
    co = oracle.derive_coefficients(r, 12)
    xs = [_dyadic(rng, d, -64, 64, 2.0**-6) for _ in range(P)]
    sk = [oracle.sketch(x, co, c) for x in xs]
    merged = oracle.merge_tree([t for t, _ in sk])
    total = np.sum(np.stack(xs).astype(np.float64), axis=0).astype(np.float32)
    assert np.array_equal(merged, oracle.sketch(total, co, c)[0])
    # the same with the fp64 sum itself, and the magnitude tables: the merge of the workers'
    # magnitude tables is the magnitude table of sum_p |x_p|
    total64 = np.sum(np.stack(xs).astype(np.float64), axis=0)
    assert np.array_equal(merged, oracle.sketch(total64, co, c)[0])
    abs64 = np.sum(np.abs(np.stack(xs).astype(np.float64)), axis=0)
    assert np.array_equal(oracle.merge_tree([a for _, a in sk]), oracle.sketch(abs64, co, c)[1])


# ---- top-k -------------------------------------------------------------------------------

@pytest.mark.parametrize("seed", range(6))
def test_topk_bruteforce_with_ties(seed):
    rng = np.random.default_rng(seed)
    d = int(rng.integers(1, 65))
    est = rng.choice(np.array([0.0, 1.0, -1.0, 2.5, -2.5, 0.25, 3.0]), d)
    for k in range(1, d + 1):
        brute = sorted(range(d), key=lambda i: (-abs(est[i]), i))[:k]
        assert list(oracle.topk(est, k)) == sorted(brute)


def test_topk_matches_stable_argsort():
    rng = np.random.default_rng(4)
    est = np.round(rng.standard_normal(100_000), 2)
    k = 1234
    ref = np.sort(np.argsort(-np.abs(est), kind="stable")[:k])
    assert np.array_equal(oracle.topk(est, k), ref)


# ---- second round ------------------------------------------------------------------------

def test_gather_and_zero_conservation():
    rng = np.random.default_rng(21)
    d, P, k = 10_000, 8, 300
    us = [_dyadic(rng, d) for _ in range(P)]
    es = [_dyadic(rng, d) for _ in range(P)]
    idx = np.sort(rng.choice(d, k, replace=False))
    vals, us2, es2 = oracle.gather_and_zero(us, es, idx)
    before = np.sum([e.astype(np.float64) for e in es], axis=0)
    after = np.sum([e.astype(np.float64) for e in es2], axis=0)
    full = after.copy()
    full[idx] += vals
    assert np.array_equal(full, before)
    mask = np.ones(d, bool)
    mask[idx] = False
    for p in range(P):
        assert np.all(us2[p][idx] == 0) and np.all(es2[p][idx] == 0)
        assert np.array_equal(us2[p][mask].view(np.uint32), us[p][mask].view(np.uint32))
        assert np.array_equal(es2[p][mask].view(np.uint32), es[p][mask].view(np.uint32))


def test_step_output_contract():
    """Alg. 2: exact (accumulated) values on the selected set, untouched accumulators
    elsewhere; the selected set is the top-k of the estimate."""
    rng = np.random.default_rng(31)
    d, P, r, c, k = 5000, 4, 5, 512, 40
    co = oracle.derive_coefficients(r, 31)
    us = [np.zeros(d, np.float32) for _ in range(P)]
    es = [np.zeros(d, np.float32) for _ in range(P)]
    spikes = rng.choice(d, 10, replace=False)
    for t in range(3):
        gs = [(rng.standard_normal(d) * 1e-3).astype(np.float32) for _ in range(P)]
        for g in gs:
            g[spikes] += np.float32(0.1)
        res = oracle.step(us, es, gs, 0.9, co, c, k)
        assert np.array_equal(res.idx, oracle.topk(res.est, k))
        assert set(spikes.tolist()) <= set(res.idx.tolist())
        want = np.sum([e[res.idx].astype(np.float64) for e in res.es_pre], axis=0)
        assert np.array_equal(res.vals, want)
        us, es = res.us, res.es


# ---- weight update -----------------------------------------------------------------------

def test_apply_update_equals_numpy_fp32():
    rng = np.random.default_rng(55)
    d, k = 50_000, 700
    w = (rng.standard_normal(d) * 10.0 ** rng.integers(-5, 3, d)).astype(np.float32)
    idx = np.sort(rng.choice(d, k, replace=False))
    vals = (rng.standard_normal(k) * 10.0 ** rng.integers(-8, 2, k)).astype(np.float32)
    for lr in (0.1, 0.03, 1.0):
        got = oracle.apply_update(w, idx, vals, lr)
        want = w.copy()
        want[idx] = w[idx] - np.float32(lr) * vals      # numpy fp32: two roundings, no fusion
        assert np.array_equal(got.view(np.uint32), want.view(np.uint32))
        mask = np.ones(d, bool)
        mask[idx] = False
        assert np.array_equal(got[mask], w[mask])


def test_apply_update_closed_form():
    w = np.full(8, 3.0, np.float32)
    out = oracle.apply_update(w, [1, 5], np.array([2.0, -4.0], np.float32), 0.5)
    assert out.tolist() == [3.0, 2.0, 3.0, 3.0, 3.0, 5.0, 3.0, 3.0]


# ---- HEAVYMIX ----------------------------------------------------------------------------

def test_splitmix64_counter_form_matches_stream():
    lines = [l.strip() for l in open(os.path.join(GOLDEN, "splitmix64_seed1234567.txt"))
             if l.strip() and not l.startswith("#")]
    want = [int(x) for x in lines[1:]]
    assert [int(v) for v in oracle.splitmix64_at(1234567, np.arange(5))] == want
    for seed in (0, 99, 2**64 - 1):
        gen = oracle.splitmix64(seed)
        stream = [next(gen) for _ in range(50)]
        assert [int(v) for v in oracle.splitmix64_at(seed, np.arange(50))] == stream


def _heavymix_fixture(seed, d=600, r=5):
    rng = np.random.default_rng(seed)
    co = _injective_coeffs(r, seed)
    x = _dyadic(rng, d, -64, 64, 2.0**-6)
    x[rng.choice(d, 12, replace=False)] = np.float32(8.0)
    T, _ = oracle.sketch(x, co, c=d)
    return co, x, T


def test_heavymix_l2_estimate_and_h():
    co, x, T = _heavymix_fixture(1)
    d, k = x.size, 20
    idx, est, l2sq = oracle.heavymix(T, co, d, k, fill_seed=3)
    assert np.array_equal(est, x.astype(np.float64))           # collision-free rows
    assert l2sq == np.sum(x.astype(np.float64) ** 2)           # every row holds ||x||^2
    spikes = np.nonzero(x == 8.0)[0]
    assert set(spikes.tolist()) <= set(idx.tolist()) and idx.size == k


def test_heavymix_h_bound_and_large_h_branch():
    # with exact estimates sum_{i in H} x_i^2 >= |H| l2sq / k forces |H| <= k ...
    rng = np.random.default_rng(6)
    x = rng.standard_normal(2000)
    for k in (1, 5, 50, 500):
        h = x * x >= np.sum(x * x) / k
        assert h.sum() <= k
    # ... so |H| > k comes from estimation noise; with an underestimated l2sq, H is a
    # superset of the top-k and the top-k of H by |est| is the plain top-k, ties by index
    est = np.array([3.0, -5.0, 5.0, 1.0, 4.0, -4.0, 0.5])
    idx = oracle.heavymix_select(est, l2sq=1.0, k=3, fill_seed=0)   # H = |est| >= 0.577...
    assert idx.tolist() == [1, 2, 4]
    assert np.array_equal(idx, oracle.topk(est, 3))


def test_heavymix_random_fill_brute_force():
    co, x, T = _heavymix_fixture(2)
    d, k, seed = x.size, 200, 12345
    idx, _, l2sq = oracle.heavymix(T, co, d, k, fill_seed=seed)
    h = [i for i in range(d) if float(x[i]) ** 2 >= l2sq / k]
    assert len(h) < k
    xi = {i: int(oracle.splitmix64_at(seed, [i])[0]) >> 33 for i in range(d)}
    nh = sorted((i for i in range(d) if i not in set(h)), key=lambda i: (xi[i], i))
    assert sorted(h + nh[: k - len(h)]) == idx.tolist()


def test_heavymix_select_brute_force_threshold_on_the_square():
    """H = {i : est_i^2 >= l2sq / k}, written out per coordinate, with estimates on both
    sides of sqrt(l2sq / k) and of l2sq / k itself (where a threshold on |est| would differ),
    and the fill by (xi_i, i) over the rest."""
    est = np.array([3.0, -2.0, 1.9, 2.5, -0.7, 0.1, 4.5, -3.9, 0.05, 1.0, -2.1, 0.3])
    d = est.size
    # |H| >= k (top-k of H) and |H| < k (H plus the fill), with est_i^2 exactly at the threshold
    # for i = 1 (l2sq / k = 4) in several of them
    for k, l2sq, seed in [(3, 12.0, 0), (4, 16.0, 9), (5, 20.0, 77), (2, 8.0, 2**64 - 5), (6, 3.0, 1),
                          (8, 32.0, 5), (10, 40.0, 12345), (9, 36.0, 2**63), (11, 176.0, 7), (12, 1e6, 3)]:
        thr = l2sq / k
        h = [i for i in range(d) if est[i] * est[i] >= thr]
        if len(h) >= k:
            want = sorted(sorted(h, key=lambda i: (-abs(est[i]), i))[:k])
        else:
            xi = {i: int(oracle.splitmix64_at(seed, [i])[0]) >> 33 for i in range(d)}
            rest = sorted((i for i in range(d) if i not in h), key=lambda i: (xi[i], i))
            want = sorted(h + rest[: k - len(h)])
        assert oracle.heavymix_select(est, l2sq, k, seed).tolist() == want


def test_heavymix_fill_is_uniform():
    co, x, T = _heavymix_fixture(4, d=300)
    d, k = x.size, 60
    counts = np.zeros(d)
    trials = 400
    for seed in range(trials):
        idx, _, l2sq = oracle.heavymix(T, co, d, k, fill_seed=seed)
        counts[idx] += 1
    in_h = x.astype(np.float64) ** 2 >= l2sq / k
    assert np.all(counts[in_h] == trials)
    nh = ~in_h
    p = (k - in_h.sum()) / nh.sum()
    z = (counts[nh] - trials * p) / np.sqrt(trials * p * (1 - p))
    assert abs(z.mean()) < 0.2 and np.max(np.abs(z)) < 5.0


# ---- momentum and error kept as sketches -------------------------------------------------

def test_sketch_sparse_is_sketch_of_dense():
    rng = np.random.default_rng(61)
    d, r, c = 3000, 5, 256
    co = oracle.derive_coefficients(r, 61)
    idx = np.sort(rng.choice(d, 40, replace=False))
    vals = _dyadic(rng, 40)
    dense = np.zeros(d, np.float32)
    dense[idx] = vals
    T, A = oracle.sketch_sparse(idx, vals, co, c)
    T2, A2 = oracle.sketch(dense, co, c)
    assert np.array_equal(T, T2) and np.array_equal(A, A2)
    assert np.array_equal(oracle.query_at(T, co, idx), oracle.query(T, co, d)[idx])


def test_sketched_state_removal_and_momentum_closed_form():
    # collision-free rows: every estimate is exact, so after the step the selected
    # coordinates read exactly 0 in both sketches and everything else is untouched
    rng = np.random.default_rng(62)
    d, r, k, P = 500, 3, 20, 4
    co = _injective_coeffs(r, 62)
    zeros = np.zeros((r, d))
    gs = [_dyadic(rng, d, -64, 64, 2.0**-6) for _ in range(P)]
    res = oracle.sketched_state_step(zeros, zeros, zeros, zeros, gs, 0.5, co, d, k)
    total = np.sum(np.stack(gs).astype(np.float64), axis=0)
    assert np.array_equal(res.est, total)          # U = S, E = U after the first step
    assert np.array_equal(res.idx, oracle.topk(total, k))
    assert np.array_equal(res.delta, total[res.idx])
    assert np.all(oracle.query_at(res.E, co, res.idx) == 0)
    assert np.all(oracle.query_at(res.U, co, res.idx) == 0)
    rest = np.setdiff1d(np.arange(d), res.idx)
    assert np.array_equal(oracle.query_at(res.E, co, rest), total[rest])
    # momentum/error recursion, rho = 1/2, g = 1/4 everywhere, k = 1: step t takes
    # coordinate t - 1 (all remaining ones tie and the smaller index wins), and every
    # coordinate not yet taken follows U_t = (2 - 2^(1-t))/4, E_t = (2t - 2 + 2^(1-t))/4
    g = [np.full(d, 0.25, np.float32)]
    U = E = AU = AE = np.zeros((r, d))
    for t in range(1, 6):
        res = oracle.sketched_state_step(U, E, AU, AE, g, 0.5, co, d, 1)
        U, E, AU, AE = res.U, res.E, res.AU, res.AE
        assert res.idx.tolist() == [t - 1]
        rest = np.arange(t, d)
        assert np.all(oracle.query_at(U, co, rest) == (2 - 2.0 ** (1 - t)) / 4)
        assert np.all(oracle.query_at(E, co, rest) == (2 * t - 2 + 2.0 ** (1 - t)) / 4)
        assert oracle.query_at(E, co, [t - 1])[0] == 0 and oracle.query_at(U, co, [t - 1])[0] == 0


# ---- pieces of a long vector (linearity over disjoint coordinate ranges) ------------------

def test_sketch_in_pieces_equals_whole():
    """Sec. III-A's linearity over a partition of the coordinates: sketching x piece by piece,
    each piece hashed at its own global coordinates, and summing gives exactly the sketch of x
    (dyadic values: every sum is exact in fp64).  The same holds for the magnitude table, and
    the median query evaluated piece by piece concatenates to the whole query."""
    rng = np.random.default_rng(31)
    d, r, c = 10_007, 5, 97
    co = oracle.derive_coefficients(r, 31)
    x = _dyadic(rng, d, -1000, 1000, 2.0**-10)
    T, A = oracle.sketch(x, co, c)
    Tp, Ap = np.zeros_like(T), np.zeros_like(A)
    cuts = [0, 1, 17, 4096, 4097, 9000, d]
    for a, b in zip(cuts[:-1], cuts[1:]):
        t, m = oracle.sketch(x[a:b], co, c, idx=np.arange(a, b))
        Tp += t
        Ap += m
    assert np.array_equal(T, Tp) and np.array_equal(A, Ap)
    est = oracle.query(T, co, d)
    parts = [oracle.query(T, co, b - a, idx=np.arange(a, b)) for a, b in zip(cuts[:-1], cuts[1:])]
    assert np.array_equal(est, np.concatenate(parts))
    # a piece hashed at the wrong coordinates (its local 0 .. n-1) does not give the sketch
    bad = sum(oracle.sketch(x[a:b], co, c)[0] for a, b in zip(cuts[:-1], cuts[1:]))
    assert not np.array_equal(bad, T)


def test_topk_by_threshold_equals_topk():
    """The partition-based top-k returns exactly the sorted definition's set, with heavy ties
    (including ties at the k-th value) and with k = 1 and k = d."""
    rng = np.random.default_rng(32)
    for trial in range(40):
        d = int(rng.integers(1, 400))
        est = rng.integers(-6, 7, d).astype(np.float64) * (0.5 if trial % 2 else 1.0)
        for k in {1, d, int(rng.integers(1, d + 1))}:
            assert np.array_equal(oracle.topk_by_threshold(est, k), oracle.topk(est, k))
