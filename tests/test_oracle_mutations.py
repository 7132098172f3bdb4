"""Plant plausible mistakes in the oracle (on the CPU) and check that the pins catch them.

Each case swaps one oracle function for a subtly wrong variant, runs the pin that should
detect it, and expects that pin to fail.
"""

import numpy as np
import pytest

import oracle
from oracle import countsketch as cs
from oracle import gssgd
import tests.test_oracle_pins as pins


def _query_without_sign(T, coeffs, d):
    c = T.shape[1]
    buckets, _ = cs.hash_rows(coeffs, c, np.arange(d, dtype=np.uint64))
    vals = np.stack([T[j][buckets[j]] for j in range(buckets.shape[0])])
    return np.median(vals, axis=0)


def _query_mean(T, coeffs, d):
    c = T.shape[1]
    buckets, signs = cs.hash_rows(coeffs, c, np.arange(d, dtype=np.uint64))
    vals = np.stack([signs[j] * T[j][buckets[j]] for j in range(buckets.shape[0])])
    return vals.mean(axis=0)


def _accumulate_fused(u, e, g, rho):
    r = np.float64(np.float32(rho))
    u1 = (r * u.astype(np.float64) + g.astype(np.float64)).astype(np.float32)   # one rounding
    return u1, (e.astype(np.float64) + u1).astype(np.float32)


def _accumulate_wrong_error(u, e, g, rho):
    u1, _ = gssgd.accumulate(u, e, g, rho)
    return u1, (e.astype(np.float64) + g.astype(np.float64)).astype(np.float32)


def _merge_drop_odd(tables):
    work = [np.array(t, dtype=np.float64) for t in tables]
    while len(work) > 1:
        work = [work[m] + work[m + 1] for m in range(0, len(work) - 1, 2)]
    return work[0]


def _topk_ties_high(est, k):
    est = np.asarray(est, dtype=np.float64)
    order = np.lexsort((-np.arange(est.size), -np.abs(est)))
    return np.sort(order[:k])


def _affine_mod_2_61(a, b, i):
    m = np.uint64((1 << 61) - 1)
    return (np.uint64(a) * i + np.uint64(b)) & m


MUTATIONS = [
    ("query", _query_without_sign, pins.test_collision_free_sketch_is_exact, {"r": 3}),
    ("query", _query_mean, pins.test_median_ignores_one_contaminated_row, {"r": 5}),
    ("accumulate", _accumulate_fused, pins.test_accumulate_equals_numpy_fp32_arithmetic, {}),
    ("accumulate", _accumulate_wrong_error, pins.test_accumulate_closed_form_dyadic, {}),
    ("merge_tree", _merge_drop_odd, pins.test_merge_equals_flat_sum_and_is_order_invariant,
     {"P": 5}),
    ("topk", _topk_ties_high, pins.test_topk_bruteforce_with_ties, {"seed": 0}),
]


@pytest.mark.parametrize("name,bad,pin,kw", MUTATIONS, ids=[m[1].__name__ for m in MUTATIONS])
def test_pin_catches_mutation(monkeypatch, name, bad, pin, kw):
    monkeypatch.setattr(oracle, name, bad)
    with pytest.raises(AssertionError):
        pin(**kw)


def test_pin_catches_wrong_modulus(monkeypatch):
    monkeypatch.setattr(cs, "_affine_mod_p", _affine_mod_2_61)
    with pytest.raises(AssertionError):
        pins.test_hash_numpy_matches_bigint(1 << 14)
