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


# ---- the later oracle functions (weight update, HEAVYMIX, sketched state) -----------------

_REAL = {n: getattr(gssgd, n) for n in ("apply_update", "gather_and_zero", "heavymix_select",
                                         "sketched_state_step", "merge_schedule", "sketch",
                                         "heavymix_select_from")}
_REAL["derive_coefficients"] = cs.derive_coefficients
_REAL["splitmix64_at"] = cs.splitmix64_at


def _apply_update_fused(w, idx, vals, lr):
    out = np.array(w, dtype=np.float32, copy=True)
    idx = np.asarray(idx)
    v = np.asarray(vals, dtype=np.float64)
    out[idx] = (out[idx].astype(np.float64) - np.float64(np.float32(lr)) * v).astype(np.float32)  # one rounding
    return out


def _apply_update_ascent(w, idx, vals, lr):
    return _REAL["apply_update"](w, idx, -np.asarray(vals, dtype=np.float32), lr)


def _gather_keeps_momentum(us, es, idx):
    vals, _, es2 = _REAL["gather_and_zero"](us, es, idx)
    return vals, [np.array(u, copy=True) for u in us], es2


def _gather_sums_momentum(us, es, idx):
    _, us2, es2 = _REAL["gather_and_zero"](us, es, idx)
    return np.sum([u[np.asarray(idx)].astype(np.float64) for u in us], axis=0), us2, es2


def _merge_schedule_first_idles(P):
    rounds, step = [], 1
    while step < P:
        parts = list(range(0, P, step))
        if len(parts) % 2:
            parts = parts[1:]          # the smallest id sits the round out
        rounds.append([(parts[m], parts[m + 1]) for m in range(0, len(parts) - 1, 2)])
        step *= 2
    return rounds


def _heavymix_threshold_on_abs(est, l2sq, k, fill_seed):
    # |est| >= l2sq / k in place of est^2 >= l2sq / k
    return _REAL["heavymix_select"](est, k * (l2sq / k) ** 2, k, fill_seed)


def _splitmix64_at_off_by_one(seed, idx):
    return _REAL["splitmix64_at"](seed, np.asarray(idx, dtype=np.uint64) + np.uint64(1))


def _coefficients_draw_order(r, seed):
    a, b, a2, b2 = _REAL["derive_coefficients"](r, seed)
    return a, a2, b, b2                # draws taken as a, a', b, b'


def _sketched_state_keeps_momentum(U, E, AU, AE, gs, rho, coeffs, c, k, rel=1e-5):
    res = _REAL["sketched_state_step"](U, E, AU, AE, gs, rho, coeffs, c, k, rel)
    res.U = res.U_pre                  # the extracted mass not removed from U
    return res


def _sketched_state_error_from_s(U, E, AU, AE, gs, rho, coeffs, c, k, rel=1e-5):
    res = _REAL["sketched_state_step"](U, E, AU, AE, gs, rho, coeffs, c, k, rel)
    res.E = res.E - res.U_pre + res.S  # E <- E + S in place of E + U
    return res


def _topk_threshold_ties_high(est, k):
    a = np.abs(np.asarray(est, dtype=np.float64))
    tau = np.partition(a, a.size - k)[a.size - k]
    gt = np.nonzero(a > tau)[0]
    eq = np.nonzero(a == tau)[0]
    return np.sort(np.concatenate([gt, eq[eq.size - (k - gt.size):]])).astype(np.int64)  # larger indices


def _sketch_ignores_global_coordinates(x, coeffs, c, hashes=None, idx=None):
    return _REAL["sketch"](x, coeffs, c, hashes)       # every piece hashed at 0 .. len - 1


def _heavymix_members_strict(est, l2sq, k):
    est = np.asarray(est, dtype=np.float64)
    return est * est > l2sq / k                          # > in place of >=


def _heavymix_fill_largest_xi(in_h, est, k, fill_seed):
    in_h = np.asarray(in_h, dtype=bool)
    if int(in_h.sum()) >= k:
        return _REAL["heavymix_select_from"](in_h, est, k, fill_seed)
    NH = np.nonzero(~in_h)[0]
    xi = (cs.splitmix64_at(fill_seed, NH) >> np.uint64(33)).astype(np.int64)
    fill = NH[np.lexsort((NH, -xi))[: k - int(in_h.sum())]]   # largest xi first
    return np.sort(np.concatenate([np.nonzero(in_h)[0], fill])).astype(np.int64)


LATER = [
    ("topk_by_threshold", _topk_threshold_ties_high, pins.test_topk_by_threshold_equals_topk, {}),
    ("sketch", _sketch_ignores_global_coordinates, pins.test_sketch_in_pieces_equals_whole, {}),
    ("heavymix_members", _heavymix_members_strict, pins.test_heavymix_select_brute_force_threshold_on_the_square,
     {}),
    ("heavymix_select_from", _heavymix_fill_largest_xi, pins.test_heavymix_select_brute_force_threshold_on_the_square,
     {}),
    ("heavymix_select_from", _heavymix_fill_largest_xi, pins.test_heavymix_random_fill_brute_force, {}),
    ("apply_update", _apply_update_fused, pins.test_apply_update_equals_numpy_fp32, {}),
    ("apply_update", _apply_update_ascent, pins.test_apply_update_closed_form, {}),
    ("gather_and_zero", _gather_keeps_momentum, pins.test_gather_and_zero_conservation, {}),
    ("gather_and_zero", _gather_sums_momentum, pins.test_gather_and_zero_conservation, {}),
    ("merge_schedule", _merge_schedule_first_idles, pins.test_merge_schedule_structure, {}),
    ("heavymix_select", _heavymix_threshold_on_abs, pins.test_heavymix_select_brute_force_threshold_on_the_square,
     {}),
    ("splitmix64_at", _splitmix64_at_off_by_one, pins.test_splitmix64_counter_form_matches_stream, {}),
    ("derive_coefficients", _coefficients_draw_order, pins.test_coefficients_ranges_and_order, {}),
    ("sketched_state_step", _sketched_state_keeps_momentum,
     pins.test_sketched_state_removal_and_momentum_closed_form, {}),
    ("sketched_state_step", _sketched_state_error_from_s,
     pins.test_sketched_state_removal_and_momentum_closed_form, {}),
]


@pytest.mark.parametrize("name,bad,pin,kw", LATER, ids=[m[1].__name__ for m in LATER])
def test_pin_catches_mutation_in_later_functions(monkeypatch, name, bad, pin, kw):
    # patched where the pins call it and where other oracle functions call it
    monkeypatch.setattr(oracle, name, bad)
    for mod in (gssgd, cs):
        if hasattr(mod, name):
            monkeypatch.setattr(mod, name, bad)
    with pytest.raises(AssertionError):
        pin(**kw)


def test_pin_catches_wrong_modulus(monkeypatch):
    monkeypatch.setattr(cs, "_affine_mod_p", _affine_mod_2_61)
    with pytest.raises(AssertionError):
        pins.test_hash_numpy_matches_bigint(1 << 14)
