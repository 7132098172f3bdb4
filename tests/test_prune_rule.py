"""The row-skipping rule of the median query and the integer shortcuts of its kernels, checked
on the host (no GPU).

The query stops reading a coordinate's rows once, with f = r/2 + 1, at least f of the signed
cells read so far are < t and at least f are > -t.  The claim that makes this safe: then the
fp32 median (the middle value for odd r, the fp32 mean of the two middle values for even r)
lies strictly inside (-t, t), whatever the unread cells hold.  Here the unread cells are drawn
adversarially (huge, of either sign, or at +-t) and t is taken at and next to the cells.
"""

from __future__ import annotations

import numpy as np
import pytest


def median_fp32(v: np.ndarray) -> np.float32:
    s = np.sort(v.astype(np.float32))
    r = s.size
    if r % 2:
        return s[r // 2]
    return np.float32(np.float32(s[r // 2 - 1] + s[r // 2]) * np.float32(0.5))


def settled(read: np.ndarray, t: np.float32, f: int) -> bool:
    return int(np.sum(read < t)) >= f and int(np.sum(read > -t)) >= f


@pytest.mark.parametrize("r", range(3, 17))
def test_settled_rows_bound_the_median(r):
    f = r // 2 + 1
    rng = np.random.default_rng(1000 + r)
    fills = [np.float32(3e38), np.float32(-3e38)]
    checked = 0
    for _ in range(1000):
        n = int(rng.integers(f, r + 1))
        read = (rng.standard_normal(n) * rng.choice([1e-3, 1.0, 1e3])).astype(np.float32)
        cand = np.abs(read[rng.integers(0, n, 3)])
        for t in np.concatenate([cand, np.nextafter(cand, np.float32(np.inf)), [np.float32(1.0)]]).astype(np.float32):
            if t <= 0 or not settled(read, t, f):
                continue
            for fill in fills + [t, -t, np.float32(0.0)]:
                for mix in range(3):
                    rest = np.full(r - n, fill, np.float32)
                    if mix == 1 and r - n > 0:
                        rest[::2] = -fill
                    elif mix == 2:
                        rest = rng.choice(np.array([3e38, -3e38, t, -t], np.float32), r - n)
                    m = median_fp32(np.concatenate([read, rest]))
                    assert -t < m < t, (read, rest, t, m)
                    checked += 1
    assert checked > 300


def test_even_r_mean_stays_below_the_threshold():
    """Two middle values just under t: their fp32 mean is still below t (monotone rounding of
    a sum bounded by twice an fp32 value, which is exact)."""
    for t in (np.float32(1.0), np.float32(3.0e-39), np.float32(1.7e38), np.float32(0.1)):
        below = np.nextafter(t, np.float32(0.0))
        v = np.array([below, below, -3e38, 3e38], np.float32)
        assert median_fp32(v) < t
        v = np.array([-below, -below, -3e38, 3e38], np.float32)
        assert median_fp32(v) > -t


def test_unsettled_rows_can_reach_the_threshold():
    """The rule is not loose in the other direction: with f - 1 cells below t after the first
    f rows, the unread cells decide, and the median can reach t."""
    f = 3   # r = 5
    t = np.float32(1.0)
    read = np.array([0.1, -0.2, 2.0], np.float32)
    assert not settled(read, t, f)
    assert median_fp32(np.concatenate([read, np.array([2.0, 2.0], np.float32)])) >= t


# ---- the query's integer shortcuts, checked against their definitions ----------------------

P61 = (1 << 61) - 1
M64 = (1 << 64) - 1


def _reduce61(s):
    """The query's compare-free reduction, in 64-bit wrap-around arithmetic."""
    return ((s + (((s + 1) & M64) >> 61)) & M64) & P61


def _fold61(x):
    return (x & P61) + (x >> 61)


def _affine61_nb(a, b, i):
    p0 = (a & 0xFFFFFFFF) * i
    p1 = (a >> 32) * i
    s = (p1 >> 29) + ((p1 & ((1 << 29) - 1)) << 32) + _fold61(p0) + b
    assert s < 3 << 61
    return _reduce61(_fold61(s))


def test_compare_free_modular_steps():
    """For s < 2p, (s + ((s + 1) >> 61)) & p is s mod p; the affine evaluation built on it equals
    (a i + b) mod p for a, b < p and i < 2^32, at the extremes and on random values."""
    rng = np.random.default_rng(61)
    edges = [0, 1, 2, P61 - 2, P61 - 1, 1 << 60, (1 << 60) - 1, (1 << 32) - 1, 1 << 32]
    for x in edges:
        for a in edges:
            assert _reduce61(x + a) == (x + a) % P61
    for _ in range(20000):
        x, a = int(rng.integers(0, P61)), int(rng.integers(0, P61))
        assert _reduce61(x + a) == (x + a) % P61
    for a in [1, 2, P61 - 1, P61 - 2, (1 << 32) - 1, 1 << 32, (1 << 60) + 12345]:
        for b in [0, 1, P61 - 1]:
            for i in [0, 1, (1 << 31) - 1, 1 << 31, (1 << 32) - 1]:
                assert _affine61_nb(a, b, i) == (a * i + b) % P61
    for _ in range(20000):
        a, b, i = int(rng.integers(1, P61)), int(rng.integers(0, P61)), int(rng.integers(0, 1 << 32))
        assert _affine61_nb(a, b, i) == (a * i + b) % P61


def _cell_class(T, pk):
    bits = int(np.float32(T).view(np.uint32))
    key = bits & 0x7FFFFFFF
    if key > 0x7F800000:
        return 0
    if key < pk:
        return 3
    return 2 if bits >> 31 else 1


def _tally(v, pk):
    bits = int(np.float32(v).view(np.uint32))
    key = bits & 0x7FFFFFFF
    inside, number = key < pk, key <= 0x7F800000
    return int(inside or (number and bits >> 31 == 1)), int(inside or (number and bits >> 31 == 0))


def test_class_bits_count_like_the_values():
    """A cell's two class bits, swapped by a negative sign and added into a packed pair of
    counters by one multiply, count below t and above -t exactly as the signed value does."""
    pk = int(np.float32(1.0).view(np.uint32)) & 0x7FFFFFFF
    values = [0.0, -0.0, 0.5, -0.5, 1.0, -1.0, 2.0, -2.0, np.inf, -np.inf, 1e-30, -1e-30,
              np.float32(1.0) * (1 - 2.0**-24), -np.float32(1.0) * (1 - 2.0**-24)]
    nans = [np.uint32(0x7FC00000).view(np.float32), np.uint32(0xFFC00000).view(np.float32)]
    for T in values + nans:
        for s in (0, 1):
            v = np.float32(T) if s == 0 else np.uint32(int(np.float32(T).view(np.uint32)) ^ 0x80000000).view(np.float32)
            c = _cell_class(T, pk)
            packed = ((c * (0x81 if s else 0x201)) >> (1 - s)) & 0x101
            assert (packed & 0xFF, packed >> 8) == _tally(v, pk), (T, s)
