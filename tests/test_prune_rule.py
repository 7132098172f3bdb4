"""The row-skipping rule of the median query, checked on the host by brute force (no GPU).

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
