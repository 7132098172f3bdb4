"""Count Sketch hash family for the oracle (test infrastructure only).

The paper compresses each worker's gradient into a Count Sketch S(g) (Sec. III-A, citing
Charikar et al.) but does not print the hash family.  The family used throughout is the
classic Carter-Wegman construction over the Mersenne prime p = 2^61 - 1:

    bucket  h_j(i) = ((a_j * i + b_j) mod p) mod c
    sign    s_j(i) = +1 if ((a'_j * i + b'_j) mod p) is even, else -1

for rows j = 0..r-1, with coefficients drawn from a seed by splitmix64 (Steele, Lea and
Flood, "Fast splittable pseudorandom number generators", OOPSLA 2014), four draws per row
in the order a_j, b_j, a'_j, b'_j:

    a = 1 + (x mod (p - 1)),   b = x mod p.

``bucket_exact`` / ``sign_exact`` evaluate the definition with Python integers and are the
ground truth.  ``hash_rows`` evaluates the same definition vectorised in numpy uint64 by
splitting the multiplier into 31-bit limbs so that no product overflows 64 bits.
"""

from __future__ import annotations

import numpy as np

MERSENNE_P = (1 << 61) - 1
_MASK64 = (1 << 64) - 1


def splitmix64(seed: int):
    """Yield the splitmix64 output stream for ``seed`` (published definition, 2014).

    state += 0x9E3779B97F4A7C15; z = state;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EB;
    output z ^ (z >> 31)       (all arithmetic mod 2^64)
    """
    state = seed & _MASK64
    while True:
        state = (state + 0x9E3779B97F4A7C15) & _MASK64
        z = state
        z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & _MASK64
        z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & _MASK64
        yield z ^ (z >> 31)


def splitmix64_at(seed: int, idx) -> np.ndarray:
    """The outputs number idx (0-based) of the splitmix64 stream seeded with ``seed``, as
    uint64: the state after idx + 1 golden-ratio increments, mixed (counter-based form of the
    same published generator)."""
    with np.errstate(over="ignore"):
        i = np.asarray(idx, dtype=np.uint64)
        z = np.uint64(seed & _MASK64) + (i + np.uint64(1)) * np.uint64(0x9E3779B97F4A7C15)
        z = (z ^ (z >> np.uint64(30))) * np.uint64(0xBF58476D1CE4E5B9)
        z = (z ^ (z >> np.uint64(27))) * np.uint64(0x94D049BB133111EB)
        return z ^ (z >> np.uint64(31))


def derive_coefficients(r: int, seed: int):
    """Coefficients (a, b, a2, b2), each a list of r Python ints, for rows 0..r-1.

    a, a2 lie in [1, p-1] (non-zero multipliers); b, b2 lie in [0, p-1].
    """
    gen = splitmix64(seed)
    a, b, a2, b2 = [], [], [], []
    for _ in range(r):
        a.append(1 + next(gen) % (MERSENNE_P - 1))
        b.append(next(gen) % MERSENNE_P)
        a2.append(1 + next(gen) % (MERSENNE_P - 1))
        b2.append(next(gen) % MERSENNE_P)
    return a, b, a2, b2


def bucket_exact(a: int, b: int, c: int, i: int) -> int:
    """h(i) = ((a*i + b) mod p) mod c with exact integers."""
    return ((a * i + b) % MERSENNE_P) % c


def sign_exact(a2: int, b2: int, i: int) -> int:
    """s(i) = +1 when ((a2*i + b2) mod p) is even, -1 when odd, exact integers."""
    return 1 if ((a2 * i + b2) % MERSENNE_P) % 2 == 0 else -1


# ---- numpy evaluation ------------------------------------------------------------------

_P = np.uint64(MERSENNE_P)
_SH61 = np.uint64(61)


def _reduce_once(x: np.ndarray) -> np.ndarray:
    """Map x in [0, 2p) to x mod p."""
    return np.where(x >= _P, x - _P, x)


def _fold(x: np.ndarray) -> np.ndarray:
    """x mod p for x < 2^63, using 2^61 = 1 (mod p)."""
    return _reduce_once((x & _P) + (x >> _SH61))


def _affine_mod_p(a: int, b: int, i: np.ndarray) -> np.ndarray:
    """(a*i + b) mod p for uint64 i < 2^31, a < 2^61, b < 2^61.

    a = a_hi * 2^31 + a_lo with a_hi < 2^30, a_lo < 2^31, so
    a*i = (a_hi*i) * 2^31 + a_lo*i where both partial products stay below 2^62.
    (t * 2^31) mod p is taken as t = t_hi*2^30 + t_lo  ->  t_hi + t_lo*2^31 (mod p).
    """
    a_hi = np.uint64(a >> 31)
    a_lo = np.uint64(a & ((1 << 31) - 1))
    t1 = a_hi * i                      # < 2^61
    t1_hi = t1 >> np.uint64(30)        # < 2^31
    t1_lo = t1 & np.uint64((1 << 30) - 1)
    m1 = _fold(t1_hi + (t1_lo << np.uint64(31)))
    m2 = _fold(a_lo * i)               # a_lo*i < 2^62
    s = _fold(m1 + m2)
    return _reduce_once(s + np.uint64(b))


def hash_rows(coeffs, c: int, idx) -> tuple[np.ndarray, np.ndarray]:
    """Buckets [r, n] (int64) and signs [r, n] (int8) for coordinates ``idx``.

    ``idx`` holds coordinates in [0, 2^31); ``coeffs`` is (a, b, a2, b2) as returned by
    ``derive_coefficients`` (or any lists of valid coefficients).
    """
    a, b, a2, b2 = coeffs
    i = np.asarray(idx, dtype=np.uint64)
    if i.size and int(i.max()) >= (1 << 31):
        raise ValueError("coordinates must be below 2^31")
    r = len(a)
    buckets = np.empty((r, i.size), dtype=np.int64)
    signs = np.empty((r, i.size), dtype=np.int8)
    for j in range(r):
        x = _affine_mod_p(a[j], b[j], i)
        buckets[j] = (x % np.uint64(c)).astype(np.int64)
        y = _affine_mod_p(a2[j], b2[j], i)
        signs[j] = (1 - 2 * (y & np.uint64(1)).astype(np.int64)).astype(np.int8)
    return buckets, signs
