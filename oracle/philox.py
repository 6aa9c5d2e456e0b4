"""Philox4x64-10, written from its published definition.

Reference: J. K. Salmon, M. A. Moraes, R. O. Dror, D. E. Shaw, "Parallel Random
Numbers: As Easy as 1, 2, 3", SC'11 (Sec. 3.3 and Table 2: the Philox S-box,
its multipliers and the Weyl key schedule).

Definition restated. The state is four 64-bit words (x0, x1, x2, x3) and the key
two 64-bit words (k0, k1). One round multiplies x0 and x2 by two fixed odd
constants into full 128-bit products, keeps their high and low halves, and
permutes:

    x0' = hi(M1 * x2) ^ x1 ^ k0
    x1' = lo(M1 * x2)
    x2' = hi(M0 * x0) ^ x3 ^ k1
    x3' = lo(M0 * x0)

Between consecutive rounds the key is bumped by the Weyl constants
(k0 += W0, k1 += W1, mod 2^64). Ten rounds (nine bumps) give Philox4x64-10.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__.py``). Pinned by
``tests/test_oracle_philox.py`` against the published known-answer vectors in
``tests/golden/philox4x64_10_kat.txt`` and against numpy's independent
implementation (``numpy.random.Philox``).
"""
import numpy as np

MASK64 = (1 << 64) - 1

# Round multipliers and key increments for N=4, W=64 (SC'11, Table 2).
PHILOX_M0 = 0xD2E7470EE14C6C93
PHILOX_M1 = 0xCA5A826395121157
PHILOX_W0 = 0x9E3779B97F4A7C15  # golden ratio
PHILOX_W1 = 0xBB67AE8584CAA73B  # sqrt(3) - 1
ROUNDS = 10


def philox4x64_10(counter, key):
    """One Philox4x64-10 block: 4-word counter, 2-word key -> 4 output words.

    Plain Python integers; the obviously correct form used as the definition.
    """
    x0, x1, x2, x3 = (int(c) & MASK64 for c in counter)
    k0, k1 = (int(k) & MASK64 for k in key)
    for rnd in range(ROUNDS):
        if rnd > 0:
            k0 = (k0 + PHILOX_W0) & MASK64
            k1 = (k1 + PHILOX_W1) & MASK64
        p0 = PHILOX_M0 * x0  # exact 128-bit products
        p1 = PHILOX_M1 * x2
        x0, x1, x2, x3 = (
            (p1 >> 64) ^ x1 ^ k0,
            p1 & MASK64,
            (p0 >> 64) ^ x3 ^ k1,
            p0 & MASK64,
        )
    return (x0, x1, x2, x3)


def _mulhilo64(a, b):
    """Vectorised 64x64 -> 128-bit product of uint64 arrays, split in 32-bit halves."""
    lo32 = np.uint64(0xFFFFFFFF)
    s32 = np.uint64(32)
    a_lo, a_hi = a & lo32, a >> s32
    b_lo, b_hi = b & lo32, b >> s32
    ll = a_lo * b_lo
    lh = a_lo * b_hi
    hl = a_hi * b_lo
    hh = a_hi * b_hi
    mid = (ll >> s32) + (lh & lo32) + (hl & lo32)
    hi = hh + (lh >> s32) + (hl >> s32) + (mid >> s32)
    lo = a * b  # wraps mod 2^64
    return hi, lo


def philox4x64_10_array(c0, c1, c2, c3, k0, k1):
    """Vectorised Philox4x64-10 over broadcastable uint64 arrays.

    Same rounds as ``philox4x64_10``; pinned against it on random inputs.
    Returns four uint64 arrays.
    """
    with np.errstate(over="ignore"):
        x0, x1, x2, x3 = np.broadcast_arrays(*(np.asarray(v, dtype=np.uint64) for v in (c0, c1, c2, c3)))
        x0, x1, x2, x3 = (v.copy() for v in (x0, x1, x2, x3))
        kk0 = np.uint64(int(k0) & MASK64)
        kk1 = np.uint64(int(k1) & MASK64)
        m0 = np.uint64(PHILOX_M0)
        m1 = np.uint64(PHILOX_M1)
        for rnd in range(ROUNDS):
            if rnd > 0:
                kk0 = np.uint64((int(kk0) + PHILOX_W0) & MASK64)
                kk1 = np.uint64((int(kk1) + PHILOX_W1) & MASK64)
            hi0, lo0 = _mulhilo64(m0, x0)
            hi1, lo1 = _mulhilo64(m1, x2)
            x0, x1, x2, x3 = hi1 ^ x1 ^ kk0, lo1, hi0 ^ x3 ^ kk1, lo0
    return x0, x1, x2, x3
