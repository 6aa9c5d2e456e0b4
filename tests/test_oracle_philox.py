"""Pins of the oracle's Philox4x64-10 (SC'11) against published vectors and numpy."""
import os

import numpy as np
import pytest

from oracle.philox import philox4x64_10, philox4x64_10_array

MASK64 = (1 << 64) - 1


def _kat_rows(golden_dir):
    rows = []
    with open(os.path.join(golden_dir, "philox4x64_10_kat.txt")) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            vals = [int(x, 16) for x in line.split()]
            assert len(vals) == 10
            rows.append((vals[0:4], vals[4:6], vals[6:10]))
    assert rows
    return rows


def test_published_known_answers(golden_dir):
    for ctr, key, expect in _kat_rows(golden_dir):
        assert list(philox4x64_10(ctr, key)) == expect


def _numpy_block(ctr, key):
    """numpy's Philox advances its 256-bit counter before producing a block."""
    v = sum(int(c) << (64 * k) for k, c in enumerate(ctr))
    v = (v - 1) % (1 << 256)
    pre = [(v >> (64 * k)) & MASK64 for k in range(4)]
    bg = np.random.Philox(key=np.array([int(key[0]), int(key[1])], dtype=np.uint64),
                          counter=np.array(pre, dtype=np.uint64))
    return [int(x) for x in bg.random_raw(4)]


def test_matches_numpy_philox_random_inputs():
    rng = np.random.default_rng(123)
    for _ in range(200):
        ctr = [int(x) for x in rng.integers(0, MASK64, size=4, dtype=np.uint64, endpoint=True)]
        key = [int(x) for x in rng.integers(0, MASK64, size=2, dtype=np.uint64, endpoint=True)]
        assert list(philox4x64_10(ctr, key)) == _numpy_block(ctr, key)


def test_matches_numpy_philox_layout_counters():
    # the counters the masking process uses: (q, b, j, stream) with small words
    for seed in (0, 1, 3, 2**40 + 17):
        for ctr in ((0, 0, 0, 1), (5, 3, 7, 0), (255, 31, 15, 0), (0, 1023, 31, 1)):
            assert list(philox4x64_10(ctr, (seed, 0))) == _numpy_block(ctr, (seed, 0))


def test_array_form_matches_scalar_form():
    rng = np.random.default_rng(7)
    c0 = rng.integers(0, MASK64, size=64, dtype=np.uint64, endpoint=True)
    c1 = rng.integers(0, 2**40, size=64, dtype=np.int64).astype(np.uint64)
    for key in ((0, 0), (MASK64, 12345), (2**63 + 5, 2**62 + 1)):
        out = philox4x64_10_array(c0, c1, np.uint64(9), np.uint64(1), key[0], key[1])
        for n in range(64):
            ref = philox4x64_10((int(c0[n]), int(c1[n]), 9, 1), key)
            assert [int(o[n]) for o in out] == list(ref)


@pytest.mark.parametrize("word", [0, 1, 2, 3])
def test_output_words_roughly_uniform(word):
    # each 24-bit draw should be uniform: mean of u24/2^24 over 20k blocks ~ 0.5
    q = np.arange(20000, dtype=np.uint64)
    out = philox4x64_10_array(q, np.uint64(3), np.uint64(4), np.uint64(0), 99, 0)
    u = (out[word] >> np.uint64(40)).astype(np.float64) / 2**24
    assert abs(u.mean() - 0.5) < 5 * np.sqrt(1 / 12 / u.size)
