"""Pins of the oracle's forward masking process (Sec. 2.1; Eq. 3, 5)."""
import numpy as np
import pytest

from oracle import bgpo_oracle as O

TWO24 = 1 << 24


@pytest.mark.parametrize("T", [1, 2, 3, 1000, 2**23, 2**24 - 1, 2**24])
def test_iid_threshold_exhaustive(T):
    # over every 24-bit draw, exactly T of 2^24 values mask: P(mask) = T/2^24 = t
    u = np.arange(TWO24, dtype=np.uint64)
    assert int(O.mask_bit(u, T, TWO24).sum()) == T


@pytest.mark.parametrize("n_t,j,frac", [(16, 0, 0.0), (16, 3, 0.5), (16, 15, 1.0), (5, 2, 0.3), (3, 1, 0.99)])
def test_stratified_threshold_exhaustive(n_t, j, frac):
    # T = j 2^24 + u + 1 with u in [0, 2^24); the mask count is ceil(T / n_t)
    T = j * TWO24 + int(frac * (TWO24 - 1)) + 1
    D = n_t * TWO24
    u = np.arange(TWO24, dtype=np.uint64)
    cnt = int(O.mask_bit(u, T, D).sum())
    assert cnt == -(-T // n_t)
    # and the mask probability differs from t = T/D by less than 2^-24
    assert abs(cnt / TWO24 - T / D) < 2.0 ** -24


def test_vectorised_matches_scalar():
    for t_mode in (0, 1):
        for (B, R, j, n_t) in ((3, 37, 2, 4), (2, 1, 0, 1), (4, 64, 7, 8)):
            a = O.sample_t_mask(5, B, R, j, n_t, t_mode)
            b = O.sample_t_mask_scalar(5, B, R, j, n_t, t_mode)
            assert (a[0] == b[0]).all() and a[1] == b[1]
            assert np.array_equal(a[3], b[3])


def test_t_ranges():
    n_t = 8
    for j in range(n_t):
        T, D, t, _ = O.sample_t_mask(11, 64, 4, j, n_t, 0)
        assert D == TWO24 and (T >= 1).all() and (T <= TWO24).all()
        assert (t > 0).all() and (t <= 1).all()
        T, D, t, _ = O.sample_t_mask(11, 64, 4, j, n_t, 1)
        assert D == n_t * TWO24
        assert (t > j / n_t).all() and (t <= (j + 1) / n_t).all()


def test_t_iid_uniform_mean():
    # t_{b,j} ~ U(0,1]: the mean of 4096 draws is 1/2 within 5 sigma
    ts = np.concatenate([O.sample_t_mask(2, 512, 1, j, 8, 0)[2] for j in range(8)])
    assert abs(ts.mean() - 0.5) < 5 * np.sqrt(1 / 12 / ts.size)


def test_masked_fraction_matches_t():
    # one sequence with a very long response: each token masked with probability t
    R = 400_000
    for j in range(3):
        T, D, t, mask = O.sample_t_mask(17, 1, R, j, 3, 0)
        p = float(t[0])
        assert abs(mask.mean() - p) < 5 * np.sqrt(p * (1 - p) / R) + 1e-12


def test_masks_are_a_pure_function_of_seed_b_j():
    # resuming the n_t loop at sample j regenerates the same draws
    full = [O.sample_t_mask(3, 4, 50, j, 6, 1) for j in range(6)]
    again = O.sample_t_mask(3, 4, 50, 4, 6, 1)
    assert np.array_equal(full[4][3], again[3]) and (full[4][0] == again[0]).all()
    # and different (b, j) draw differently
    assert not np.array_equal(full[0][3], full[1][3])


def test_different_sequences_draw_independently():
    T, D, t, mask = O.sample_t_mask(8, 32, 64, 0, 1, 0)
    assert len(set(T.tolist())) == 32


def test_shard_draws_match_the_full_batch():
    # a data-parallel shard [b0, b0 + B) draws what the whole batch draws there
    for t_mode in (0, 1):
        Tf, Df, tf, mf = O.sample_t_mask(13, 12, 40, 3, 5, t_mode)
        for b0, nb in ((0, 5), (5, 7), (11, 1)):
            T, D, t, m = O.sample_t_mask(13, nb, 40, 3, 5, t_mode, b_offset=b0)
            assert D == Df and (T == Tf[b0:b0 + nb]).all()
            assert np.array_equal(m, mf[b0:b0 + nb])


def test_padding_positions_are_never_masked():
    # variable-length responses: positions at or past the length stay unmasked,
    # the draws of the real positions are those of the full-length response
    lens = np.array([37, 0, 12, 40])
    T0, D0, t0, m0 = O.sample_t_mask(21, 4, 40, 2, 4, 0)
    T, D, t, m = O.sample_t_mask(21, 4, 40, 2, 4, 0, resp_len=lens)
    assert (T == T0).all() and np.array_equal(t, t0)
    for b, n in enumerate(lens):
        assert np.array_equal(m[b, :n], m0[b, :n]) and not m[b, n:].any()


def test_brute_force_unbiased_with_padding():
    # Eq. 3-4 over the real tokens only: E_mask[l] = sum_{i < len} log p(y^i)
    import itertools
    import torch
    rng = np.random.default_rng(31)
    R, n = 9, 6
    X = rng.standard_normal((1, R, 5))
    W = rng.standard_normal((7, 5))
    Y = rng.integers(0, 7, size=(1, R))
    z = torch.from_numpy(X[0, :n]) @ torch.from_numpy(W).T
    exact = float(torch.log_softmax(z, 1).gather(1, torch.from_numpy(Y[0, :n]).long()[:, None]).sum())
    t = 0.42
    acc = 0.0
    for bits in itertools.product((0, 1), repeat=n):
        m = np.zeros((1, R), dtype=np.uint8)
        m[0, :n] = bits
        k = sum(bits)
        acc += t ** k * (1 - t) ** (n - k) * O.elbo_term(X, W, Y, 0, m, np.array([t]))[0]
    assert abs(acc - exact) < 1e-12 * abs(exact)
