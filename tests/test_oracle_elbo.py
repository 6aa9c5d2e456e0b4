"""Pins of the oracle's LM-head log-probabilities and per-step ELBO term (Eq. 4, 5)."""
import itertools
import math

import numpy as np
import torch

from oracle import bgpo_oracle as O


def _tiny(B=2, P=3, R=6, H=8, V=16, seed=0, scale=1.0):
    rng = np.random.default_rng(seed)
    X = rng.standard_normal((B, P + R, H))
    W = rng.standard_normal((V, H)) * scale
    Y = rng.integers(0, V, size=(B, R))
    return X, W, Y


def test_zero_head_gives_uniform_logp():
    X, W, Y = _tiny()
    W[:] = 0.0
    V = W.shape[0]
    logp, lse = O.token_logprobs(X[0, 3:], W, Y[0])
    assert np.allclose(logp, -math.log(V), rtol=0, atol=1e-15)
    mask = np.array([[1, 0, 1, 1, 0, 0], [0, 0, 0, 0, 0, 1]], dtype=np.uint8)
    t = np.array([0.25, 0.5])
    ell = O.elbo_term(X, W, Y, 3, mask, t)
    assert np.allclose(ell, [-(3 / 0.25) * math.log(V), -(1 / 0.5) * math.log(V)], rtol=1e-15)


def test_logp_matches_torch_log_softmax():
    X, W, Y = _tiny(B=1, P=0, R=40, H=24, V=300, seed=4, scale=3.0)
    logp, lse = O.token_logprobs(X[0], W, Y[0], chunk=37)
    z = torch.from_numpy(X[0]) @ torch.from_numpy(W).T
    ref = torch.log_softmax(z, dim=1).gather(1, torch.from_numpy(Y[0]).long()[:, None])[:, 0]
    assert np.allclose(logp, ref.numpy(), rtol=0, atol=1e-12)
    assert np.allclose(lse, torch.logsumexp(z, dim=1).numpy(), rtol=0, atol=1e-12)


def test_softmax_rows_sum_to_one():
    X, W, Y = _tiny(B=1, P=0, R=10, H=16, V=1000, seed=5, scale=4.0)
    _, lse = O.token_logprobs(X[0], W, Y[0], chunk=128)
    z = X[0] @ W.T
    assert np.allclose(np.exp(z - lse[:, None]).sum(axis=1), 1.0, rtol=0, atol=1e-12)


def test_large_logits_stay_finite():
    X, W, Y = _tiny(B=1, P=0, R=5, H=4, V=50, seed=6, scale=300.0)
    logp, lse = O.token_logprobs(X[0], W, Y[0])
    assert np.all(np.isfinite(logp)) and np.all(logp <= 0)


def test_prompt_rows_never_enter():
    X, W, Y = _tiny(P=4)
    mask = np.ones((2, 6), dtype=np.uint8)
    t = np.array([0.7, 0.3])
    ref = O.elbo_term(X, W, Y, 4, mask, t)
    X2 = X.copy()
    X2[:, :4] = np.nan
    assert np.array_equal(O.elbo_term(X2, W, Y, 4, mask, t), ref)


def test_empty_mask_gives_zero():
    X, W, Y = _tiny()
    ell = O.elbo_term(X, W, Y, 3, np.zeros((2, 6), dtype=np.uint8), np.array([0.1, 0.9]))
    assert np.array_equal(ell, np.zeros(2))


def _exact_loglik(X, W, Y, P):
    """sum_i log p(y^i | x) over all response positions, through torch (independent)."""
    B, R = Y.shape
    out = []
    for b in range(B):
        z = torch.from_numpy(X[b, P:P + R]) @ torch.from_numpy(W).T
        lp = torch.log_softmax(z, dim=1).gather(1, torch.from_numpy(Y[b]).long()[:, None])
        out.append(float(lp.sum()))
    return np.array(out)


def test_brute_force_unbiased_over_all_masks():
    # Sec. 2.1 / Eq. 3-4: with every token masked independently with prob. t,
    # E_mask[l] = sum_i log p(y^i) exactly, for every t (hidden states fixed).
    R = 10
    X, W, Y = _tiny(B=2, P=2, R=R, H=8, V=16, seed=9, scale=1.5)
    exact = _exact_loglik(X, W, Y, 2)
    for t in (0.05, 0.37, 0.5, 0.93, 1.0):
        acc = np.zeros(2)
        for bits in itertools.product((0, 1), repeat=R):
            m = np.array(bits, dtype=np.uint8)
            k = int(m.sum())
            weight = t ** k * (1 - t) ** (R - k)
            if weight == 0.0:
                continue
            acc += weight * O.elbo_term(X, W, Y, 2, np.stack([m, m]), np.array([t, t]))
        assert np.allclose(acc, exact, rtol=1e-12, atol=0)


def test_brute_force_unbiased_with_drawn_t():
    # same identity with t = T / 2^24 produced by the masking process itself
    R = 8
    X, W, Y = _tiny(B=3, P=1, R=R, H=6, V=12, seed=10)
    exact = _exact_loglik(X, W, Y, 1)
    T, D, t, _ = O.sample_t_mask(21, 3, R, 0, 1, 0)
    acc = np.zeros(3)
    for bits in itertools.product((0, 1), repeat=R):
        m = np.array(bits, dtype=np.uint8)
        k = int(m.sum())
        w = t ** k * (1 - t) ** (R - k)
        acc += w * O.elbo_term(X, W, Y, 1, np.stack([m] * 3), t)
    assert np.allclose(acc, exact, rtol=1e-12)


def test_mc_elbo_estimate_converges():
    # Eq. 5 with many MC samples approaches sum_i log p (statistical, loose)
    X, W, Y = _tiny(B=1, P=0, R=24, H=8, V=10, seed=11)
    exact = _exact_loglik(X, W, Y, 0)[0]
    n_t = 3000
    ts, masks = O.sample_masks(5, 1, 24, n_t, 1)   # stratified t lowers the variance
    ell = O.elbo_all(X, W, Y, 0, ts, masks)[0]
    se = ell.std() / math.sqrt(n_t)
    assert abs(ell.mean() - exact) < 6 * se + 1e-9


def test_logp_from_precomputed_logit_chunks():
    X, W, Y = _tiny(B=1, P=0, R=30, H=12, V=100, seed=9, scale=2.0)
    zs = O.logit_chunks(X[0], W, chunk=33)
    assert [z.shape[1] for z in zs] == [33, 33, 33, 1]
    a = O.token_logprobs(X[0], W, Y[0], chunk=33)
    b = O.token_logprobs(X[0], W, Y[0], chunk=33, z_chunks=zs)
    assert np.allclose(a[0], b[0], rtol=0, atol=1e-13) and np.allclose(a[1], b[1], rtol=0, atol=1e-13)
