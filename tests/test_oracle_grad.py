"""Pins of the oracle's analytic gradients (Algorithm 1 backward, Sec. 3.2 Equivalence)."""
import numpy as np
import torch

from oracle import bgpo_oracle as O


def _case(seed=0, B=3, P=2, R=9, H=6, V=23, n_t=3, t_mode=0, off_policy=True):
    rng = np.random.default_rng(seed)
    X = rng.standard_normal((B, P + R, H))
    W = rng.standard_normal((V, H)) * 0.7
    Y = rng.integers(0, V, size=(B, R))
    A = rng.standard_normal(B)
    A[0] = abs(A[0])            # both branches present
    A[1] = -abs(A[1])
    ts, masks = O.sample_masks(seed + 100, B, R, n_t, t_mode)
    ell_self = O.elbo_all(X, W, Y, P, ts, masks)
    eps = rng.standard_normal((B, n_t)) * 0.3 if off_policy else np.zeros((B, n_t))
    ell_old = ell_self + eps
    return X, W, Y, P, A, ell_old, ts, masks


def _fd_check(loss_fn, X, W, dX, dW, P, n=25, h=1e-6, seed=0):
    rng = np.random.default_rng(seed)
    V, H = W.shape
    B, R = dX.shape[:2]
    for _ in range(n):
        v, k = rng.integers(V), rng.integers(H)
        Wp, Wm = W.copy(), W.copy()
        Wp[v, k] += h
        Wm[v, k] -= h
        fd = (loss_fn(X, Wp) - loss_fn(X, Wm)) / (2 * h)
        assert abs(fd - dW[v, k]) <= 1e-6 * max(1.0, abs(fd)), (v, k, fd, dW[v, k])
    for _ in range(n):
        b, i, k = rng.integers(B), rng.integers(R), rng.integers(H)
        Xp, Xm = X.copy(), X.copy()
        Xp[b, P + i, k] += h
        Xm[b, P + i, k] -= h
        fd = (loss_fn(Xp, W) - loss_fn(Xm, W)) / (2 * h)
        assert abs(fd - dX[b, i, k]) <= 1e-6 * max(1.0, abs(fd)), (b, i, k, fd, dX[b, i, k])


def test_gradients_match_finite_differences_off_policy():
    X, W, Y, P, A, ell_old, ts, masks = _case(seed=1)
    ls = 0.5
    out = O.bgpo_step(X, W, Y, P, A, ell_old, ts, masks, ls)
    f = lambda X_, W_: O.bgpo_loss(X_, W_, Y, P, A, ell_old, ts, masks, ls)
    _fd_check(f, X, W, out["dX"], out["dW"], P, seed=1)


def test_gradients_match_finite_differences_stratified():
    X, W, Y, P, A, ell_old, ts, masks = _case(seed=2, n_t=4, t_mode=1)
    out = O.bgpo_step(X, W, Y, P, A, ell_old, ts, masks, 1.0)
    f = lambda X_, W_: O.bgpo_loss(X_, W_, Y, P, A, ell_old, ts, masks, 1.0)
    _fd_check(f, X, W, out["dX"], out["dW"], P, seed=2)


def test_gradients_match_torch_autograd():
    # an independent statement of the same loss, differentiated by torch autograd
    X, W, Y, P, A, ell_old, ts, masks = _case(seed=3, B=4, R=12, H=10, V=40, n_t=5)
    ls = 0.25
    out = O.bgpo_step(X, W, Y, P, A, ell_old, ts, masks, ls)
    Xt = torch.tensor(X, requires_grad=True)
    Wt = torch.tensor(W, requires_grad=True)
    n_t = len(ts)
    total = torch.zeros((), dtype=torch.float64)
    for j in range(n_t):
        for b in range(X.shape[0]):
            m = torch.from_numpy(masks[j, b].astype(bool))
            resp = Xt[b, P:]
            lp = torch.log_softmax(resp @ Wt.T, dim=1).gather(1, torch.from_numpy(Y[b]).long()[:, None])[:, 0]
            ell = (lp * m).sum() / float(ts[j, b])
            d = ell - float(ell_old[b, j])
            g = (1 + d) * A[b] / n_t if A[b] >= 0 else torch.exp(d) * A[b] / n_t
            total = total - ls * g
    total.backward()
    assert abs(float(total.detach()) - out["loss"]) < 1e-10 * max(1, abs(out["loss"]))
    assert np.allclose(Wt.grad.numpy(), out["dW"], rtol=1e-10, atol=1e-12)
    assert np.allclose(Xt.grad[:, P:].numpy(), out["dX"], rtol=1e-10, atol=1e-12)
    assert np.array_equal(Xt.grad[:, :P].numpy(), np.zeros_like(Xt.grad[:, :P].numpy()))


def test_equivalence_gradient_on_policy():
    # Sec. 3.2: on-policy, grad R_lb = grad R_hat; R_hat (Eq. 7) differentiated numerically
    X, W, Y, P, A, ell_old, ts, masks = _case(seed=4, off_policy=False)
    out = O.bgpo_step(X, W, Y, P, A, ell_old, ts, masks, 1.0)
    assert np.allclose(out["d"], 0.0, atol=0)
    assert np.allclose(out["R_lb"], A, rtol=1e-13)
    f = lambda X_, W_: O.vrpo_loss(X_, W_, Y, P, A, ell_old, ts, masks, 1.0)
    _fd_check(f, X, W, out["dX"], out["dW"], P, seed=4)


def test_dw_rows_sum_to_zero():
    # each dz_r = w_r (onehot - softmax) sums to zero over the vocabulary
    X, W, Y, P, A, ell_old, ts, masks = _case(seed=5, V=57)
    out = O.bgpo_step(X, W, Y, P, A, ell_old, ts, masks, 1.0)
    scale = np.abs(out["dW"]).max()
    assert np.abs(out["dW"].sum(axis=0)).max() < 1e-12 * max(1.0, scale)


def test_linearity_accumulation_equals_one_shot():
    # Linearity (Sec. 3): summing per-sample gradients = gradient of sum_j L_j;
    # here the per-sample pieces are accumulated in reverse order and in halves
    X, W, Y, P, A, ell_old, ts, masks = _case(seed=6, n_t=6)
    out = O.bgpo_step(X, W, Y, P, A, ell_old, ts, masks, 1.0)
    coef = out["coef"]
    dW = np.zeros_like(W)
    dX = np.zeros_like(out["dX"])
    for j in reversed(range(6)):
        gx, gw = O.elbo_term_grads(X, W, Y, P, masks[j], ts[j], coef[:, j], chunk=5)
        dX += gx
        dW += gw
    assert np.allclose(dW, out["dW"], rtol=1e-12, atol=1e-14)
    assert np.allclose(dX, out["dX"], rtol=1e-12, atol=1e-14)


def test_vrpo_coefficients_give_the_eq7_gradient_off_policy():
    # the gradient of Eq. 7 assembled from per-sample coefficients, checked by
    # central differences of the VRPO loss itself
    X, W, Y, P, A, ell_old, ts, masks = _case(seed=7, n_t=4)
    ell = O.elbo_all(X, W, Y, P, ts, masks)
    R, coef = O.vrpo_coeffs(ell, ell_old, A, 0.5)
    assert np.allclose(R, O.vrpo_ratio(ell, ell_old, A), rtol=1e-14)
    dX = np.zeros((X.shape[0], masks.shape[2], X.shape[2]))
    dW = np.zeros_like(W)
    for j in range(len(ts)):
        gx, gw = O.elbo_term_grads(X, W, Y, P, masks[j], ts[j], coef)
        dX += gx
        dW += gw
    f = lambda X_, W_: O.vrpo_loss(X_, W_, Y, P, A, ell_old, ts, masks, 0.5)
    _fd_check(f, X, W, dX, dW, P, seed=7)


def test_vrpo_and_bgpo_coefficients_agree_on_policy():
    # Sec. 3.2: with d = 0 both objectives weight every sample by -loss_scale A / n_t
    rng = np.random.default_rng(8)
    ell = rng.standard_normal((9, 5)) * 40
    A = rng.standard_normal(9)
    _, cv = O.vrpo_coeffs(ell, ell, A, 0.25)
    _, _, cb = O.bound_coeffs(ell, ell, A[:, None], 5, 0.25)
    assert np.allclose(cb, cv[:, None], rtol=1e-15, atol=0)


def test_grad_std_bias_definitions():
    # closed forms: constant repeats have zero std; a known offset is the bias
    g = np.stack([np.full((3, 4), 2.0)] * 5)
    assert O.grad_std_bias(g, np.full((3, 4), 1.5)) == (0.0, 0.5)
    # two repeats +-1 around the golden value: std 1, bias 0
    g = np.stack([np.ones((2, 2)), -np.ones((2, 2))])
    assert O.grad_std_bias(g, np.zeros((2, 2))) == (1.0, 0.0)


def test_mc_gradient_std_shrinks_with_n_t():
    # Sec. 4.3: more MC samples, smaller spread of the gradient estimate
    X, W, Y, P, A, _, _, _ = _case(seed=9, B=2, R=10, H=5, V=11, n_t=1)
    stds = []
    for n_t in (1, 4, 16):
        grads = []
        for rep in range(12):
            ts, masks = O.sample_masks(1000 + 97 * rep, 2, 10, n_t, 0)
            ell = O.elbo_all(X, W, Y, P, ts, masks)
            grads.append(O.bgpo_step(X, W, Y, P, A, ell, ts, masks, 1.0)["dW"])
        stds.append(O.grad_std_bias(np.stack(grads), np.zeros_like(W))[0])
    assert stds[0] > stds[1] > stds[2]


def test_gradient_pass_returns_the_elbo_of_the_same_log_probabilities():
    # with_ell: l of Eq. 4 from the gradient pass itself; closed form at W = 0
    # (every log p = -log V) and equal to elbo_term otherwise
    X, W, Y, P, A, ell_old, ts, masks = _case(seed=10, n_t=2)
    coef = np.linspace(-1.0, 1.0, X.shape[0])
    ell, gx, gw = O.elbo_term_grads(X, W, Y, P, masks[1], ts[1], coef, chunk=7, with_ell=True)
    assert np.allclose(ell, O.elbo_term(X, W, Y, P, masks[1], ts[1]), rtol=1e-14, atol=0)
    gx2, gw2 = O.elbo_term_grads(X, W, Y, P, masks[1], ts[1], coef, chunk=7)
    assert np.array_equal(gx, gx2) and np.array_equal(gw, gw2)
    Z = np.zeros_like(W)
    ell0, _, _ = O.elbo_term_grads(X, Z, Y, P, masks[0], ts[0], coef, with_ell=True)
    V = W.shape[0]
    k = masks[0].sum(axis=1).astype(np.float64)
    assert np.allclose(ell0, -k / ts[0] * np.log(V), rtol=1e-14, atol=0)


def _per_sample_case(seed, n_t=3, **kw):
    X, W, Y, P, A, _, ts, masks = _case(seed=seed, n_t=n_t, **kw)
    rng = np.random.default_rng(seed + 50)
    # each MC sample sees its own hidden states (Sec. 2.1: p_theta conditions on y_t)
    Xs = np.stack([X + 0.5 * rng.standard_normal(X.shape) for _ in range(n_t)])
    ell_self = np.stack([O.elbo_term(Xs[j], W, Y, P, masks[j], ts[j]) for j in range(n_t)], axis=1)
    ell_old = ell_self + rng.standard_normal(ell_self.shape) * 0.3
    return Xs, W, Y, P, A, ell_old, ts, masks


def test_per_sample_hidden_states_match_finite_differences():
    Xs, W, Y, P, A, ell_old, ts, masks = _per_sample_case(seed=11)
    ls = 0.5
    out = O.bgpo_step_per_sample_x(Xs, W, Y, P, A, ell_old, ts, masks, ls)
    rng = np.random.default_rng(11)
    h = 1e-6
    f = lambda Xs_, W_: O.bgpo_loss_per_sample_x(Xs_, W_, Y, P, A, ell_old, ts, masks, ls)
    n_t, B, R, H = out["dX"].shape
    for _ in range(25):
        j, b, i, k = rng.integers(n_t), rng.integers(B), rng.integers(R), rng.integers(H)
        Xp, Xm = Xs.copy(), Xs.copy()
        Xp[j, b, P + i, k] += h
        Xm[j, b, P + i, k] -= h
        fd = (f(Xp, W) - f(Xm, W)) / (2 * h)
        assert abs(fd - out["dX"][j, b, i, k]) <= 1e-6 * max(1.0, abs(fd)), (j, b, i, k)
    V = W.shape[0]
    for _ in range(25):
        v, k = rng.integers(V), rng.integers(H)
        Wp, Wm = W.copy(), W.copy()
        Wp[v, k] += h
        Wm[v, k] -= h
        fd = (f(Xs, Wp) - f(Xs, Wm)) / (2 * h)
        assert abs(fd - out["dW"][v, k]) <= 1e-6 * max(1.0, abs(fd)), (v, k)


def test_per_sample_hidden_states_match_torch_autograd():
    # the loss restated with torch ops on a leaf tensor per MC sample's hidden states
    Xs, W, Y, P, A, ell_old, ts, masks = _per_sample_case(seed=12, n_t=4, B=3, R=10, H=7, V=29)
    ls = 0.25
    out = O.bgpo_step_per_sample_x(Xs, W, Y, P, A, ell_old, ts, masks, ls)
    Xt = torch.tensor(Xs, requires_grad=True)
    Wt = torch.tensor(W, requires_grad=True)
    n_t = len(ts)
    total = torch.zeros((), dtype=torch.float64)
    for j in range(n_t):
        for b in range(Xs.shape[1]):
            m = torch.from_numpy(masks[j, b].astype(bool))
            z = Xt[j, b, P:] @ Wt.T
            lp = torch.log_softmax(z, dim=1).gather(1, torch.from_numpy(Y[b]).long()[:, None])[:, 0]
            ell = (lp * m).sum() / float(ts[j, b])
            d = ell - float(ell_old[b, j])
            g = (1 + d) * A[b] / n_t if A[b] >= 0 else torch.exp(d) * A[b] / n_t
            total = total - ls * g
    total.backward()
    assert abs(float(total.detach()) - out["loss"]) < 1e-10 * max(1, abs(out["loss"]))
    assert np.allclose(Wt.grad.numpy(), out["dW"], rtol=1e-10, atol=1e-12)
    assert np.allclose(Xt.grad[:, :, P:].numpy(), out["dX"], rtol=1e-10, atol=1e-12)
    assert not np.any(Xt.grad[:, :, :P].numpy())


def test_shared_hidden_states_reduce_to_the_accumulated_step():
    # the same X for every sample: per-sample dX_j sum to bgpo_step's accumulated dX
    X, W, Y, P, A, ell_old, ts, masks = _case(seed=13, n_t=3)
    Xs = np.stack([X] * 3)
    a = O.bgpo_step_per_sample_x(Xs, W, Y, P, A, ell_old, ts, masks, 0.5)
    b = O.bgpo_step(X, W, Y, P, A, ell_old, ts, masks, 0.5)
    assert np.allclose(a["dX"].sum(axis=0), b["dX"], rtol=1e-12, atol=1e-14)
    assert np.allclose(a["dW"], b["dW"], rtol=1e-12, atol=1e-14)
    assert np.array_equal(a["ell"], b["ell"])


def test_kept_and_recomputed_logit_chunks_agree(monkeypatch):
    # the gradient pass keeps each sequence's logit chunks between its passes
    # when they are small; forcing the recompute path changes nothing
    X, W, Y, P, A, ell_old, ts, masks = _case(seed=14, n_t=2, V=41)
    coef = np.array([0.7, -1.3, 0.2])
    kept = O.elbo_term_grads(X, W, Y, P, masks[1], ts[1], coef, chunk=6, with_ell=True)
    monkeypatch.setattr(O, "Z_KEEP_ELEMS", 0)
    again = O.elbo_term_grads(X, W, Y, P, masks[1], ts[1], coef, chunk=6, with_ell=True)
    for a, b in zip(kept, again):
        assert np.allclose(a, b, rtol=1e-14, atol=1e-15)


def test_brute_force_gradient_unbiased_over_all_masks():
    # Sec. 2.1 / Eq. 3-4, differentiated: with every response token masked
    # independently with probability t, the mask-weighted mean of the one-sample
    # gradient of l (its 1/t weight included) is the gradient of
    # sum_i log p(y^i | x) over all response positions, for every t. The right
    # side is torch autograd on log_softmax, independent of the oracle.
    import itertools
    rng = np.random.default_rng(31)
    B, P, R, H, V = 2, 2, 8, 6, 12
    X = rng.standard_normal((B, P + R, H)) * 1.3
    W = rng.standard_normal((V, H)) * 0.8
    Y = rng.integers(0, V, size=(B, R))
    Xt = torch.from_numpy(X.copy()).requires_grad_(True)
    Wt = torch.from_numpy(W.copy()).requires_grad_(True)
    total = 0
    for b in range(B):
        z = Xt[b, P:] @ Wt.T
        total = total + torch.log_softmax(z, dim=1).gather(1, torch.from_numpy(Y[b])[:, None]).sum()
    total.backward()
    gX = Xt.grad.numpy()[:, P:]
    gW = Wt.grad.numpy()
    coef = np.ones(B)
    for t in (0.2, 0.55, 1.0):
        aX = np.zeros((B, R, H))
        aW = np.zeros((V, H))
        for bits in itertools.product((0, 1), repeat=R):
            m = np.array(bits, dtype=np.uint8)
            k = int(m.sum())
            weight = t ** k * (1 - t) ** (R - k)
            if weight == 0.0:
                continue
            dX, dW = O.elbo_term_grads(X, W, Y, P, np.stack([m] * B), np.full(B, t), coef)
            aX += weight * dX
            aW += weight * dW
        assert np.allclose(aX, gX, rtol=1e-10, atol=1e-12)
        assert np.allclose(aW, gW, rtol=1e-10, atol=1e-12)
