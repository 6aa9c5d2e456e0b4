"""fp64 oracle for the BGPO per-MC-sample ELBO term, its bound and its gradient.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__.py``): plain numpy in float64,
written from the paper (arxiv 2510.11683) and checked against it by
``tests/test_oracle_*.py``. bf16 inputs arrive as float64 arrays (exact widening).

Notation (paper's): a batch of B responses y, each with prompt length P and
response length R; hidden states X[b, P+i, :] of size H feed the LM head W [V, H];
targets Y[b, i] = y^i. For MC sample j the timestep is t_{b,j} and the mask
m_{b,i} = 1[y_t^i = M].

Readings of the paper used here (each also listed in the design notes):
  * t endpoints. Sec. 2.1 says t in (0,1), Eq. 3/5 say U[0,1]. Reading: t in (0, 1],
    t = T/D with integer T >= 1, so 1/t in Eq. 4 is always finite.
  * Random draws. The paper only says "sample". Reading: Philox4x64-10 with key
    (seed, 0) and counter (c0, b, j, stream); stream 0 draws the mask (word k of
    block c0 = q covers response position i = 4q + k), stream 1 draws t (word 0
    of block c0 = 0); a uniform 24-bit integer is u24 = word >> 40.
  * t_mode 0 (i.i.d., Eq. 5): T = u24 + 1, D = 2^24.
    t_mode 1 (stratified, an addition used by one workload; not in the paper):
    T = j 2^24 + u24 + 1, D = n_t 2^24, so t lies in (j/n_t, (j+1)/n_t].
  * Mask (Sec. 2.1: each response token masked independently with probability t,
    the prompt never): m = [u24 * D < T * 2^24], exact integers, so
    P(m = 1) = ceil(T 2^24 / D) / 2^24 (= t exactly when D = 2^24).
  * Eq. 4 has no length normalisation; an empty mask gives l = 0.
  * Eq. 13 branch at A = 0: the Taylor branch ("A >= 0").
  * Loss scaling: Algorithm 1 sets L_j = -g_j / G; Eq. 19 averages over prompts.
    Reading: per-sample loss L_{b,j} = -loss_scale * g_{b,j}, loss_scale = 1/G by
    default, summed over the batch (Algorithm 1).
  * Eq. 18 std: population std (ddof = 0); a group with zero std gets A = 0.
"""
import numpy as np

from .philox import philox4x64_10, philox4x64_10_array

U24_SHIFT = 40          # u24 = top 24 bits of a Philox output word
TWO24 = 1 << 24
STREAM_MASK = 0         # counter word c3 for mask draws
STREAM_T = 1            # counter word c3 for the timestep draw
T_MODE_IID = 0
T_MODE_STRATIFIED = 1


# ---------------------------------------------------------------------------
# Forward masking process q(. | t, y, x)  (Sec. 2.1; Eq. 3, 5; Algorithm 1)
# ---------------------------------------------------------------------------

def t_numerator(seed, b, j, n_t, t_mode):
    """Exact timestep t_{b,j} = T / D for sequence b, MC sample j (Eq. 5 draw)."""
    word = philox4x64_10((0, b, j, STREAM_T), (seed, 0))[0]
    u24 = word >> U24_SHIFT
    if t_mode == T_MODE_IID:
        return u24 + 1, TWO24
    if t_mode == T_MODE_STRATIFIED:
        return j * TWO24 + u24 + 1, n_t * TWO24
    raise ValueError("t_mode must be 0 (iid) or 1 (stratified)")


def mask_bit(u24, T, D):
    """1 when a response token is replaced by the mask token: u24 / 2^24 < T / D.

    Exact integers: u24 * D < T * 2^24. Works on Python ints or uint64 arrays
    (both products stay below 2^64 for n_t < 2^16).
    """
    if isinstance(u24, np.ndarray):
        lhs = u24.astype(np.uint64) * np.uint64(D)
        rhs = np.asarray(T, dtype=np.uint64) * np.uint64(TWO24)
        return (lhs < rhs).astype(np.uint8)
    return int(int(u24) * int(D) < int(T) * TWO24)


def sample_t_mask(seed, B, R, j, n_t, t_mode, b_offset=0, resp_len=None):
    """Timesteps and response masks of MC sample j for B sequences.

    Sequence b of this batch has global index b_offset + b in the counters, so a
    shard of a larger batch draws what the whole batch draws for those rows.
    resp_len [B] (optional): response b holds resp_len[b] <= R tokens; positions
    i >= resp_len[b] are padding and never masked (the draws are unchanged).
    Returns (T [B] int64, D int, t [B] float64, mask [B, R] uint8). Prompt
    positions are never masked (Sec. 2.1), so only the R response positions
    appear here.
    """
    T = np.zeros(B, dtype=np.int64)
    D = None
    for b in range(B):
        T[b], D = t_numerator(seed, b_offset + b, j, n_t, t_mode)
    Q = (R + 3) // 4
    q = np.arange(Q, dtype=np.uint64)[None, :]
    bb = (np.arange(B, dtype=np.uint64) + np.uint64(b_offset))[:, None]
    words = philox4x64_10_array(q, bb, np.uint64(j), np.uint64(STREAM_MASK), seed, 0)
    u = np.stack(words, axis=-1).reshape(B, Q * 4)[:, :R] >> np.uint64(U24_SHIFT)
    mask = mask_bit(u, T.astype(np.uint64)[:, None], D)
    if resp_len is not None:
        mask = mask * (np.arange(R)[None, :] < np.asarray(resp_len)[:, None]).astype(np.uint8)
    t = T.astype(np.float64) / float(D)
    return T, D, t, mask


def sample_t_mask_scalar(seed, B, R, j, n_t, t_mode):
    """Same as ``sample_t_mask`` with one scalar Philox call per block (small cases)."""
    T = np.zeros(B, dtype=np.int64)
    mask = np.zeros((B, R), dtype=np.uint8)
    D = None
    for b in range(B):
        T[b], D = t_numerator(seed, b, j, n_t, t_mode)
        for q in range((R + 3) // 4):
            words = philox4x64_10((q, b, j, STREAM_MASK), (seed, 0))
            for k in range(4):
                i = 4 * q + k
                if i < R:
                    mask[b, i] = mask_bit(words[k] >> U24_SHIFT, int(T[b]), D)
    return T, D, T.astype(np.float64) / float(D), mask


# ---------------------------------------------------------------------------
# LM head: log p_theta(y^i | y_t, x) = log_softmax(W x)[y^i]   (Eq. 4)
# ---------------------------------------------------------------------------

# Logit chunks of one sequence are kept between passes when they hold at most
# this many elements (2 GiB of fp64); larger ones are recomputed per pass.
Z_KEEP_ELEMS = 1 << 28


def logit_chunks(rows, W, chunk=8192):
    """z = W x_r for each row, as a list of [n, chunk] fp64 column blocks."""
    rows = np.asarray(rows, dtype=np.float64)
    W = np.asarray(W, dtype=np.float64)
    return [rows @ W[v0:v0 + chunk].T for v0 in range(0, W.shape[0], chunk)]


def token_logprobs(rows, W, y, chunk=8192, z_chunks=None):
    """log softmax(W x_r)[y_r] for each row x_r, in fp64, over vocab chunks.

    rows [n, H], W [V, H], y [n] -> (logp [n], lse [n]). The max shift is the
    textbook one: lse = m + log sum exp(z - m). z_chunks: the logits as
    logit_chunks(rows, W, chunk) returns them, if already computed (otherwise
    each pass computes them again).
    """
    rows = np.asarray(rows, dtype=np.float64)
    W = np.asarray(W, dtype=np.float64)
    n = rows.shape[0]
    V = W.shape[0]
    if n == 0:
        return np.zeros(0), np.zeros(0)

    def z_of(c, v0):
        return z_chunks[c] if z_chunks is not None else rows @ W[v0:v0 + chunk].T

    m = np.full(n, -np.inf)
    for c, v0 in enumerate(range(0, V, chunk)):
        m = np.maximum(m, z_of(c, v0).max(axis=1))
    s = np.zeros(n)
    for c, v0 in enumerate(range(0, V, chunk)):
        s += np.exp(z_of(c, v0) - m[:, None]).sum(axis=1)
    lse = m + np.log(s)
    z_y = np.einsum("nh,nh->n", rows, W[np.asarray(y, dtype=np.int64)])
    return z_y - lse, lse


def response_rows(X, P, b, idx):
    """Final hidden states of response positions idx of sequence b: X[b, P + idx]."""
    return np.asarray(X[b, P + np.asarray(idx, dtype=np.int64)], dtype=np.float64)


def elbo_term(X, W, Y, P, mask, t):
    """Per-step loss l(y_t, t, y | x) of Eq. 4 for every sequence of one MC sample.

    l_b = (1/t_b) * sum_i 1[y_t^i = M] log p(y^i | y_t, x): a sum over masked
    response positions, no length normalisation. Returns l [B] (fp64).
    """
    B = mask.shape[0]
    ell = np.zeros(B)
    for b in range(B):
        idx = np.nonzero(mask[b])[0]
        if idx.size == 0:
            continue
        logp, _ = token_logprobs(response_rows(X, P, b, idx), W, Y[b, idx])
        ell[b] = logp.sum() / t[b]
    return ell


# ---------------------------------------------------------------------------
# BGPO bound (Eq. 10, 13, 14) and loss (Algorithm 1, Eq. 19)
# ---------------------------------------------------------------------------

def bound_coeffs(ell, ell_old, A, n_t, loss_scale):
    """d_j (Eq. 10), g_j (Eq. 13) and coef = dL_j / dl_j for L_j = -loss_scale g_j.

    A >= 0 (Taylor, Lemma 1): g = (1 + d) A / n_t, dg/dl = A / n_t.
    A <  0 (Jensen, Lemma 2): g = e^d A / n_t,     dg/dl = e^d A / n_t.
    """
    ell = np.asarray(ell, dtype=np.float64)
    ell_old = np.asarray(ell_old, dtype=np.float64)
    A = np.asarray(A, dtype=np.float64)
    d = ell - ell_old
    taylor = A >= 0
    with np.errstate(over="raise"):
        e = np.exp(np.where(taylor, 0.0, d))
    g = np.where(taylor, (1.0 + d) * A / n_t, e * A / n_t)
    dg_dl = np.where(taylor, A / n_t, e * A / n_t)
    coef = -loss_scale * dg_dl
    if not (np.all(np.isfinite(g)) and np.all(np.isfinite(coef))):
        raise FloatingPointError("non-finite BGPO bound coefficient")
    return d, g, coef


def vrpo_ratio(ell, ell_old, A):
    """R_hat of Eq. 7: exp(B_hat_theta - B_hat_old) A with B_hat the mean over j (Eq. 5).

    ell, ell_old [B, n_t]; A [B]. Returns R_hat [B].
    """
    ell = np.asarray(ell, dtype=np.float64)
    ell_old = np.asarray(ell_old, dtype=np.float64)
    return np.exp(ell.mean(axis=1) - ell_old.mean(axis=1)) * np.asarray(A, dtype=np.float64)


def vrpo_coeffs(ell, ell_old, A, loss_scale):
    """R_hat (Eq. 7) and dL/dl_{b,j} for L = -loss_scale * sum_b R_hat_b.

    With B_hat the mean over the n_t samples (Eq. 5), dR_hat/dl_{b,j} =
    e^{mean_j d_{b,j}} A_b / n_t for every j (Sec. 3.2). ell, ell_old [B, n_t];
    returns (R_hat [B], coef [B]).
    """
    ell = np.asarray(ell, dtype=np.float64)
    ell_old = np.asarray(ell_old, dtype=np.float64)
    A = np.asarray(A, dtype=np.float64)
    n_t = ell.shape[1]
    e = np.exp(ell.mean(axis=1) - ell_old.mean(axis=1))
    R = e * A
    coef = -loss_scale * e * A / n_t
    if not (np.all(np.isfinite(R)) and np.all(np.isfinite(coef))):
        raise FloatingPointError("non-finite VRPO coefficient")
    return R, coef


def group_advantage(rewards, G):
    """Eq. 18: (r - mean_G r) / std_G r within consecutive groups of G responses.

    Population std (ddof = 0); a zero-std group gets advantage 0.
    """
    r = np.asarray(rewards, dtype=np.float64).reshape(-1, G)
    mu = r.mean(axis=1, keepdims=True)
    sd = r.std(axis=1, keepdims=True)
    safe = np.where(sd > 0, sd, 1.0)
    A = np.where(sd > 0, (r - mu) / safe, 0.0)
    return A.reshape(-1)


# ---------------------------------------------------------------------------
# Gradients of one MC sample (backpropagation of L_j, Algorithm 1)
# ---------------------------------------------------------------------------

def elbo_term_grads(X, W, Y, P, mask, t, coef, chunk=8192, with_ell=False):
    """Gradient of sum_b coef_b * l_b (one MC sample) w.r.t. X and W.

    With w_r = coef_b / t_b for masked row r of sequence b and p_r = softmax(W x_r):
      dz_r = w_r (onehot(y_r) - p_r),  dX[b, i] = W^T dz_r,  dW = sum_r dz_r x_r^T.
    Returns (dX_resp [B, R, H], dW [V, H]) in fp64; dX covers response rows only
    (prompt rows get no gradient from Eq. 4). with_ell=True also returns the
    per-step ELBO term l [B] of Eq. 4 from the same log-probabilities, first:
    (l, dX_resp, dW).
    """
    W = np.asarray(W, dtype=np.float64)
    B, R = mask.shape
    V, H = W.shape
    dX = np.zeros((B, R, H))
    dW = np.zeros((V, H))
    ell = np.zeros(B)
    for b in range(B):
        idx = np.nonzero(mask[b])[0]
        if idx.size == 0:
            continue
        rows = response_rows(X, P, b, idx)
        y = np.asarray(Y[b, idx], dtype=np.int64)
        zs = logit_chunks(rows, W, chunk) if rows.shape[0] * V <= Z_KEEP_ELEMS else None
        logp, lse = token_logprobs(rows, W, y, chunk, zs)
        ell[b] = logp.sum() / t[b]
        w = coef[b] / t[b]
        for c, v0 in enumerate(range(0, V, chunk)):
            v1 = min(V, v0 + chunk)
            z = zs[c] if zs is not None else rows @ W[v0:v1].T
            dz = -w * np.exp(z - lse[:, None])
            hit = (y >= v0) & (y < v1)
            dz[np.nonzero(hit)[0], y[hit] - v0] += w
            dW[v0:v1] += dz.T @ rows
            dX[b, idx] += dz @ W[v0:v1]
    if with_ell:
        return ell, dX, dW
    return dX, dW


# ---------------------------------------------------------------------------
# Algorithm 1, inner loops: all n_t MC samples of one batch
# ---------------------------------------------------------------------------

def sample_masks(seed, B, R, n_t, t_mode, b_offset=0, resp_len=None):
    """(t [n_t, B], mask [n_t, B, R]) for every MC sample j."""
    ts, masks = [], []
    for j in range(n_t):
        _, _, t, m = sample_t_mask(seed, B, R, j, n_t, t_mode, b_offset, resp_len)
        ts.append(t)
        masks.append(m)
    return np.stack(ts), np.stack(masks)


def elbo_all(X, W, Y, P, ts, masks):
    """l_{b,j} for every sequence and MC sample: [B, n_t] (Eq. 4 for each j)."""
    return np.stack([elbo_term(X, W, Y, P, masks[j], ts[j]) for j in range(len(ts))], axis=1)


def bgpo_step(X, W, Y, P, A, ell_old, ts, masks, loss_scale):
    """BGPO objective and accumulated gradients over the n_t samples (Algorithm 1).

    ell_old [B, n_t] is the old policy's l on the same (t, mask) draws (Eq. 10).
    Returns dict: ell [B, n_t], d, g, coef [B, n_t], R_lb [B] (Eq. 14),
    loss = -loss_scale * sum_b R_lb_b, dX [B, R, H], dW [V, H].
    """
    n_t = len(ts)
    ell = elbo_all(X, W, Y, P, ts, masks)
    d, g, coef = bound_coeffs(ell, ell_old, np.asarray(A)[:, None], n_t, loss_scale)
    B, R = masks.shape[1:]
    V, H = np.asarray(W).shape
    dX = np.zeros((B, R, H))
    dW = np.zeros((V, H))
    for j in range(n_t):   # gradient accumulation, one MC sample at a time
        gx, gw = elbo_term_grads(X, W, Y, P, masks[j], ts[j], coef[:, j])
        dX += gx
        dW += gw
    R_lb = g.sum(axis=1)
    return dict(ell=ell, d=d, g=g, coef=coef, R_lb=R_lb,
                loss=-loss_scale * R_lb.sum(), dX=dX, dW=dW)


def bgpo_step_per_sample_x(Xs, W, Y, P, A, ell_old, ts, masks, loss_scale):
    """Algorithm 1 with hidden states that differ between MC samples.

    In the paper p_theta(y^i | y_t, x) conditions on the masked sequence y_t
    (Sec. 2.1, Eq. 4), so every MC sample j runs the network on its own input
    and its LM head sees its own final hidden states X_j. Xs [n_t, B, P+R, H]
    holds X_j for each j. Each sample's l_j, bound coefficients (Eq. 10, 13) and
    gradient are those of bgpo_step with X replaced by X_j; the gradient of
    dHidden is per sample (it flows back through sample j's own forward pass),
    while dW accumulates over the samples (Algorithm 1).
    Returns dict: ell, d, g, coef [B, n_t], R_lb [B], loss, dX [n_t, B, R, H]
    (dL/dX_j for each j), dW [V, H].
    """
    n_t = len(ts)
    ell = np.stack([elbo_term(Xs[j], W, Y, P, masks[j], ts[j]) for j in range(n_t)], axis=1)
    d, g, coef = bound_coeffs(ell, ell_old, np.asarray(A)[:, None], n_t, loss_scale)
    B, R = masks.shape[1:]
    V, H = np.asarray(W).shape
    dX = np.zeros((n_t, B, R, H))
    dW = np.zeros((V, H))
    for j in range(n_t):   # gradient accumulation, one MC sample at a time
        gx, gw = elbo_term_grads(Xs[j], W, Y, P, masks[j], ts[j], coef[:, j])
        dX[j] = gx
        dW += gw
    R_lb = g.sum(axis=1)
    return dict(ell=ell, d=d, g=g, coef=coef, R_lb=R_lb,
                loss=-loss_scale * R_lb.sum(), dX=dX, dW=dW)


def bgpo_loss_per_sample_x(Xs, W, Y, P, A, ell_old, ts, masks, loss_scale):
    """Scalar loss of bgpo_step_per_sample_x with the draws held fixed."""
    ell = np.stack([elbo_term(Xs[j], W, Y, P, masks[j], ts[j]) for j in range(len(ts))], axis=1)
    _, g, _ = bound_coeffs(ell, ell_old, np.asarray(A)[:, None], len(ts), loss_scale)
    return -loss_scale * g.sum()


def bgpo_loss(X, W, Y, P, A, ell_old, ts, masks, loss_scale):
    """Scalar loss -loss_scale * sum_b sum_j g_{b,j} with the draws held fixed."""
    ell = elbo_all(X, W, Y, P, ts, masks)
    _, g, _ = bound_coeffs(ell, ell_old, np.asarray(A)[:, None], len(ts), loss_scale)
    return -loss_scale * g.sum()


def vrpo_loss(X, W, Y, P, A, ell_old, ts, masks, loss_scale):
    """Scalar -loss_scale * sum_b R_hat_b with R_hat of Eq. 7 (draws held fixed)."""
    ell = elbo_all(X, W, Y, P, ts, masks)
    return -loss_scale * vrpo_ratio(ell, ell_old, A).sum()


# ---------------------------------------------------------------------------
# Gradient variance and bias vs n_t (Sec. 4.3)
# ---------------------------------------------------------------------------

def grad_std_bias(grads, golden):
    """Sec. 4.3 statistics of repeated gradient estimates of one batch.

    grads [K, ...]: K gradients computed with independent MC draws; golden: the
    reference gradient (the paper uses n_t = 256). Reading of the figure, whose
    values are not printed: std = mean over parameters of the per-parameter
    standard deviation over the K repeats (population, ddof = 0); bias = mean
    over parameters of |mean over repeats - golden|.
    """
    g = np.asarray(grads, dtype=np.float64)
    gold = np.asarray(golden, dtype=np.float64)
    std = g.std(axis=0).mean()
    bias = np.abs(g.mean(axis=0) - gold).mean()
    return float(std), float(bias)
