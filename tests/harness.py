"""Test-side drivers: the BGPO inner loops (Algorithm 1) through the C ABI on the
GPU, and the same loops through the fp64 oracle on the CPU, on the same seeded
inputs."""
import numpy as np

from oracle import bgpo_oracle as O


def ensure_built(checked=False):
    """Builds lib/libbgpo.so (checked=True: lib/libbgpo_checked.so) when it is
    missing (nvcc cross-compiles without a GPU)."""
    import os
    from paper_2510_11683_gb300 import build as B
    path = B.CHECKED_LIB_PATH if checked else B.LIB_PATH
    if not os.path.exists(path):
        B.build(checked=checked)
    return path


def to64(t):
    """torch tensor (bf16/f32/int) -> numpy float64 / int64 (exact widening)."""
    import torch
    if t.dtype in (torch.int32, torch.int64):
        return t.cpu().numpy().astype(np.int64)
    return t.cpu().to(torch.float64).numpy()


def oracle_advantages(wl, inp):
    if inp["A"] is not None:
        return to64(inp["A"])
    return O.group_advantage(to64(inp["rewards"]), wl.G)


def record_margin(test, **values):
    """Appends one JSON line of parity margins (errors reached against the
    oracle) to the file named by BGPO_MARGINS_OUT, when that is set."""
    import json
    import os
    path = os.environ.get("BGPO_MARGINS_OUT")
    if path:
        with open(path, "a") as f:
            f.write(json.dumps({"test": test, **{k: float(v) for k, v in values.items()}}) + "\n")


def oracle_run(wl, inp, loss_scale=None, b_offset=0, resp_len=None, W_old=None):
    """Algorithm 1 inner loops in fp64: draws, l_self, l_old, bound, grads.

    l_old = l_self + eps, or, with a second head W_old, the old policy's own
    l on the same draws (Eq. 10)."""
    X, W, Y = to64(inp["X"]), to64(inp["W"]), to64(inp["Y"])
    ls = 1.0 / wl.G if loss_scale is None else loss_scale
    A = oracle_advantages(wl, inp)
    ts, masks = O.sample_masks(wl.seed, wl.B, wl.R, wl.n_t, wl.t_mode, b_offset, resp_len)
    ell_self = O.elbo_all(X, W, Y, wl.P, ts, masks)
    if W_old is None:
        ell_old = ell_self + to64(inp["eps"])
    else:
        ell_old = O.elbo_all(X, to64(W_old), Y, wl.P, ts, masks)
    out = O.bgpo_step(X, W, Y, wl.P, A, ell_old, ts, masks, ls)
    out.update(ts=ts, masks=masks, A=A, ell_old=ell_old, ell_self=ell_self)
    return out


def default_vocab_chunk(V, rows=None):
    """The library's chunk width without dW pairing for a vocabulary V split
    into ceil(V / 32768) equal pieces rounded up to 256 columns (0 when that
    is one piece). With `rows` = B R, the default proper: 0 (the whole
    vocabulary) also when its dL/dz, roundup(rows, 256) x roundup(V, 64) bf16
    values, takes at most 1 GiB."""
    if rows is not None and 2 * (-(-rows // 256) * 256) * (-(-V // 64) * 64) <= 1 << 30:
        return 0
    n = -(-V // 32768)
    w = -(-(-(-V // n)) // 256) * 256
    return 0 if w >= V else w


def gpu_run(wl, inp, dev="cuda", loss_scale=None, trace=None, b_offset=0, resp_len=None,
            keep_logits=False, pair_dw=False, W_old=None, vocab_chunk=0):
    """Algorithm 1 inner loops through the C ABI; inputs already on `dev`.

    The old-policy pass is forward-only and keeps no logits; `keep_logits`
    sets BGPO_FLAG_KEEP_LOGITS for the inner loop (the workspace is sized for
    it, and the old-policy pass runs on the same workspace without the flag);
    `pair_dw` sets BGPO_FLAG_PAIR_DW for the inner loop in the same way.
    W_old (device bf16 [V, H]): the old-policy pass runs with this head and
    l_old is its output (no eps); otherwise l_old = l_self + eps.
    vocab_chunk: bgpo_problem.vocab_chunk of the inner loop (0 = default).

    Returns dict of torch tensors: ell [B, n_t], ell_old, coef, g, t [n_t, B],
    masks [n_t, B, R], A, dX [B, R, H], dW [V, H], ws.
    """
    import torch
    import paper_2510_11683_gb300 as bg

    lens = None
    if resp_len is not None:
        lens = torch.as_tensor(np.asarray(resp_len), dtype=torch.int32, device=dev)
    prob = bg.problem_from(wl, trace=trace, loss_scale=loss_scale, b_offset=b_offset,
                           resp_len=lens, keep_logits=keep_logits, pair_dw=pair_dw,
                           vocab_chunk=vocab_chunk)
    prob_old = bg.problem_from(wl, trace=trace, loss_scale=loss_scale, b_offset=b_offset,
                               resp_len=lens, vocab_chunk=vocab_chunk)
    ws = bg.alloc_workspace(prob, dev)
    bg.clear_device_error(ws)
    B, n_t = wl.B, wl.n_t
    X, W, Y = inp["X"], inp["W"], inp["Y"]
    if inp["A"] is not None:
        A = inp["A"].contiguous()
    else:
        A = torch.empty(B, dtype=torch.float32, device=dev)
        bg.group_advantage(prob, inp["rewards"], A)
    t = torch.empty((n_t, B), dtype=torch.float32, device=dev)
    masks = torch.empty((n_t, B, wl.R), dtype=torch.uint8, device=dev)
    ell_self = torch.empty((n_t, B), dtype=torch.float32, device=dev)
    for j in range(n_t):          # old-policy pass (same draws, Eq. 10)
        bg.sample_mask(prob_old, j, ws, t[j], masks[j])
        bg.elbo_fwd(prob_old, j, X, W if W_old is None else W_old, Y, ws, ell_self[j])
    if W_old is None:
        ell_old = (ell_self + inp["eps"].T.contiguous()).contiguous()
    else:
        ell_old = ell_self.clone()
    ell = torch.empty((n_t, B), dtype=torch.float32, device=dev)
    coef = torch.empty((n_t, B), dtype=torch.float32, device=dev)
    g = torch.empty((n_t, B), dtype=torch.float32, device=dev)
    dX = torch.zeros((B, wl.R, wl.H), dtype=torch.float32, device=dev)
    dW = torch.zeros((wl.V, wl.H), dtype=torch.float32, device=dev)
    for j in range(n_t):          # Algorithm 1, one MC sample at a time
        bg.sample_mask(prob, j, ws)
        bg.elbo_fwd(prob, j, X, W, Y, ws, ell[j])
        bg.bound_coeffs(prob, j, ell[j], ell_old[j], A, coef[j], g[j], ws)
        bg.elbo_bwd_accumulate(prob, j, X, W, Y, coef[j], ws, dX, dW)
    torch.cuda.synchronize()
    return dict(ell=ell.T, ell_old=ell_old.T, coef=coef.T, g=g.T, t=t, masks=masks, A=A,
                dX=dX, dW=dW, ws=ws, prob=prob, ell_self=ell_self.T, lens=lens)


def rel_ell_err(got, ref):
    """|l_gpu - l_ref| / max(|l_ref|, 1) elementwise (the per-sequence tolerance rule)."""
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    return np.abs(got - ref) / np.maximum(np.abs(ref), 1.0)


def normwise(got, ref):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    den = np.linalg.norm(ref)
    return np.linalg.norm(got - ref) / (den if den > 0 else 1.0)


def oracle_run_vrpo(wl, inp, loss_scale=None):
    """The ELBO-based objective of Eq. 7 in fp64: R_hat and its accumulated gradients."""
    X, W, Y = to64(inp["X"]), to64(inp["W"]), to64(inp["Y"])
    ls = 1.0 / wl.G if loss_scale is None else loss_scale
    A = oracle_advantages(wl, inp)
    ts, masks = O.sample_masks(wl.seed, wl.B, wl.R, wl.n_t, wl.t_mode)
    ell = O.elbo_all(X, W, Y, wl.P, ts, masks)
    ell_old = ell + to64(inp["eps"])
    R, coef = O.vrpo_coeffs(ell, ell_old, A, ls)
    dX = np.zeros((wl.B, wl.R, wl.H))
    dW = np.zeros((wl.V, wl.H))
    for j in range(wl.n_t):
        gx, gw = O.elbo_term_grads(X, W, Y, wl.P, masks[j], ts[j], coef)
        dX += gx
        dW += gw
    return dict(ell=ell, R=R, coef=coef, dX=dX, dW=dW)


def gpu_run_vrpo(wl, inp, strategy, dev="cuda"):
    """Eq. 7 through the C ABI. strategy "retain": one workspace per MC sample
    (forward state kept for all n_t samples); "recompute": one workspace, each
    sample's forward run again before its backward."""
    import torch
    import paper_2510_11683_gb300 as bg

    prob = bg.problem_from(wl)
    B, n_t = wl.B, wl.n_t
    X, W, Y = inp["X"], inp["W"], inp["Y"]
    A = torch.empty(B, dtype=torch.float32, device=dev)
    if inp["A"] is not None:
        A.copy_(inp["A"])
    else:
        bg.group_advantage(prob, inp["rewards"], A)
    n_ws = n_t if strategy == "retain" else 1
    wss = [bg.alloc_workspace(prob, dev) for _ in range(n_ws)]
    for ws in wss:
        bg.clear_device_error(ws)
    ell = torch.empty((n_t, B), dtype=torch.float32, device=dev)
    for j in range(n_t):
        ws = wss[j % n_ws]
        bg.sample_mask(prob, j, ws)
        bg.elbo_fwd(prob, j, X, W, Y, ws, ell[j])
    ell_old = (ell + inp["eps"].T).contiguous()
    coef = torch.empty(B, dtype=torch.float32, device=dev)
    R = torch.empty(B, dtype=torch.float32, device=dev)
    bg.vrpo_coeffs(prob, ell, ell_old, A, coef, R, wss[0])
    dX = torch.zeros((B, wl.R, wl.H), dtype=torch.float32, device=dev)
    dW = torch.zeros((wl.V, wl.H), dtype=torch.float32, device=dev)
    tmp = torch.empty(B, dtype=torch.float32, device=dev)
    for j in range(n_t):
        ws = wss[j % n_ws]
        if strategy != "retain":
            bg.sample_mask(prob, j, ws)
            bg.elbo_fwd(prob, j, X, W, Y, ws, tmp)
        bg.elbo_bwd_accumulate(prob, j, X, W, Y, coef, ws, dX, dW)
    torch.cuda.synchronize()
    return dict(ell=ell.T, R=R, coef=coef, dX=dX, dW=dW, ws=wss)
