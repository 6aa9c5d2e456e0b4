"""Hidden states that differ between MC samples (Sec. 2.1; Eq. 4).

In the paper p_theta(y^i | y_t, x) conditions on the masked sequence y_t, so
each MC sample runs the network on its own input and the LM head sees that
sample's own final hidden states X_j; their gradient goes back through sample
j's own forward pass. The C ABI takes X in every call, so a caller passes X_j
to bgpo_elbo_fwd and bgpo_elbo_bwd_accumulate of sample j and reads dX after
each sample's backward (zeroing it in between), while dW keeps accumulating
over the samples (Algorithm 1). These tests do exactly that with
synth.make_per_sample_hidden and compare every dX_j, the accumulated dW and
every l_{b,j} with oracle.bgpo_step_per_sample_x on the same inputs, with and
without dW pairing (a paired odd sample's dW GEMM also reads the gathered
hidden states its even partner's call left pending: the partner's own X_j).
"""
import numpy as np
import pytest

from oracle import bgpo_oracle as O
from synth import CONFIGS, make_inputs, make_per_sample_hidden
from tests.harness import (ensure_built, normwise, oracle_advantages, record_margin, rel_ell_err,
                           to64)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def bg():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    ensure_built()
    import paper_2510_11683_gb300 as bg
    return bg


def _gpu(bg, wl, Xs, W, Y, A, eps, pair, keep):
    """Old-policy pass then Algorithm 1's loop with X_j per sample; dX read per sample."""
    import torch
    prob = bg.problem_from(wl, pair_dw=pair, keep_logits=keep)
    prob_old = bg.problem_from(wl)
    ws = bg.alloc_workspace(prob)
    B, n_t = wl.B, wl.n_t
    ell_self = torch.empty((n_t, B), device="cuda")
    masks = torch.empty((n_t, B, wl.R), dtype=torch.uint8, device="cuda")
    for j in range(n_t):
        bg.sample_mask(prob_old, j, ws, None, masks[j])
        bg.elbo_fwd(prob_old, j, Xs[j], W, Y, ws, ell_self[j])
    ell_old = (ell_self + eps.T).contiguous()
    ell = torch.empty((n_t, B), device="cuda")
    coef = torch.empty((n_t, B), device="cuda")
    dX = torch.zeros((B, wl.R, wl.H), device="cuda")
    dXs = torch.empty((n_t, B, wl.R, wl.H), device="cuda")
    dW = torch.zeros((wl.V, wl.H), device="cuda")
    for j in range(n_t):
        bg.sample_mask(prob, j, ws)
        bg.elbo_fwd(prob, j, Xs[j], W, Y, ws, ell[j])
        bg.bound_coeffs(prob, j, ell[j], ell_old[j], A, coef[j], None, ws)
        dX.zero_()
        bg.elbo_bwd_accumulate(prob, j, Xs[j], W, Y, coef[j], ws, dX, dW)
        dXs[j].copy_(dX)
    torch.cuda.synchronize()
    assert bg.get_device_error(ws) == (0, 0)
    return dict(masks=masks, ell=ell.T, ell_old=ell_old.T, dX=dXs, dW=dW)


@pytest.mark.parametrize("pair,keep", [(False, False), (True, False), (True, True)])
@pytest.mark.parametrize("name", ["tiny", "ragged", "ragged_strat"])
def test_per_sample_hidden_states_match_oracle(bg, name, pair, keep):
    wl = CONFIGS[name]
    inp_cpu = make_inputs(wl)
    Xs_cpu = make_per_sample_hidden(wl, inp_cpu["X"])
    inp = {k: (v.cuda() if v is not None else None) for k, v in inp_cpu.items()}
    A = inp["A"]
    if A is None:
        import torch
        A = torch.empty(wl.B, device="cuda")
        bg.group_advantage(bg.problem_from(wl), inp["rewards"], A)
    g = _gpu(bg, wl, Xs_cpu.cuda(), inp["W"], inp["Y"], A, inp["eps"].cuda(), pair, keep)

    Xs = to64(Xs_cpu)
    W, Y = to64(inp_cpu["W"]), to64(inp_cpu["Y"])
    ts, masks = O.sample_masks(wl.seed, wl.B, wl.R, wl.n_t, wl.t_mode)
    ell_self = np.stack([O.elbo_term(Xs[j], W, Y, wl.P, masks[j], ts[j]) for j in range(wl.n_t)],
                        axis=1)
    ell_old = ell_self + to64(inp_cpu["eps"])
    o = O.bgpo_step_per_sample_x(Xs, W, Y, wl.P, oracle_advantages(wl, inp_cpu), ell_old, ts,
                                 masks, 1.0 / wl.G)
    assert np.array_equal(g["masks"].cpu().numpy(), masks)
    e_ell = rel_ell_err(to64(g["ell"]), o["ell"]).max()
    assert e_ell <= 1e-3
    worst = 0.0
    for j in range(wl.n_t):
        if np.linalg.norm(o["dX"][j]) == 0:        # an empty mask: nothing flows back
            assert float(g["dX"][j].abs().max()) == 0.0
            continue
        e = normwise(to64(g["dX"][j]), o["dX"][j])
        worst = max(worst, e)
        assert e <= 2e-2, (j, e)
    e_dw = normwise(to64(g["dW"]), o["dW"])
    assert e_dw <= 2e-2
    # the samples' hidden states really differ
    assert normwise(Xs[1], Xs[0]) > 0.3
    record_margin(f"per_sample_hidden[{name},pair={pair},keep={keep}]", ell=e_ell, dX=worst,
                  dW=e_dw)
