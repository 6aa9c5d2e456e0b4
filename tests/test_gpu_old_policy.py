"""A separate old-policy head (Eq. 10): the old policy's l on the same draws.

BGPO evaluates the current policy and the old one on the same t and masks
(Eq. 10). Here the old-policy pass runs bgpo_elbo_fwd with a second LM head
W_old = W + 0.05 N(0, 1/H) (synth.make_old_head) on regenerated draws, so
d = l - l_old comes from two different heads, and the advantages are given
both signs so that both branches of Eq. 13 (Taylor for A >= 0, Jensen for
A < 0; Lemmas 1-2) run in one batch. l, l_old, the coefficients, dX and dW are
compared with the oracle run with the same W_old.

Tolerances: l and l_old within 1e-3 relative; coefficients within 1e-3 of the
fully independent oracle and within 1e-5 of the oracle fed the device's own
fp32 l and l_old; dX and dW within 2e-2 normwise.
"""
import numpy as np
import pytest

from oracle import bgpo_oracle as O
from synth import CONFIGS, make_inputs, make_old_head
from tests.harness import (ensure_built, gpu_run, normwise, oracle_advantages, oracle_run,
                           record_margin, rel_ell_err, to64)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def bg():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    ensure_built()
    import paper_2510_11683_gb300 as bg
    return bg


@pytest.mark.parametrize("pair", [False, True])
@pytest.mark.parametrize("name", ["tiny", "ragged", "ragged_strat"])
def test_separate_old_head_matches_oracle(bg, name, pair):
    wl = CONFIGS[name]
    inp_cpu = make_inputs(wl)
    A = inp_cpu["A"].clone()
    A[0] = -A[0].abs() - 0.1          # Jensen branch (Lemma 2)
    A[1] = A[1].abs() + 0.1           # Taylor branch (Lemma 1)
    inp_cpu["A"] = A
    W_old = make_old_head(wl, inp_cpu["W"])
    inp = {k: (v.cuda() if v is not None else None) for k, v in inp_cpu.items()}
    g = gpu_run(wl, inp, pair_dw=pair, W_old=W_old.cuda())
    o = oracle_run(wl, inp_cpu, W_old=W_old)
    assert bg.get_device_error(g["ws"]) == (0, 0)
    assert np.array_equal(g["masks"].cpu().numpy(), o["masks"])
    assert np.abs(o["d"]).max() > 0.05                       # the heads differ
    assert (o["A"] < 0).any() and (o["A"] >= 0).any()

    e_ell = rel_ell_err(to64(g["ell"]), o["ell"]).max()
    e_old = rel_ell_err(to64(g["ell_old"]), o["ell_old"]).max()
    assert e_ell <= 1e-3 and e_old <= 1e-3
    coef = to64(g["coef"])
    e_coef = (np.abs(coef - o["coef"]) / np.maximum(np.abs(o["coef"]), 1e-12)).max()
    assert e_coef <= 1e-3
    A64 = oracle_advantages(wl, inp_cpu)[:, None]
    _, g_same, c_same = O.bound_coeffs(to64(g["ell"]), to64(g["ell_old"]), A64, wl.n_t, 1.0 / wl.G)
    assert np.allclose(coef, c_same, rtol=1e-5, atol=1e-9)
    assert np.allclose(to64(g["g"]), g_same, rtol=1e-5, atol=1e-7)
    e_dx, e_dw = normwise(to64(g["dX"]), o["dX"]), normwise(to64(g["dW"]), o["dW"])
    assert e_dx <= 2e-2 and e_dw <= 2e-2
    assert np.linalg.norm(o["dW"]) > 0
    record_margin(f"separate_old_head[{name},pair={pair}]", ell=e_ell, ell_old=e_old,
                  coef=e_coef, dX=e_dx, dW=e_dw)
