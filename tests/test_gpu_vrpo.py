"""The ELBO-based objective BGPO bounds (VRPO, Eq. 7) through the C ABI.

Its per-sample weight e^{mean d} A / n_t depends on all n_t samples, so the
backward pass can only start after every sample's forward: either every
sample's workspace is kept (memory grows with n_t) or each forward is run
twice. Both strategies are checked against the fp64 oracle, and on-policy
(d = 0) against BGPO itself, whose gradient must then be identical
(Equivalence, Sec. 3.2).
"""
import numpy as np
import pytest

from oracle import bgpo_oracle as O
from synth import CONFIGS, make_inputs
from tests.harness import (ensure_built, gpu_run, gpu_run_vrpo, normwise, oracle_run_vrpo,
                           rel_ell_err, to64)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def bg():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    ensure_built()
    import paper_2510_11683_gb300 as bg
    return bg


def test_vrpo_coeffs_on_identical_inputs(bg):
    import torch
    rng = np.random.default_rng(11)
    B, n_t = 257, 7
    p = bg.problem(B, 1, 1, 64, 8, n_t, 8)
    ws = bg.alloc_workspace(p)
    bg.clear_device_error(ws)
    ell = (rng.standard_normal((n_t, B)) * 30).astype(np.float32)
    old = (ell + rng.standard_normal((n_t, B)) * 0.2).astype(np.float32)
    A = rng.standard_normal(B).astype(np.float32)
    cuda = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()
    coef = torch.empty(B, device="cuda")
    R = torch.empty(B, device="cuda")
    bg.vrpo_coeffs(p, cuda(ell), cuda(old), cuda(A), coef, R, ws)
    R_ref, c_ref = O.vrpo_coeffs(ell.T.astype(np.float64), old.T.astype(np.float64),
                                 A.astype(np.float64), 1.0 / 8)
    assert np.allclose(R.cpu().numpy(), R_ref, rtol=1e-5, atol=1e-7)
    assert np.allclose(coef.cpu().numpy(), c_ref, rtol=1e-5, atol=1e-9)
    assert bg.get_device_error(ws) == (0, 0)


@pytest.mark.parametrize("name", ["tiny", "ragged"])
@pytest.mark.parametrize("strategy", ["retain", "recompute"])
def test_vrpo_gradients_match_oracle(bg, name, strategy):
    wl = CONFIGS[name]
    inp = make_inputs(wl, device="cuda")
    g = gpu_run_vrpo(wl, inp, strategy)
    o = oracle_run_vrpo(wl, {k: (v.cpu() if v is not None else None) for k, v in inp.items()})
    assert rel_ell_err(to64(g["ell"]), o["ell"]).max() <= 1e-3
    assert np.allclose(to64(g["coef"]), o["coef"], rtol=2e-3, atol=1e-7)
    assert normwise(to64(g["dW"]), o["dW"]) <= 2e-2
    assert normwise(to64(g["dX"]), o["dX"]) <= 2e-2
    for ws in g["ws"]:
        assert bg.get_device_error(ws) == (0, 0)


def test_on_policy_vrpo_equals_bgpo_bitwise(bg):
    import torch
    wl = CONFIGS["ragged"].with_(eps_std=0.0)
    inp = make_inputs(wl, device="cuda")
    v = gpu_run_vrpo(wl, inp, "recompute")
    b = gpu_run(wl, inp)
    assert torch.equal(v["dW"], b["dW"]) and torch.equal(v["dX"], b["dX"])
    assert torch.equal(v["R"], b["A"])
