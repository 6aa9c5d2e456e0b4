"""Sec. 4.3 study (gradient std and bias vs n_t) on the device, checked at a
small size against the fp64 oracle computing the same statistic on the same
MC draws."""
import numpy as np
import pytest

from oracle import bgpo_oracle as O
from synth import CONFIGS, make_inputs
from tests.harness import ensure_built, oracle_advantages, to64

pytestmark = pytest.mark.gpu


def test_grad_std_bias_match_oracle():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    ensure_built()
    import bench
    import paper_2510_11683_gb300 as bg
    wl = CONFIGS["tiny"].with_(eps_std=0.0)
    nts, repeats, golden_nt = (1, 4), 4, 32
    got = bench.grad_variance(bg, wl, nts, repeats, golden_nt, torch.device("cuda", 0))
    inp = make_inputs(wl)
    X, W, Y = to64(inp["X"]), to64(inp["W"]), to64(inp["Y"])
    A = oracle_advantages(wl, inp)

    def grad(n_t, seed):
        ts, masks = O.sample_masks(seed, wl.B, wl.R, n_t, wl.t_mode)
        ell = O.elbo_all(X, W, Y, wl.P, ts, masks)
        return O.bgpo_step(X, W, Y, wl.P, A, ell, ts, masks, 1.0 / wl.G)["dW"]

    golden = grad(golden_nt, bench.grad_seed(wl, golden_nt, -1))
    for point, n_t in zip(got, nts):
        grads = np.stack([grad(n_t, bench.grad_seed(wl, n_t, r)) for r in range(repeats)])
        std, bias = O.grad_std_bias(grads, golden)
        assert point["n_t"] == n_t
        assert abs(point["std"] - std) <= 0.03 * std
        assert abs(point["bias"] - bias) <= 0.03 * bias
    assert got[0]["std"] > got[1]["std"]
