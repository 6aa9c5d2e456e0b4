"""The synthetic parity workloads exercise what they are meant to.

A gradient comparison is vacuous when every advantage is zero (then every
bound coefficient, dL/dz, dX and dW is exactly zero on both sides): Eq. 18 gives
A = 0 for a group whose rewards are all equal.
"""
import numpy as np
import pytest

from oracle import bgpo_oracle as O
from synth import CONFIGS, make_inputs


@pytest.mark.parametrize("name", ["tiny", "ragged", "ragged_strat", "llada8b_r256"])
def test_parity_workloads_have_nonzero_advantages(name):
    wl = CONFIGS[name]
    inp = make_inputs(wl, need_w=False)
    if inp["A"] is not None:
        A = inp["A"].numpy().astype(np.float64)
    else:
        A = O.group_advantage(inp["rewards"].numpy().astype(np.float64), wl.G)
    assert np.count_nonzero(A) >= max(1, wl.B // 2), A


def test_parity_workloads_mask_something_in_every_sample():
    for name in ("tiny", "ragged", "ragged_strat"):
        wl = CONFIGS[name]
        _, masks = O.sample_masks(wl.seed, wl.B, wl.R, wl.n_t, wl.t_mode)
        assert (masks.reshape(wl.n_t, -1).sum(axis=1) > 0).all(), name
