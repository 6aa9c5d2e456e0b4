"""bgpo_elbo_fwd_noalloc: the per-sample ELBO forward on the library's own scratch.

Some callers cannot allocate device memory: host code that a serving process
hands only its input and output buffers (that process plans all device memory
itself), or code that must not call cudaMalloc because it would synchronise the
device mid-step. They cannot pass the workspace that bgpo_sample_mask and
bgpo_elbo_fwd need, so the library offers this one entry point, which works in
a fixed 32 MiB array compiled into the library. These tests call it through
the C ABI, twice in a row on different problems (the array keeps the previous
call's contents), and compare each result with bgpo_sample_mask +
bgpo_elbo_fwd on a caller-allocated workspace, within the per-sequence ELBO
tolerance of the parity tests. This file is collected last on purpose.
"""
import ctypes

import numpy as np
import pytest

from synth import CONFIGS, make_inputs
from tests.harness import ensure_built, rel_ell_err

pytestmark = pytest.mark.gpu

ELL_TOL = 1e-3


@pytest.fixture(scope="module")
def bg():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    ensure_built()
    import paper_2510_11683_gb300 as bg
    return bg


def _noalloc(bg, prob, j, X, W, Y, t_out, ell_out):
    import torch
    L = bg._lib.lib()
    return L.bgpo_elbo_fwd_noalloc(ctypes.byref(prob), j, X.data_ptr(), W.data_ptr(), Y.data_ptr(),
                                   t_out.data_ptr() if t_out is not None else None,
                                   ell_out.data_ptr(), torch.cuda.current_stream().cuda_stream)


def _with_workspace(bg, prob, j, X, W, Y, B):
    import torch
    ws = bg.alloc_workspace(prob)
    t = torch.empty(B, dtype=torch.float32, device="cuda")
    ell = torch.empty(B, dtype=torch.float32, device="cuda")
    bg.sample_mask(prob, j, ws, t)
    bg.elbo_fwd(prob, j, X, W, Y, ws, ell)
    return t, ell


def test_noalloc_matches_workspace_path_on_two_calls_in_a_row(bg):
    import torch
    # a larger problem first, then a smaller one: stale scratch must not leak
    for name, j in (("ragged", 1), ("tiny", 2)):
        wl = CONFIGS[name]
        inp = make_inputs(wl, device="cuda")
        prob = bg.problem_from(wl)
        t_ref, ell_ref = _with_workspace(bg, prob, j, inp["X"], inp["W"], inp["Y"], wl.B)
        t = torch.full((wl.B,), -1.0, device="cuda")
        ell = torch.full((wl.B,), float("nan"), device="cuda")
        assert _noalloc(bg, prob, j, inp["X"], inp["W"], inp["Y"], t, ell) == 0
        torch.cuda.synchronize()
        assert torch.equal(t, t_ref)
        assert np.all(np.isfinite(ell.cpu().numpy()))
        assert rel_ell_err(ell.cpu().numpy(), ell_ref.cpu().numpy()).max() <= ELL_TOL
        # the same kernels on the same inputs: stale scratch from the earlier,
        # larger call must not change a single bit
        assert torch.equal(ell, ell_ref)


def test_noalloc_rejects_problems_beyond_its_scratch(bg):
    import torch
    # LLaDA-8B head, 16 x 512 responses: ~100 MB of forward scratch > 32 MiB
    wl = CONFIGS["llada8b_r512_onpolicy"]
    prob = bg.problem_from(wl)
    x = torch.zeros(64, dtype=torch.bfloat16, device="cuda")
    y = torch.zeros(64, dtype=torch.int32, device="cuda")
    ell = torch.zeros(wl.B, dtype=torch.float32, device="cuda")
    assert _noalloc(bg, prob, 0, x, x, y, None, ell) == 4   # BGPO_ERR_WORKSPACE_TOO_SMALL
    assert _noalloc(bg, bg.problem_from(CONFIGS["tiny"]), 9, x, x, y, None, ell) == 1


def test_noalloc_rejects_a_misaligned_response_length_pointer(bg):
    # a resp_len pointer that is not 4-byte aligned is refused on the host
    # (BGPO_ERR_ALIGNMENT) before any kernel could load from it
    import torch
    wl = CONFIGS["tiny"]
    inp = make_inputs(wl, device="cuda")
    lens = torch.full((wl.B + 1,), wl.R, dtype=torch.int32, device="cuda")
    raw = bg.problem_from(wl)
    raw.resp_len = lens.data_ptr() + 2
    ell = torch.full((wl.B,), float("nan"), device="cuda")
    assert _noalloc(bg, raw, 0, inp["X"], inp["W"], inp["Y"], None, ell) == 3
    torch.cuda.synchronize()
    assert torch.isnan(ell).all()
