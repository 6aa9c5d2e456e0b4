"""BGPO_FLAG_PAIR_DW: MC samples 2k and 2k + 1 share one dW GEMM whose K range
holds both samples' masked rows (Algorithm 1's gradient accumulation, with the
dW term of two samples summed before it reaches dW).

Checked against the fp64 oracle on the same seeded inputs (masks bit-exact, l
within 1e-3 relative, dX and dW within 2e-2 normwise) and against the unpaired
path (l and dX bit-identical, dW equal up to fp32 summation order), for even
and odd n_t, with and without kept logits, at the full LLaDA-8B head; and the
misuse that the device error word reports.
"""
import numpy as np
import pytest

from synth import CONFIGS, make_inputs
from tests.harness import ensure_built, gpu_run, normwise, oracle_run, rel_ell_err, to64

pytestmark = pytest.mark.gpu

ELL_TOL = 1e-3
GRAD_TOL = 2e-2
# paired and unpaired dW differ only in the order of fp32 additions
ORDER_TOL = 1e-5
# dX summed over the whole LLaDA-8B vocabulary at once or in 4 chunks: fp32
# order over a 126,464-long K whose terms mostly cancel (measured 2.0e-5)
VOCAB_ORDER_TOL = 1e-4

KID_MASK_COMPACT, KID_DW_GEMM = 0, 9


@pytest.fixture(scope="module")
def bg():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    ensure_built()
    import paper_2510_11683_gb300 as bg
    return bg


def _cpu(inp):
    return {k: (v.cpu() if v is not None else None) for k, v in inp.items()}


@pytest.mark.parametrize("keep", [False, True])
@pytest.mark.parametrize("name,n_t", [("tiny", None), ("tiny", 3), ("ragged", None), ("ragged", 6),
                                      ("ragged_strat", None)])
def test_paired_dw_matches_oracle_and_unpaired(bg, name, n_t, keep):
    import torch
    wl = CONFIGS[name] if n_t is None else CONFIGS[name].with_(n_t=n_t)
    inp = make_inputs(wl, device="cuda")
    a = gpu_run(wl, inp, keep_logits=keep)
    p = gpu_run(wl, inp, keep_logits=keep, pair_dw=True)
    assert bg.get_device_error(a["ws"]) == (0, 0)
    assert bg.get_device_error(p["ws"]) == (0, 0)
    assert torch.equal(p["ell"], a["ell"]) and torch.equal(p["dX"], a["dX"])
    assert normwise(to64(p["dW"]), to64(a["dW"])) <= ORDER_TOL
    assert not torch.equal(p["dW"], torch.zeros_like(p["dW"]))
    o = oracle_run(wl, _cpu(inp))
    assert np.array_equal(p["masks"].cpu().numpy(), o["masks"])
    assert rel_ell_err(to64(p["ell"]), o["ell"]).max() <= ELL_TOL
    assert normwise(to64(p["dX"]), o["dX"]) <= GRAD_TOL
    assert normwise(to64(p["dW"]), o["dW"]) <= GRAD_TOL


def test_paired_dw_at_the_full_head(bg):
    """Full LLaDA-8B head (494 vocabulary tiles, K = 4096), 4 samples with few
    masked rows each: the whole dW and dX against the oracle and the unpaired
    path. With so few rows both walk the whole vocabulary at once by default:
    the same l and dX bits, dW up to fp32 order. Walked in the 4 chunks of
    31,744 columns that larger batches use by default, paired and unpaired
    again agree bit for bit in dX, and the chunked dX equals the
    whole-vocabulary one up to fp32 order."""
    import torch
    from tests.harness import default_vocab_chunk
    wl = CONFIGS["llada8b_r256"].with_(B=2, P=8, R=24, n_t=4, G=2)
    inp_cpu = make_inputs(wl)
    inp = {k: (v.cuda() if v is not None else None) for k, v in inp_cpu.items()}
    p = gpu_run(wl, inp, pair_dw=True)
    assert bg.get_device_error(p["ws"]) == (0, 0)
    res = {k: p[k].cpu() for k in ("masks", "ell", "dX", "dW")}
    del p
    a = gpu_run(wl, inp)
    assert torch.equal(res["ell"], a["ell"].cpu()) and torch.equal(res["dX"], a["dX"].cpu())
    assert normwise(to64(res["dW"]), to64(a["dW"])) <= ORDER_TOL
    del a
    chunk = default_vocab_chunk(wl.V)
    assert chunk == 31744
    u = gpu_run(wl, inp, vocab_chunk=chunk)
    c = gpu_run(wl, inp, pair_dw=True, vocab_chunk=chunk)
    assert bg.get_device_error(u["ws"]) == (0, 0) and bg.get_device_error(c["ws"]) == (0, 0)
    assert torch.equal(c["ell"], u["ell"]) and torch.equal(c["dX"], u["dX"])
    assert normwise(to64(c["dW"]), to64(u["dW"])) <= ORDER_TOL
    assert normwise(to64(u["dX"]), to64(res["dX"])) <= VOCAB_ORDER_TOL
    del u, c
    torch.cuda.empty_cache()
    o = oracle_run(wl, inp_cpu)
    assert np.array_equal(res["masks"].numpy(), o["masks"])
    assert normwise(to64(res["dW"]), o["dW"]) <= GRAD_TOL
    assert normwise(to64(res["dX"]), o["dX"]) <= GRAD_TOL


def _sample(bg, p, j, inp, ws, dX, dW, coef_value=-0.25, remask=False):
    import torch
    wl_B = inp["X"].shape[0]
    ell = torch.empty(wl_B, device="cuda")
    coef = torch.full((wl_B,), coef_value, device="cuda")
    bg.sample_mask(p, j, ws)
    if remask:
        bg.sample_mask(p, j, ws)
    bg.elbo_fwd(p, j, inp["X"], inp["W"], inp["Y"], ws, ell)
    bg.elbo_bwd_accumulate(p, j, inp["X"], inp["W"], inp["Y"], coef, ws, dX, dW)


def _buffers(wl):
    import torch
    return (torch.zeros((wl.B, wl.R, wl.H), device="cuda"),
            torch.zeros((wl.V, wl.H), device="cuda"))


def test_masking_another_sample_while_one_is_pending_is_reported(bg):
    wl = CONFIGS["tiny"]
    inp = make_inputs(wl, device="cuda")
    p = bg.problem_from(wl, pair_dw=True)
    ws = bg.alloc_workspace(p)
    dX, dW = _buffers(wl)
    _sample(bg, p, 0, inp, ws, dX, dW)
    assert bg.get_device_error(ws) == (0, 0)
    assert float(dW.abs().max()) == 0.0      # sample 0's dW waits for sample 1
    assert float(dX.abs().max()) > 0.0       # dX does not wait
    bg.sample_mask(p, 2, ws)                 # sample 1 skipped: sample 0's dW is dropped
    assert bg.get_device_error(ws) == (1, KID_MASK_COMPACT * 16 + 5)


def test_odd_sample_without_its_partner_is_reported(bg):
    import torch
    wl = CONFIGS["tiny"]
    inp = make_inputs(wl, device="cuda")
    p = bg.problem_from(wl, pair_dw=True)
    ws = bg.alloc_workspace(p)
    dX, dW = _buffers(wl)
    _sample(bg, p, 1, inp, ws, dX, dW)
    assert bg.get_device_error(ws) == (1, KID_DW_GEMM * 16 + 5)
    # the dW GEMM then adds sample 1 alone, as the unpaired path does
    q = bg.problem_from(wl)
    ws1 = bg.alloc_workspace(q)
    dX1, dW1 = _buffers(wl)
    _sample(bg, q, 1, inp, ws1, dX1, dW1)
    assert bg.get_device_error(ws1) == (0, 0)
    assert torch.equal(dX, dX1)
    assert normwise(to64(dW), to64(dW1)) <= ORDER_TOL and float(dW1.abs().max()) > 0.0


def test_clearing_the_error_word_forgets_a_pending_sample(bg):
    wl = CONFIGS["tiny"]
    inp = make_inputs(wl, device="cuda")
    p = bg.problem_from(wl, pair_dw=True)
    ws = bg.alloc_workspace(p)
    dX, dW = _buffers(wl)
    _sample(bg, p, 0, inp, ws, dX, dW)
    bg.clear_device_error(ws)
    bg.sample_mask(p, 2, ws)                 # nothing pending any more: no error
    assert bg.get_device_error(ws) == (0, 0)


def test_masking_a_sample_twice_keeps_the_pairing(bg):
    """An old-policy pass that masks sample j again (same draws) between the
    two calls of a pair does not break the pairing: same dW bits."""
    import torch
    wl = CONFIGS["ragged"].with_(n_t=4)
    inp = make_inputs(wl, device="cuda")
    p = bg.problem_from(wl, pair_dw=True)
    outs = []
    for remask in (False, True):
        ws = bg.alloc_workspace(p)
        dX, dW = _buffers(wl)
        for j in range(wl.n_t):
            _sample(bg, p, j, inp, ws, dX, dW, remask=remask)
        assert bg.get_device_error(ws) == (0, 0)
        outs.append((dX, dW))
    assert torch.equal(outs[0][0], outs[1][0]) and torch.equal(outs[0][1], outs[1][1])


def test_repeated_backward_adds_what_the_unpaired_path_adds(bg):
    """Backward calls 0, 1, 1: the second call of sample 1 adds sample 1's dW
    alone (its partner was added by the first), as the unpaired path does."""
    import torch
    wl = CONFIGS["ragged"].with_(n_t=4)
    inp = make_inputs(wl, device="cuda")
    outs = []
    for pair in (False, True):
        p = bg.problem_from(wl, pair_dw=pair)
        ws = bg.alloc_workspace(p)
        dX, dW = _buffers(wl)
        _sample(bg, p, 0, inp, ws, dX, dW)
        _sample(bg, p, 1, inp, ws, dX, dW)
        bg.elbo_bwd_accumulate(p, 1, inp["X"], inp["W"], inp["Y"],
                               torch.full((wl.B,), -0.25, device="cuda"), ws, dX, dW)
        assert bg.get_device_error(ws) == (0, 0)
        outs.append((dX, dW))
    assert torch.equal(outs[0][0], outs[1][0])
    assert normwise(to64(outs[1][1]), to64(outs[0][1])) <= ORDER_TOL
