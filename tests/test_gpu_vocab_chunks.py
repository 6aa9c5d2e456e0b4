"""The backward walks the vocabulary in chunks (bgpo_problem.vocab_chunk).

The gradient of Eq. 4 is a sum over vocabulary entries as well as over masked
rows, so the backward forms dL/dz for one chunk of the vocabulary, adds that
chunk's terms to dX (dX += dZ_c W_c) and its rows of dW (dW[c] += dZ_c^T Xm),
and moves on: the dL/dz buffer holds roundup(B R, 256) x chunk values instead
of the whole vocabulary's. These tests run the parity workloads with chunks of
256 columns (the narrowest: 2 to 4 chunks, ragged last chunks of 232 and 9
columns, the latter allowing no split of the dX GEMM) and compare them with the
oracle and with the whole vocabulary at once: l and dW the same bits, dX the
same sum up to fp32 order; with the logits kept; with dW pairing walking the
same chunks, the same dX bits as without pairing.
"""
import numpy as np
import pytest

from synth import CONFIGS, make_inputs
from tests.harness import ensure_built, gpu_run, normwise, oracle_run, record_margin, rel_ell_err, to64

pytestmark = pytest.mark.gpu

WHOLE = 1 << 24     # a chunk at least as wide as any vocabulary: no chunking
ORDER_TOL = 1e-5
# the same at the full LLaDA-8B head: fp32 order over a 126,464-long K whose
# terms mostly cancel
VOCAB_ORDER_TOL = 1e-4


@pytest.fixture(scope="module")
def bg():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    ensure_built()
    import paper_2510_11683_gb300 as bg
    return bg


@pytest.mark.parametrize("keep", [False, True])
@pytest.mark.parametrize("name,chunk", [("tiny", 256), ("ragged", 256), ("ragged", 512),
                                        ("ragged_strat", 256)])
def test_chunked_backward_matches_oracle_and_whole_vocabulary(bg, name, chunk, keep):
    import torch
    wl = CONFIGS[name]
    inp = make_inputs(wl, device="cuda")
    c = gpu_run(wl, inp, keep_logits=keep, vocab_chunk=chunk)
    w = gpu_run(wl, inp, keep_logits=keep, vocab_chunk=WHOLE)
    assert bg.get_device_error(c["ws"]) == (0, 0) and bg.get_device_error(w["ws"]) == (0, 0)
    assert c["ws"].numel() < w["ws"].numel()
    assert torch.equal(c["ell"], w["ell"])
    assert torch.equal(c["dW"], w["dW"])           # dW rows of a chunk: the same tiles
    assert normwise(to64(c["dX"]), to64(w["dX"])) <= ORDER_TOL
    o = oracle_run(wl, {k: (v.cpu() if v is not None else None) for k, v in inp.items()})
    assert np.array_equal(c["masks"].cpu().numpy(), o["masks"])
    e_ell = rel_ell_err(to64(c["ell"]), o["ell"]).max()
    e_dx, e_dw = normwise(to64(c["dX"]), o["dX"]), normwise(to64(c["dW"]), o["dW"])
    assert e_ell <= 1e-3 and e_dx <= 2e-2 and e_dw <= 2e-2
    record_margin(f"vocab_chunks[{name},{chunk},keep={keep}]", ell=e_ell, dX=e_dx, dW=e_dw)


@pytest.mark.parametrize("name", ["tiny", "ragged", "ragged_strat"])
def test_paired_backward_over_the_same_chunks_gives_the_same_dx_bits(bg, name):
    import torch
    wl = CONFIGS[name]
    inp = make_inputs(wl, device="cuda")
    a = gpu_run(wl, inp, vocab_chunk=256)
    p = gpu_run(wl, inp, pair_dw=True, vocab_chunk=256)
    assert bg.get_device_error(a["ws"]) == (0, 0) and bg.get_device_error(p["ws"]) == (0, 0)
    assert torch.equal(p["ell"], a["ell"]) and torch.equal(p["dX"], a["dX"])
    assert normwise(to64(p["dW"]), to64(a["dW"])) <= ORDER_TOL


def test_default_chunks_at_the_full_head(bg):
    """The LLaDA-8B head (V = 126464) runs 4 chunks of 31,744 columns by
    default once the batch's whole-vocabulary dL/dz would exceed 1 GiB (16 x
    512 responses); here the same chunks on a batch with few masked rows: the
    whole dX and dW against the oracle, and against the whole vocabulary at
    once (this batch's default)."""
    import torch
    from tests.harness import default_vocab_chunk
    wl = CONFIGS["llada8b_r256"].with_(B=2, P=8, R=24, n_t=3, G=2)
    assert default_vocab_chunk(wl.V, 16 * 512) == 31744 and default_vocab_chunk(wl.V, 48) == 0
    inp_cpu = make_inputs(wl)
    inp = {k: (v.cuda() if v is not None else None) for k, v in inp_cpu.items()}
    c = gpu_run(wl, inp, vocab_chunk=31744)
    assert bg.get_device_error(c["ws"]) == (0, 0)
    res = {k: c[k].cpu() for k in ("masks", "ell", "dX", "dW")}
    del c
    w = gpu_run(wl, inp, vocab_chunk=WHOLE)
    assert torch.equal(res["ell"], w["ell"].cpu()) and torch.equal(res["dW"], w["dW"].cpu())
    assert normwise(to64(res["dX"]), to64(w["dX"])) <= VOCAB_ORDER_TOL
    del w
    torch.cuda.empty_cache()
    o = oracle_run(wl, inp_cpu)
    assert np.array_equal(res["masks"].numpy(), o["masks"])
    assert normwise(to64(res["dW"]), o["dW"]) <= 2e-2
    assert normwise(to64(res["dX"]), o["dX"]) <= 2e-2
