"""GPU parity at the size limits the C ABI accepts, one dimension at a time.

  * V = 2^24 - 1000 (just under the largest vocabulary, ragged against every
    tile width): 65,532 vocabulary tiles in the forward GEMM, 512 vocabulary
    chunks of 32,768 columns in the backward by default, and with
    BGPO_FLAG_PAIR_DW one whole-vocabulary chunk (a 2^24-long K loop in the dX
    GEMM, 65,532 vocabulary tiles in the dW GEMM); 64-bit offsets into dZ and
    the kept logits, and into the paired dZ rows;
  * B * R = 2^22 (the most response positions): the single-CTA mask compaction
    walks 2^20 Philox blocks, about 2^21 masked rows per sample;
  * H = 16384 (the largest hidden size): 64 hidden-size tiles, 256 K blocks per
    forward tile.

Each case is checked against the fp64 oracle on the same seeded inputs: masks
bit-exact, l within 1e-3 relative, dX and dW within 2e-2 normwise.
"""
import numpy as np
import pytest

from oracle import bgpo_oracle as O
from synth import CONFIGS, make_inputs
from tests.harness import (default_vocab_chunk, ensure_built, gpu_run, normwise, oracle_run,
                           record_margin, rel_ell_err, to64)

pytestmark = pytest.mark.gpu

ELL_TOL = 1e-3
GRAD_TOL = 2e-2


@pytest.fixture(scope="module")
def bg():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    ensure_built()
    import paper_2510_11683_gb300 as bg
    return bg


def _check(wl, g, o, label=""):
    assert np.array_equal(g["masks"].cpu().numpy(), o["masks"])
    assert np.array_equal(g["t"].cpu().numpy(), o["ts"].astype(np.float32))
    err = rel_ell_err(to64(g["ell"]), o["ell"])
    e_dx, e_dw = normwise(to64(g["dX"]), o["dX"]), normwise(to64(g["dW"]), o["dW"])
    record_margin(f"limits[{wl.name}{label}]", ell=float(err.max()), dX=e_dx, dW=e_dw)
    assert err.max() <= ELL_TOL, err.max()
    assert e_dx <= GRAD_TOL
    assert e_dw <= GRAD_TOL


def test_largest_vocabulary(bg):
    import torch
    wl = CONFIGS["tiny"].with_(name="vocab_limit", B=2, P=3, R=40, H=64, V=(1 << 24) - 1000,
                               n_t=2, G=2, seed=41)
    inp_cpu = make_inputs(wl)
    inp = {k: (v.cuda() if v is not None else None) for k, v in inp_cpu.items()}
    g = gpu_run(wl, inp)
    assert bg.get_device_error(g["ws"]) == (0, 0)
    # the kept-logit mode indexes 4 * 256 * 2^24 bytes of logits: same bits
    k = gpu_run(wl, inp, keep_logits=True)
    assert bg.get_device_error(k["ws"]) == (0, 0)
    assert torch.equal(k["ell"], g["ell"]) and torch.equal(k["dX"], g["dX"])
    assert torch.equal(k["dW"], g["dW"])
    del k
    # dW pairing puts sample 1's dZ rows after sample 0's (64-bit row offsets
    # into a 2 * 256 x 2^24 bf16 region); walking the vocabulary in the same
    # 512 chunks as the unpaired backward: same l and dX bits, dW up to order
    q = gpu_run(wl, inp, pair_dw=True, vocab_chunk=default_vocab_chunk(wl.V))
    assert bg.get_device_error(q["ws"]) == (0, 0)
    assert torch.equal(q["ell"], g["ell"]) and torch.equal(q["dX"], g["dX"])
    assert normwise(to64(q["dW"]), to64(g["dW"])) <= 1e-5
    del q
    # the pairing's default: the whole vocabulary in one chunk, i.e. one dX
    # GEMM whose fp32 accumulator runs over K = 2^24 - 1000 vocabulary entries
    # (the chunked one sums 512 chunk results): both against the oracle
    q = gpu_run(wl, inp, pair_dw=True)
    assert bg.get_device_error(q["ws"]) == (0, 0)
    assert torch.equal(q["ell"], g["ell"])
    q = {key: q[key].cpu() for key in ("masks", "t", "ell", "dX", "dW")}
    g = {key: g[key].cpu() for key in ("masks", "t", "ell", "dX", "dW")}
    del inp
    torch.cuda.empty_cache()
    o = oracle_run(wl, inp_cpu)
    _check(wl, g, o)
    _check(wl, q, o)


def test_most_response_positions(bg):
    wl = CONFIGS["tiny"].with_(name="rows_limit", B=4096, P=1, R=1024, H=64, V=96, n_t=1, G=8,
                               seed=42)
    assert wl.B * wl.R == 1 << 22
    inp_cpu = make_inputs(wl)
    inp = {k: (v.cuda() if v is not None else None) for k, v in inp_cpu.items()}
    g = gpu_run(wl, inp)
    assert bg.get_device_error(g["ws"]) == (0, 0)
    o = oracle_run(wl, inp_cpu)
    assert o["masks"].sum() > (1 << 20)      # about half of the 2^22 positions
    _check(wl, g, o)


def test_largest_hidden_size(bg):
    wl = CONFIGS["tiny"].with_(name="hidden_limit", B=2, P=4, R=100, H=16384, V=1000, n_t=2,
                               G=2, seed=43)
    inp_cpu = make_inputs(wl)
    inp = {k: (v.cuda() if v is not None else None) for k, v in inp_cpu.items()}
    g = gpu_run(wl, inp)
    assert bg.get_device_error(g["ws"]) == (0, 0)
    o = oracle_run(wl, inp_cpu)
    _check(wl, g, o)
    # dW pairing at the widest Xm^T rows (64 hidden-size tiles of the dW GEMM)
    q = gpu_run(wl, inp, pair_dw=True)
    assert bg.get_device_error(q["ws"]) == (0, 0)
    _check(wl, q, o, ",pair")
