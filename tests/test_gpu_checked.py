"""The bounds-checked build (-DBGPO_CHECKED) on the GPU.

The library ships a build whose kernels test every index they read from device
memory (masked-row lists, segment offsets, row counts) and every target token
before use, recording BGPO_ERR_BOUNDS instead of touching memory out of bounds:
a memory checker built into the library, usable where no external one runs.
Here the parity workloads run through that build, in a child process that
loads it (BGPO_LIBRARY=checked): the error word must stay clear and the
results must match the oracle as the normal build's do, in both logit modes
and with the backward walking vocabulary chunks of 256 columns (with and
without dW pairing).
A target token outside the vocabulary, which the normal build cannot see (it
only ever compares targets, never indexes with them), must be reported.
"""
import json
import os
import subprocess
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from tests.harness import ensure_built  # noqa: E402

ELL_TOL = 1e-3
GRAD_TOL = 2e-2


def _child():
    import torch
    import paper_2510_11683_gb300 as bg
    from paper_2510_11683_gb300 import _lib
    from synth import CONFIGS, make_inputs
    from tests.harness import gpu_run, normwise, oracle_run, rel_ell_err, to64

    assert _lib.lib_path().endswith("libbgpo_checked.so")
    out = {"parity": {}}
    for name in ("tiny", "ragged", "ragged_strat"):
        wl = CONFIGS[name]
        inp_cpu = make_inputs(wl)
        inp = {k: (v.cuda() if v is not None else None) for k, v in inp_cpu.items()}
        g = gpu_run(wl, inp)
        k = gpu_run(wl, inp, keep_logits=True)
        # the backward over vocabulary chunks of 256 columns, unpaired and paired
        c = gpu_run(wl, inp, vocab_chunk=256)
        q = gpu_run(wl, inp, pair_dw=True, vocab_chunk=256)
        o = oracle_run(wl, inp_cpu)
        out["parity"][name] = {
            "errors": [bg.get_device_error(r["ws"]) for r in (g, k, c, q)],
            "chunked": [max(normwise(to64(r["dX"]), o["dX"]), normwise(to64(r["dW"]), o["dW"]))
                        for r in (c, q)],
            "masks": bool(np.array_equal(g["masks"].cpu().numpy(), o["masks"])),
            "ell": float(rel_ell_err(to64(g["ell"]), o["ell"]).max()),
            "dX": normwise(to64(g["dX"]), o["dX"]), "dW": normwise(to64(g["dW"]), o["dW"]),
            "keep_identical": bool(torch.equal(k["dX"], g["dX"]) and torch.equal(k["dW"], g["dW"])
                                   and torch.equal(k["ell"], g["ell"])),
        }
    wl = CONFIGS["tiny"]
    inp = make_inputs(wl, device="cuda")
    inp["Y"][0, :] = wl.V + 3                   # sequence 0's targets lie past the vocabulary
    g = gpu_run(wl, inp)
    out["bad_target"] = list(bg.get_device_error(g["ws"]))
    print(json.dumps(out))


@pytest.mark.gpu
def test_checked_build_runs_clean_and_reports_a_bad_target():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    ensure_built(checked=True)
    env = dict(os.environ, BGPO_LIBRARY="checked", PYTHONPATH=ROOT)
    r = subprocess.run([sys.executable, os.path.abspath(__file__)], env=env, cwd=ROOT,
                       capture_output=True, text=True, timeout=900)
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-4000:]
    res = json.loads(r.stdout.strip().splitlines()[-1])
    for name, p in res["parity"].items():
        assert p["errors"] == [[0, 0]] * 4, (name, p)
        assert max(p["chunked"]) <= GRAD_TOL, (name, p)
        assert p["masks"], name
        assert p["ell"] <= ELL_TOL, (name, p)
        assert p["dX"] <= GRAD_TOL and p["dW"] <= GRAD_TOL, (name, p)
        assert p["keep_identical"], name
    # BGPO_ERR_BOUNDS at the gather's target check (kernel id 1, site 11)
    assert res["bad_target"] == [9, 1 * 16 + 11]


if __name__ == "__main__":
    _child()
