"""GPU parity: the CUDA path through the C ABI against the fp64 oracle.

Tolerances (spec contract): masks bit-exact; per-sequence l within 1e-3
relative (|dl| <= 1e-3 max(|l|, 1)); accumulated dX, dW within 2e-2 normwise
relative; bound coefficients within 1e-5 relative of the oracle on identical
inputs (fp32 arithmetic of Eq. 10/13).
"""
import numpy as np
import pytest

from oracle import bgpo_oracle as O
from synth import CONFIGS, make_inputs
from tests.harness import (ensure_built, gpu_run, normwise, oracle_run, record_margin, rel_ell_err,
                           to64)

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


def _inputs(name, **over):
    wl = CONFIGS[name].with_(**over) if over else CONFIGS[name]
    return wl, make_inputs(wl, device="cuda")


@pytest.fixture(scope="module")
def runs(bg):
    """GPU and oracle runs of the parity workloads (computed once per module)."""
    out = {}
    for name in ("tiny", "ragged", "ragged_strat"):
        wl, inp = _inputs(name)
        out[name] = (wl, inp, gpu_run(wl, inp), oracle_run(wl, {k: (v.cpu() if v is not None else None)
                                                                 for k, v in inp.items()}))
    return out


@pytest.mark.parametrize("name", ["tiny", "ragged", "ragged_strat"])
def test_masks_and_t_bit_exact(runs, name):
    wl, inp, g, o = runs[name]
    assert np.array_equal(g["masks"].cpu().numpy(), o["masks"])
    # t = T / D rounded once to float32 on both sides
    assert np.array_equal(g["t"].cpu().numpy(), o["ts"].astype(np.float32))


@pytest.mark.parametrize("name", ["tiny", "ragged", "ragged_strat"])
def test_elbo_matches_oracle(runs, name):
    wl, inp, g, o = runs[name]
    err = rel_ell_err(to64(g["ell_self"]), o["ell_self"])
    assert err.max() <= ELL_TOL, err.max()
    err = rel_ell_err(to64(g["ell"]), o["ell"])
    assert err.max() <= ELL_TOL, err.max()


@pytest.mark.parametrize("name", ["tiny", "ragged", "ragged_strat"])
def test_gradients_match_oracle(runs, name):
    wl, inp, g, o = runs[name]
    # the comparison means something only if the gradients are not all zero
    assert np.abs(o["dW"]).max() > 0 and np.abs(o["dX"]).max() > 0
    e_dw, e_dx = normwise(to64(g["dW"]), o["dW"]), normwise(to64(g["dX"]), o["dX"])
    record_margin(f"parity[{name}]", ell=float(rel_ell_err(to64(g["ell"]), o["ell"]).max()),
                  dX=e_dx, dW=e_dw)
    assert e_dw <= GRAD_TOL
    assert e_dx <= GRAD_TOL


@pytest.mark.parametrize("name", ["tiny", "ragged", "ragged_strat"])
def test_bound_values_match_oracle(runs, name):
    wl, inp, g, o = runs[name]
    # d is formed from each side's own l; with l_old = l_self + eps both give d = -eps
    assert np.allclose(to64(g["g"]), o["g"], rtol=2e-3, atol=1e-5)
    assert np.allclose(to64(g["coef"]), o["coef"], rtol=2e-3, atol=1e-6)


def test_group_advantage_matches_oracle(bg):
    import torch
    rng = np.random.default_rng(5)
    r = (rng.random(64) < 0.5).astype(np.float32)
    r[:8] = 1.0   # a zero-std group
    p = bg.problem(64, 1, 1, 64, 8, 1, 8)
    A = torch.empty(64, dtype=torch.float32, device="cuda")
    bg.group_advantage(p, torch.from_numpy(r).cuda(), A)
    ref = O.group_advantage(r.astype(np.float64), 8)
    assert np.allclose(A.cpu().numpy(), ref, rtol=1e-5, atol=1e-6)
    assert np.array_equal(A[:8].cpu().numpy(), np.zeros(8, dtype=np.float32))


def test_bound_coeffs_on_identical_inputs(bg):
    import torch
    rng = np.random.default_rng(7)
    B, n_t = 300, 16
    p = bg.problem(B, 1, 1, 64, 8, n_t, 8)
    ws = bg.alloc_workspace(p)
    bg.clear_device_error(ws)
    bg.sample_mask(p, 3, ws)
    ell = rng.standard_normal(B).astype(np.float32) * 50
    ell_old = (ell + rng.standard_normal(B).astype(np.float32) * 0.5).astype(np.float32)
    A = rng.standard_normal(B).astype(np.float32)
    A[:5] = 0.0
    cuda = lambda a: torch.from_numpy(a).cuda()
    coef = torch.empty(B, device="cuda")
    gg = torch.empty(B, device="cuda")
    bg.bound_coeffs(p, 3, cuda(ell), cuda(ell_old), cuda(A), coef, gg, ws)
    _, g_ref, c_ref = O.bound_coeffs(ell.astype(np.float64), ell_old.astype(np.float64),
                                     A.astype(np.float64), n_t, 1.0 / 8)
    assert np.allclose(coef.cpu().numpy(), c_ref, rtol=1e-5, atol=1e-9)
    assert np.allclose(gg.cpu().numpy(), g_ref, rtol=1e-5, atol=1e-7)
    assert bg.get_device_error(ws) == (0, 0)


def test_backward_with_oracle_coefficients(bg):
    """K6 isolated: oracle coefficients fed in, one sample, compared with the oracle."""
    import torch
    wl, inp = _inputs("ragged")
    p = bg.problem_from(wl)
    ws = bg.alloc_workspace(p)
    bg.clear_device_error(ws)
    rng = np.random.default_rng(3)
    coef = rng.standard_normal(wl.B).astype(np.float64) * 0.3
    ell = torch.empty(wl.B, device="cuda")
    dX = torch.zeros((wl.B, wl.R, wl.H), device="cuda")
    dW = torch.zeros((wl.V, wl.H), device="cuda")
    j = 1
    bg.sample_mask(p, j, ws)
    bg.elbo_fwd(p, j, inp["X"], inp["W"], inp["Y"], ws, ell)
    bg.elbo_bwd_accumulate(p, j, inp["X"], inp["W"], inp["Y"],
                           torch.from_numpy(coef.astype(np.float32)).cuda(), ws, dX, dW)
    _, _, t, mask = O.sample_t_mask(wl.seed, wl.B, wl.R, j, wl.n_t, wl.t_mode)
    gx, gw = O.elbo_term_grads(to64(inp["X"]), to64(inp["W"]), to64(inp["Y"]), wl.P, mask, t,
                               coef.astype(np.float32).astype(np.float64))
    assert normwise(to64(dW), gw) <= GRAD_TOL
    assert normwise(to64(dX), gx) <= GRAD_TOL
    assert bg.get_device_error(ws) == (0, 0)


def test_forward_is_deterministic(bg):
    import torch
    wl, inp = _inputs("ragged")
    p = bg.problem_from(wl)
    ws = bg.alloc_workspace(p)
    a = torch.empty(wl.B, device="cuda")
    b = torch.empty(wl.B, device="cuda")
    for out in (a, b):
        bg.sample_mask(p, 2, ws)
        bg.elbo_fwd(p, 2, inp["X"], inp["W"], inp["Y"], ws, out)
    assert torch.equal(a, b)


def test_on_policy_equivalence_on_gpu(bg):
    """Sec. 3.2 on the device: d = 0 exactly, g n_t = A and coef = -A / (G n_t)."""
    import torch
    wl, inp = _inputs("ragged", eps_std=0.0)
    g = gpu_run(wl, inp)
    ell, ell_old = g["ell"].cpu().numpy(), g["ell_old"].cpu().numpy()
    assert np.array_equal(ell, ell_old)
    A = g["A"].cpu().numpy()
    assert np.allclose(g["g"].cpu().numpy() * wl.n_t, A[:, None], rtol=1e-6, atol=1e-7)
    assert np.allclose(g["coef"].cpu().numpy(), -A[:, None] / (wl.G * wl.n_t), rtol=1e-6, atol=1e-9)


def test_dw_rows_sum_to_zero(runs):
    """sum_v dz_{r,v} = 0 up to the bf16 rounding of dz: |sum_v dW| << |dW|."""
    for name in ("tiny", "ragged"):
        wl, inp, g, o = runs[name]
        dW = to64(g["dW"])
        col = np.abs(dW.sum(axis=0)).max()
        assert col <= 1e-2 * np.abs(dW).sum(axis=0).max()


def test_resume_at_sample_is_bit_identical(bg):
    import torch
    wl, inp = _inputs("tiny")
    p = bg.problem_from(wl)
    ws = bg.alloc_workspace(p)
    full = []
    for j in range(wl.n_t):
        m = torch.empty((wl.B, wl.R), dtype=torch.uint8, device="cuda")
        bg.sample_mask(p, j, ws, None, m)
        full.append(m)
    m2 = torch.empty((wl.B, wl.R), dtype=torch.uint8, device="cuda")
    bg.sample_mask(p, 2, ws, None, m2)
    assert torch.equal(full[2], m2)


def test_empty_masks_give_zero(bg):
    """R = 1 with small t: samples whose mask is empty give l = 0 and no gradient."""
    import torch
    wl = CONFIGS["tiny"].with_(B=1, R=1, n_t=64, P=3)
    inp = make_inputs(wl, device="cuda")
    p = bg.problem_from(wl)
    ws = bg.alloc_workspace(p)
    _, masks = O.sample_masks(wl.seed, 1, 1, wl.n_t, wl.t_mode)
    empty_j = [j for j in range(wl.n_t) if masks[j].sum() == 0]
    assert empty_j, "no empty sample drawn"
    dX = torch.zeros((1, 1, wl.H), device="cuda")
    dW = torch.zeros((wl.V, wl.H), device="cuda")
    ell = torch.full((1,), 7.0, device="cuda")
    coef = torch.ones(1, device="cuda")
    j = empty_j[0]
    bg.sample_mask(p, j, ws)
    bg.elbo_fwd(p, j, inp["X"], inp["W"], inp["Y"], ws, ell)
    bg.elbo_bwd_accumulate(p, j, inp["X"], inp["W"], inp["Y"], coef, ws, dX, dW)
    torch.cuda.synchronize()
    assert float(ell[0]) == 0.0
    assert float(dW.abs().max()) == 0.0 and float(dX.abs().max()) == 0.0


def test_all_rows_masked(bg):
    """Stratified t close to 1 masks (nearly) every row: M = B * R edge."""
    import torch
    wl = CONFIGS["ragged"].with_(t_mode=1, n_t=64, R=40)
    inp = make_inputs(wl, device="cuda")
    p = bg.problem_from(wl)
    ws = bg.alloc_workspace(p)
    j = 63
    _, _, t, mask = O.sample_t_mask(wl.seed, wl.B, wl.R, j, wl.n_t, wl.t_mode)
    ell = torch.empty(wl.B, device="cuda")
    bg.sample_mask(p, j, ws)
    bg.elbo_fwd(p, j, inp["X"], inp["W"], inp["Y"], ws, ell)
    ref = O.elbo_term(to64(inp["X"]), to64(inp["W"]), to64(inp["Y"]), wl.P, mask, t)
    assert mask.mean() > 0.9
    assert rel_ell_err(ell.cpu().numpy(), ref).max() <= ELL_TOL


def test_stale_sample_sets_device_error(bg):
    import torch
    wl, inp = _inputs("tiny")
    p = bg.problem_from(wl)
    ws = bg.alloc_workspace(p)
    bg.clear_device_error(ws)
    bg.sample_mask(p, 0, ws)
    ell = torch.empty(wl.B, device="cuda")
    bg.elbo_fwd(p, 1, inp["X"], inp["W"], inp["Y"], ws, ell)   # workspace holds sample 0
    code, where = bg.get_device_error(ws)
    assert code == 1
    assert float(ell.abs().max()) == 0.0
    bg.clear_device_error(ws)
    assert bg.get_device_error(ws) == (0, 0)


def test_nonfinite_coefficient_sets_device_error(bg):
    import torch
    p = bg.problem(4, 1, 1, 64, 8, 2, 2)
    ws = bg.alloc_workspace(p)
    bg.clear_device_error(ws)
    ell = torch.tensor([1.0, 2.0, 500.0, 0.0], device="cuda")
    old = torch.zeros(4, device="cuda")
    A = torch.tensor([1.0, -1.0, -1.0, 1.0], device="cuda")   # e^500 overflows fp32
    coef = torch.empty(4, device="cuda")
    bg.bound_coeffs(p, 0, ell, old, A, coef, None, ws)
    assert bg.get_device_error(ws)[0] == 5


def test_trace_records_every_kernel(bg):
    import torch
    wl, inp = _inputs("tiny")
    tr = bg.Trace(64)
    p = bg.problem_from(wl, trace=tr)
    ws = bg.alloc_workspace(p)
    ell = torch.empty(wl.B, device="cuda")
    coef = torch.zeros(wl.B, device="cuda")
    dX = torch.zeros((wl.B, wl.R, wl.H), device="cuda")
    dW = torch.zeros((wl.V, wl.H), device="cuda")
    bg.sample_mask(p, 0, ws)
    bg.elbo_fwd(p, 0, inp["X"], inp["W"], inp["Y"], ws, ell)
    bg.bound_coeffs(p, 0, ell, ell, inp["A"], coef, None, ws)
    bg.elbo_bwd_accumulate(p, 0, inp["X"], inp["W"], inp["Y"], coef, ws, dX, dW)
    names = [n for n, ms in tr.records()]
    assert names == ["mask_compact", "gather_rows", "lmhead_fwd_lse", "lse_combine", "seq_reduce",
                     "bound_coeffs", "xm_transpose", "lmhead_dz", "dx_gemm", "dx_reduce", "dw_gemm"]
    assert all(ms >= 0 for _, ms in tr.records())
    tr.close()
    # the backward over two vocabulary chunks of 256 columns: each chunk's dZ,
    # dX and dW GEMMs, then one split reduction of dX
    tr = bg.Trace(64)
    p = bg.problem_from(wl, trace=tr, vocab_chunk=256)
    ws = bg.alloc_workspace(p)
    bg.sample_mask(p, 0, ws)
    bg.elbo_fwd(p, 0, inp["X"], inp["W"], inp["Y"], ws, ell)
    bg.elbo_bwd_accumulate(p, 0, inp["X"], inp["W"], inp["Y"], coef, ws, dX, dW)
    assert [n for n, ms in tr.records()][5:] == ["xm_transpose"] + 2 * ["lmhead_dz", "dx_gemm",
                                                                        "dw_gemm"] + ["dx_reduce"]
    assert bg.get_device_error(ws) == (0, 0)
    tr.close()
    # with BGPO_FLAG_KEEP_LOGITS the backward reads the logits the forward kept
    tr = bg.Trace(64)
    p = bg.problem_from(wl, trace=tr, keep_logits=True)
    ws = bg.alloc_workspace(p)
    bg.sample_mask(p, 0, ws)
    bg.elbo_fwd(p, 0, inp["X"], inp["W"], inp["Y"], ws, ell)
    bg.elbo_bwd_accumulate(p, 0, inp["X"], inp["W"], inp["Y"], coef, ws, dX, dW)
    assert [n for n, ms in tr.records()][-5:] == ["xm_transpose", "dz_from_logits", "dx_gemm",
                                                  "dx_reduce", "dw_gemm"]
    assert bg.get_device_error(ws) == (0, 0)
    tr.close()


@pytest.mark.parametrize("name", ["tiny", "ragged", "ragged_strat"])
def test_kept_and_recomputed_logits_give_identical_bits(bg, runs, name):
    # the forward's kept fp32 logits equal the backward GEMM's recomputed ones
    # (same tiles, same K order) and dz is formed by the same arithmetic, so the
    # two modes agree bit for bit; both agree with the oracle (test above)
    import torch
    wl, inp, g, _ = runs[name]
    r = gpu_run(wl, inp, keep_logits=True)
    assert torch.equal(r["ell"], g["ell"])
    assert torch.equal(r["dW"], g["dW"])
    assert torch.equal(r["dX"], g["dX"])
    assert bg.get_device_error(r["ws"]) == (0, 0) and bg.get_device_error(g["ws"]) == (0, 0)


def test_backward_without_kept_logits_is_refused(bg):
    # the last forward of the sample kept no logits: the backward records
    # BGPO_ERR_INVALID_ARG and leaves dX and dW untouched
    import torch
    wl, inp = _inputs("ragged")
    keep = bg.problem_from(wl, keep_logits=True)
    lean = bg.problem_from(wl)
    ws = bg.alloc_workspace(keep)
    ell = torch.empty(wl.B, device="cuda")
    coef = torch.full((wl.B,), -0.5, device="cuda")
    dX = torch.zeros((wl.B, wl.R, wl.H), device="cuda")
    dW = torch.zeros((wl.V, wl.H), device="cuda")
    bg.sample_mask(keep, 1, ws)
    bg.elbo_fwd(keep, 1, inp["X"], inp["W"], inp["Y"], ws, ell)
    bg.elbo_fwd(lean, 1, inp["X"], inp["W"], inp["Y"], ws, ell)     # overrides: no logits kept
    bg.elbo_bwd_accumulate(keep, 1, inp["X"], inp["W"], inp["Y"], coef, ws, dX, dW)
    code, where = bg.get_device_error(ws)
    assert code == 1 and where == 13 * 16 + 2
    assert float(dX.abs().max()) == 0.0 and float(dW.abs().max()) == 0.0
    # a fresh sample that keeps its logits runs normally again
    bg.clear_device_error(ws)
    bg.sample_mask(keep, 2, ws)
    bg.elbo_fwd(keep, 2, inp["X"], inp["W"], inp["Y"], ws, ell)
    bg.elbo_bwd_accumulate(keep, 2, inp["X"], inp["W"], inp["Y"], coef, ws, dX, dW)
    assert bg.get_device_error(ws) == (0, 0)
    assert float(dW.abs().max()) > 0.0


@pytest.mark.parametrize("pair", [False, True])
def test_sequence_shards_reproduce_the_full_batch(bg, pair):
    """Data-parallel decomposition on one device: two shards with b_offset give
    the whole batch's draws and l, and their dW sum to the whole batch's dW
    (with and without dW pairing inside each shard)."""
    import torch
    # two groups of 3 Bernoulli rewards (both mixed at this seed): each shard
    # normalises its own group (Eq. 18)
    wl = CONFIGS["ragged"].with_(B=6, G=3, advantages="bernoulli")
    inp = make_inputs(wl, device="cuda")
    full = gpu_run(wl, inp)
    assert float(full["dW"].abs().max()) > 0
    half = wl.with_(B=3)
    parts = []
    for k in range(2):
        sl = slice(3 * k, 3 * k + 3)
        sub = {"X": inp["X"][sl].contiguous(), "W": inp["W"], "Y": inp["Y"][sl].contiguous(),
               "A": None, "rewards": inp["rewards"][sl].contiguous(),
               "eps": inp["eps"][sl].contiguous()}
        parts.append(gpu_run(half, sub, b_offset=3 * k, pair_dw=pair))
    assert torch.equal(torch.cat([p["masks"] for p in parts], dim=1), full["masks"])
    ell = torch.cat([p["ell"] for p in parts])
    assert torch.allclose(ell, full["ell"], rtol=1e-6, atol=1e-6)
    dW = parts[0]["dW"] + parts[1]["dW"]
    assert normwise(to64(dW), to64(full["dW"])) <= 1e-5
    dX = torch.cat([p["dX"] for p in parts])
    assert normwise(to64(dX), to64(full["dX"])) <= 1e-5


def test_bounded_wait_times_out_and_context_survives(bg):
    """Failure detection on the device: a wait on a barrier nothing arrives at
    gives up after its limit, the error word says BGPO_ERR_TIMEOUT, and the
    next call on the same context works."""
    import torch
    wl, inp = _inputs("tiny")
    p = bg.problem_from(wl)
    ws = bg.alloc_workspace(p)
    bg.clear_device_error(ws)
    bg.selftest_bounded_wait(ws, timeout_us=5000)
    code, where = bg.get_device_error(ws)
    assert code == 8 and where == 11 * 16
    bg.clear_device_error(ws)
    ell = torch.empty(wl.B, device="cuda")
    bg.sample_mask(p, 0, ws)
    bg.elbo_fwd(p, 0, inp["X"], inp["W"], inp["Y"], ws, ell)
    torch.cuda.synchronize()
    assert bg.get_device_error(ws) == (0, 0)
    assert torch.isfinite(ell).all()


@pytest.mark.parametrize("keep,pair", [(False, False), (True, False), (False, True)])
def test_variable_length_responses(bg, keep, pair):
    """Padded batches: positions at or past resp_len[b] are never masked and get
    no gradient; everything else matches the oracle on the same draws (both
    logit modes, and with dW pairing)."""
    wl = CONFIGS["ragged"]
    inp = make_inputs(wl, device="cuda")
    lens = np.array([301, 0, 117])
    g = gpu_run(wl, inp, resp_len=lens, keep_logits=keep, pair_dw=pair)
    o = oracle_run(wl, {k: (v.cpu() if v is not None else None) for k, v in inp.items()},
                   resp_len=lens)
    assert np.array_equal(g["masks"].cpu().numpy(), o["masks"])
    assert not g["masks"][:, 1].any() and not g["masks"][:, 2, 117:].any()
    assert rel_ell_err(to64(g["ell"]), o["ell"]).max() <= ELL_TOL
    assert np.array_equal(to64(g["ell"])[1], np.zeros(wl.n_t))
    assert np.abs(o["dW"]).max() > 0
    assert normwise(to64(g["dW"]), o["dW"]) <= GRAD_TOL
    assert normwise(to64(g["dX"]), o["dX"]) <= GRAD_TOL
    assert float(g["dX"][2, 117:].abs().max()) == 0.0


@pytest.mark.parametrize("keep,pair,chunk", [(False, False, 0), (True, False, 0), (False, True, 0),
                                             (True, True, 0), (False, False, 256),
                                             (True, True, 256)])
def test_whole_step_replays_from_a_cuda_graph(bg, keep, pair, chunk):
    # the n_t loop allocates nothing, never synchronises and keeps M (and the
    # dW pairing state) on the device, so one step captures into a CUDA graph;
    # a replay gives the bits of the eager step (also over vocabulary chunks)
    import torch
    wl, inp = _inputs("ragged")
    p = bg.problem_from(wl, keep_logits=keep, pair_dw=pair, vocab_chunk=chunk)
    X, W, Y = inp["X"], inp["W"], inp["Y"]
    ws = bg.alloc_workspace(p)
    A = inp["A"].contiguous()
    ell_old = torch.empty((wl.n_t, wl.B), device="cuda")
    for j in range(wl.n_t):
        bg.sample_mask(p, j, ws)
        bg.elbo_fwd(p, j, X, W, Y, ws, ell_old[j])
    ell_old += inp["eps"].T

    def step(out):
        for j in range(wl.n_t):
            bg.sample_mask(p, j, ws)
            bg.elbo_fwd(p, j, X, W, Y, ws, out["ell"][j])
            bg.bound_coeffs(p, j, out["ell"][j], ell_old[j], A, out["coef"][j], None, ws)
            bg.elbo_bwd_accumulate(p, j, X, W, Y, out["coef"][j], ws, out["dX"], out["dW"])

    def buffers():
        return dict(ell=torch.empty((wl.n_t, wl.B), device="cuda"),
                    coef=torch.empty((wl.n_t, wl.B), device="cuda"),
                    dX=torch.zeros((wl.B, wl.R, wl.H), device="cuda"),
                    dW=torch.zeros((wl.V, wl.H), device="cuda"))

    eager = buffers()
    step(eager)
    torch.cuda.synchronize()
    graphed = buffers()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        step(graphed)
    graphed["dX"].zero_()
    graphed["dW"].zero_()
    graph.replay()
    torch.cuda.synchronize()
    assert bg.get_device_error(ws) == (0, 0)
    for k in ("ell", "coef", "dX", "dW"):
        assert torch.equal(graphed[k], eager[k]), k


@pytest.mark.parametrize("shape", [
    dict(B=1, P=0, R=1, H=64, V=1, n_t=1, G=1),      # one token, one-word vocabulary: l = 0
    dict(B=2, P=0, R=5, H=64, V=2, n_t=1, G=2),      # no prompt, two-word vocabulary
    dict(B=3, P=0, R=70, H=128, V=65, n_t=2, G=3),   # V one past a 64-column boundary
])
def test_degenerate_shapes_match_oracle(bg, shape):
    import torch
    wl = CONFIGS["tiny"].with_(name="degenerate", seed=77, **shape)
    inp_cpu = make_inputs(wl)
    inp = {k: (v.cuda() if v is not None else None) for k, v in inp_cpu.items()}
    g = gpu_run(wl, inp)
    o = oracle_run(wl, inp_cpu)
    assert bg.get_device_error(g["ws"]) == (0, 0)
    assert np.array_equal(g["masks"].cpu().numpy(), o["masks"])
    assert rel_ell_err(to64(g["ell"]), o["ell"]).max() <= ELL_TOL
    # (with V = 1 the oracle's l and gradients are exactly zero; normwise then
    # measures the absolute size of what the GPU returns)
    assert normwise(to64(g["dX"]), o["dX"]) <= GRAD_TOL
    assert normwise(to64(g["dW"]), o["dW"]) <= GRAD_TOL
    if wl.V == 1:
        assert float(g["ell"].abs().max()) <= 1e-4


@pytest.mark.parametrize("pair", [False, True])
def test_peak_device_memory_flat_in_n_t(bg, pair):
    # Linearity (Sec. 3): one sample's state at a time (two with dW pairing), so
    # the device memory a step needs does not grow with n_t; only the caller's
    # [n_t, B] vectors do
    import torch
    peaks = {}
    for n_t in (1, 4, 16):
        wl = CONFIGS["ragged"].with_(n_t=n_t)
        inp = make_inputs(wl, device="cuda")     # same X, W, Y for every n_t (same seed)
        torch.cuda.synchronize()
        torch.cuda.empty_cache()
        torch.cuda.reset_peak_memory_stats()
        base = torch.cuda.memory_allocated()
        g = gpu_run(wl, inp, pair_dw=pair)
        assert bg.get_device_error(g["ws"]) == (0, 0)
        peaks[n_t] = torch.cuda.max_memory_allocated() - base
        del g, inp
    vectors = 16 * 4 * wl.B * 8          # [n_t, B] float vectors of the harness, generously
    assert peaks[16] - peaks[1] <= vectors + (1 << 20), peaks


@pytest.mark.parametrize("H", [72, 200, 328, 768, 1000])
def test_hidden_sizes_not_a_multiple_of_64(bg, H):
    """H a multiple of 8 only: the forward and dZ GEMMs end on a partial K
    block (read as zeros), the dX and dW GEMMs on a partial hidden-size tile
    and 32-column sub-tile (8 columns of H = 200, 72 and 328), the transpose
    on a partial 64-column tile; with and without vocabulary chunks and dW
    pairing. The dX GEMM's tiles are two 256-column blocks of H wide: H = 768
    has an odd number of blocks (the last tile's second block lies wholly past
    H), H = 1000 ends inside the last tile's second block."""
    wl = CONFIGS["ragged"].with_(name="odd_hidden", H=H, seed=90 + H)
    inp_cpu = make_inputs(wl)
    inp = {k: (v.cuda() if v is not None else None) for k, v in inp_cpu.items()}
    o = oracle_run(wl, inp_cpu)
    for kw in (dict(), dict(vocab_chunk=256), dict(pair_dw=True), dict(keep_logits=True)):
        g = gpu_run(wl, inp, **kw)
        assert bg.get_device_error(g["ws"]) == (0, 0), kw
        assert np.array_equal(g["masks"].cpu().numpy(), o["masks"])
        e_ell = float(rel_ell_err(to64(g["ell"]), o["ell"]).max())
        e_dx, e_dw = normwise(to64(g["dX"]), o["dX"]), normwise(to64(g["dW"]), o["dW"])
        record_margin(f"hidden_size[{H},{sorted(kw)}]", ell=e_ell, dX=e_dx, dW=e_dw)
        assert e_ell <= ELL_TOL, kw
        assert e_dx <= GRAD_TOL, kw
        assert e_dw <= GRAD_TOL, kw


def test_row_groups_of_the_forward_and_dz_gemms(bg):
    """H = 16384, so that a sample of about 3,000 masked rows holds about
    100 MB of gathered rows Xm: the forward and dZ GEMMs walk its row blocks in
    groups (more than 52 MB of Xm: groups of at most 40 MB), the other sample
    stays in one group. Every l, all of dX and dW against the oracle, with the
    default flags, dW pairing and kept logits."""
    wl = CONFIGS["ragged_strat"].with_(name="row_groups", B=4, P=3, R=1001, H=16384, V=1000,
                                       n_t=2, G=4, seed=77)
    inp_cpu = make_inputs(wl)
    inp = {k: (v.cuda() if v is not None else None) for k, v in inp_cpu.items()}
    o = oracle_run(wl, inp_cpu)
    rows = o["masks"].reshape(wl.n_t, -1).sum(axis=1)
    xm_bytes = [-(-int(m) // 256) * 256 * wl.H * 2 for m in rows]
    assert max(xm_bytes) > 52 << 20 >= min(xm_bytes), rows    # grouped and ungrouped samples
    for kw in (dict(), dict(pair_dw=True), dict(keep_logits=True)):
        g = gpu_run(wl, inp, **kw)
        assert bg.get_device_error(g["ws"]) == (0, 0), kw
        assert np.array_equal(g["masks"].cpu().numpy(), o["masks"])
        e_ell = float(rel_ell_err(to64(g["ell"]), o["ell"]).max())
        e_dx, e_dw = normwise(to64(g["dX"]), o["dX"]), normwise(to64(g["dW"]), o["dW"])
        record_margin(f"row_groups[{sorted(kw)}]", ell=e_ell, dX=e_dx, dW=e_dw,
                      masked_rows=int(max(rows)))
        assert e_ell <= ELL_TOL, kw
        assert e_dx <= GRAD_TOL, kw
        assert e_dw <= GRAD_TOL, kw
