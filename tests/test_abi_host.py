"""C-ABI library: loads, exports every declared symbol, validates on the host.

No GPU is needed: every call here either is host-only or fails validation
before any CUDA call (on a machine without a GPU, a valid launching call
returns BGPO_ERR_UNSUPPORTED_DEVICE instead of launching).
"""
import ctypes
import os
import re

import pytest

from tests.harness import ensure_built

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def L():
    ensure_built()
    from paper_2510_11683_gb300 import _lib
    return _lib.lib()


@pytest.fixture()
def bg():
    import paper_2510_11683_gb300 as bg
    return bg


def _declared_functions():
    src = open(os.path.join(ROOT, "include", "bgpo.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    names = re.findall(r"\b(bgpo_[a-z_0-9]+)\s*\(", src)
    return sorted(set(names))


def test_every_declared_symbol_is_exported(L):
    from paper_2510_11683_gb300 import _lib
    names = _declared_functions()
    assert len(names) == len(_lib.SIGNATURES) == 20
    for n in names:
        assert hasattr(L, n), n
        assert n in _lib.SIGNATURES, f"binding lacks {n}"


def test_abi_version_and_names(L, bg):
    assert L.bgpo_abi_version() == 3
    assert L.bgpo_status_string(0) == b"BGPO_OK"
    assert L.bgpo_status_string(8) == b"BGPO_ERR_TIMEOUT"
    assert L.bgpo_status_string(9) == b"BGPO_ERR_BOUNDS"
    assert bg.kernel_name(2) == "lmhead_fwd_lse"
    assert bg.kernel_name(99) == "?"


def test_problem_struct_layout(bg):
    assert ctypes.sizeof(bg.BgpoProblem) == 72
    assert bg.BgpoProblem.seed.offset == 32
    assert bg.BgpoProblem.trace.offset == 48
    assert bg.BgpoProblem.resp_len.offset == 56
    assert bg.BgpoProblem.flags.offset == 64
    assert bg.BgpoProblem.vocab_chunk.offset == 68


def _prob(bg, **kw):
    args = dict(B=2, P=16, R=32, H=64, V=512, n_t=4, G=2, t_mode=0, seed=1)
    args.update(kw)
    return bg.problem(**args)


@pytest.mark.parametrize("kw,status", [
    (dict(B=0), 2), (dict(R=0), 2), (dict(P=-1), 2), (dict(H=100), 2), (dict(H=0), 2),
    (dict(H=56), 2), (dict(H=16392), 2),
    (dict(V=0), 2), (dict(n_t=0), 2), (dict(n_t=65536), 2), (dict(G=0), 2),
    (dict(t_mode=2), 1), (dict(B=1 << 12, R=1 << 11), 2), (dict(V=(1 << 24) + 1), 2),
])
def test_validation_rejects_bad_problems(L, bg, kw, status):
    p = _prob(bg, **kw)
    assert L.bgpo_validate_problem(ctypes.byref(p)) == status
    assert L.bgpo_workspace_bytes(ctypes.byref(p)) == 0


def test_hidden_sizes_in_16_byte_rows_are_accepted(L, bg):
    # H needs 16-byte rows of bf16 (a multiple of 8) and at least one 64-wide K block
    for H in (64, 72, 96, 200, 3584, 4104, 16384):
        assert L.bgpo_validate_problem(ctypes.byref(_prob(bg, H=H))) == 0, H


def test_validation_rejects_bad_offset_and_nonfinite_scale(L, bg):
    p = _prob(bg)
    p.b_offset = -1
    assert L.bgpo_validate_problem(ctypes.byref(p)) == 1
    p.b_offset = (1 << 31) - 1
    assert L.bgpo_validate_problem(ctypes.byref(p)) == 2
    p = _prob(bg, loss_scale=float("nan"))
    assert L.bgpo_validate_problem(ctypes.byref(p)) == 1
    assert L.bgpo_validate_problem(None) == 1


def test_validation_of_flags(L, bg):
    p = _prob(bg)
    for f in (bg.FLAG_KEEP_LOGITS, bg.FLAG_PAIR_DW, bg.FLAG_KEEP_LOGITS | bg.FLAG_PAIR_DW):
        p.flags = f
        assert L.bgpo_validate_problem(ctypes.byref(p)) == 0
    p.flags = 4                      # unknown bit
    assert L.bgpo_validate_problem(ctypes.byref(p)) == 1
    assert L.bgpo_workspace_bytes(ctypes.byref(p)) == 0
    p.flags = 0
    for bad in (7, -256, 100, 255):        # vocab_chunk: a non-negative multiple of 256
        p.vocab_chunk = bad
        assert L.bgpo_validate_problem(ctypes.byref(p)) == 1
    for good in (0, 256, 512, 1 << 24):
        p.vocab_chunk = good
        assert L.bgpo_validate_problem(ctypes.byref(p)) == 0


def test_logit_region_is_the_only_difference_of_the_flag(L, bg):
    # the kept fp32 logits take 4 * roundup(B R, 256) * roundup(V, 64) bytes
    # (rounded to the 1 KB region alignment), appended after every other region
    for (B, R, V) in ((2, 32, 512), (3, 301, 1000), (16, 512, 126464)):
        keep = L.bgpo_workspace_bytes(ctypes.byref(_prob(bg, B=B, R=R, V=V, keep_logits=True)))
        lean = L.bgpo_workspace_bytes(ctypes.byref(_prob(bg, B=B, R=R, V=V)))
        m_pad = -(-B * R // 256) * 256
        v_pad = -(-V // 64) * 64
        assert keep - lean == -(-4 * m_pad * v_pad // 1024) * 1024


def _default_chunk(V, m_pad):
    # default vocabulary chunk: the whole vocabulary (roundup(V, 64)) when its
    # dZ, m_pad x roundup(V, 64) bf16, fits 1 GiB; else V split into
    # ceil(V / 32768) equal pieces rounded up to 256 columns (one piece: whole)
    v_pad = -(-V // 64) * 64
    if 2 * m_pad * v_pad <= 1 << 30:
        return v_pad
    n = -(-V // 32768)
    w = -(-(-(-V // n)) // 256) * 256
    return v_pad if w >= V else w


def test_pairing_doubles_xm_transpose_and_keeps_dz_for_the_whole_vocabulary(L, bg):
    # BGPO_FLAG_PAIR_DW gives Xm^T [H, rows] twice the rows and dZ twice the rows
    # over the whole vocabulary (roundup(V, 64) columns) instead of one chunk:
    # 2 m_pad H + 2 (2 m_pad v_pad - m_pad chunk) more bytes, with or without the
    # logit region
    for (B, R, V, H) in ((2, 32, 512, 64), (3, 301, 1000, 192), (16, 512, 126464, 4096),
                         (32, 1024, 152064, 3584)):
        m_pad = -(-B * R // 256) * 256
        v_pad = -(-V // 64) * 64
        for keep in (False, True):
            lean = L.bgpo_workspace_bytes(ctypes.byref(_prob(bg, B=B, R=R, V=V, H=H, keep_logits=keep)))
            pair = L.bgpo_workspace_bytes(ctypes.byref(
                _prob(bg, B=B, R=R, V=V, H=H, keep_logits=keep, pair_dw=True)))
            assert pair - lean == 2 * m_pad * H + 2 * (2 * m_pad * v_pad - m_pad * _default_chunk(V, m_pad))


def test_vocabulary_chunk_sets_the_dz_buffer(L, bg):
    # dZ holds roundup(B R, 256) x chunk bf16 values: the default chunk, an
    # explicit one, and the whole vocabulary (a chunk of V or more)
    B, R, V, H = 16, 512, 126464, 4096
    m_pad = B * R
    assert _default_chunk(V, m_pad) == 31744
    size = lambda **kw: L.bgpo_workspace_bytes(ctypes.byref(_prob(bg, B=B, R=R, V=V, H=H, **kw)))
    whole = size(vocab_chunk=1 << 17)
    assert whole - size() == 2 * m_pad * (V - 31744)
    assert whole - size(vocab_chunk=8192) == 2 * m_pad * (V - 8192)
    assert size(vocab_chunk=V // 256 * 256 + 256) == whole
    # with pairing the default keeps the whole vocabulary; an explicit chunk
    # only sets how the backward walks it, not the buffer
    assert size(pair_dw=True) == size(pair_dw=True, vocab_chunk=8192)


def test_workspace_independent_of_n_t(L, bg):
    for pair in (False, True):
        sizes = {n: L.bgpo_workspace_bytes(ctypes.byref(_prob(bg, n_t=n, pair_dw=pair)))
                 for n in (1, 2, 3, 16, 32, 1000)}
        assert len(set(sizes.values())) == 1 and sizes[1] > 0


def test_workspace_grows_with_rows_and_vocab(L, bg):
    a = L.bgpo_workspace_bytes(ctypes.byref(_prob(bg)))
    assert L.bgpo_workspace_bytes(ctypes.byref(_prob(bg, B=16))) > a
    assert L.bgpo_workspace_bytes(ctypes.byref(_prob(bg, V=4096))) > a


def test_workspace_of_paper_shapes_fits_hbm(L, bg):
    # LLaDA-8B head, 16 x 512 responses; Dream-7B head, 32 x 1024 (bytes, not n_t-dependent)
    p = bg.problem(16, 256, 512, 4096, 126464, 16, 8, 1, 3)
    assert 0.5e9 < L.bgpo_workspace_bytes(ctypes.byref(p)) < 1.5e9
    p = bg.problem(16, 256, 512, 4096, 126464, 16, 8, 1, 3, keep_logits=True)
    assert 1e9 < L.bgpo_workspace_bytes(ctypes.byref(p)) < 8e9
    p = bg.problem(16, 256, 512, 4096, 126464, 16, 8, 1, 3, pair_dw=True)
    assert 1e9 < L.bgpo_workspace_bytes(ctypes.byref(p)) < 5e9
    p = bg.problem(32, 512, 1024, 3584, 152064, 16, 8, 0, 5)
    assert L.bgpo_workspace_bytes(ctypes.byref(p)) < 5e9
    p = bg.problem(32, 512, 1024, 3584, 152064, 16, 8, 0, 5, keep_logits=True)
    assert L.bgpo_workspace_bytes(ctypes.byref(p)) < 40e9


FAKE = 1 << 20  # an aligned, never dereferenced address


def test_sample_index_out_of_range(L, bg):
    p = _prob(bg)
    ws = L.bgpo_workspace_bytes(ctypes.byref(p))
    for j in (-1, 4, 100):
        assert L.bgpo_sample_mask(ctypes.byref(p), j, FAKE, ws, None, None, None) == 1
        assert L.bgpo_elbo_fwd(ctypes.byref(p), j, FAKE, FAKE, FAKE, FAKE, ws, FAKE, None) == 1


def test_null_and_misaligned_pointers(L, bg):
    p = _prob(bg)
    ws = L.bgpo_workspace_bytes(ctypes.byref(p))
    assert L.bgpo_sample_mask(ctypes.byref(p), 0, None, ws, None, None, None) == 1
    assert L.bgpo_sample_mask(ctypes.byref(p), 0, FAKE + 16, ws, None, None, None) == 3
    assert L.bgpo_elbo_fwd(ctypes.byref(p), 0, None, FAKE, FAKE, FAKE, ws, FAKE, None) == 1
    assert L.bgpo_elbo_fwd(ctypes.byref(p), 0, FAKE + 2, FAKE, FAKE, FAKE, ws, FAKE, None) == 3
    assert L.bgpo_elbo_fwd(ctypes.byref(p), 0, FAKE, FAKE + 8, FAKE, FAKE, ws, FAKE, None) == 3
    assert L.bgpo_bound_coeffs(ctypes.byref(p), 0, FAKE, None, FAKE, FAKE, None, FAKE, ws, None) == 1
    assert L.bgpo_bound_coeffs(ctypes.byref(p), 0, FAKE + 1, FAKE, FAKE, FAKE, None, FAKE, ws, None) == 3
    assert L.bgpo_elbo_bwd_accumulate(ctypes.byref(p), 0, FAKE, FAKE, FAKE, FAKE, FAKE, ws,
                                      FAKE, None, None) == 1
    assert L.bgpo_elbo_bwd_accumulate(ctypes.byref(p), 0, FAKE, FAKE, FAKE, FAKE, FAKE, ws,
                                      FAKE + 4, FAKE, None) == 3
    assert L.bgpo_group_advantage(ctypes.byref(p), None, FAKE, None) == 1


def test_noalloc_forward_validates_before_any_cuda_call(L, bg):
    # bgpo_elbo_fwd_noalloc: every pointer check, including resp_len's
    # alignment, returns before the library touches the device
    p = _prob(bg)
    t, ell = FAKE, FAKE
    assert L.bgpo_elbo_fwd_noalloc(ctypes.byref(p), 0, None, FAKE, FAKE, t, ell, None) == 1
    assert L.bgpo_elbo_fwd_noalloc(ctypes.byref(p), 0, FAKE + 8, FAKE, FAKE, t, ell, None) == 3
    assert L.bgpo_elbo_fwd_noalloc(ctypes.byref(p), 0, FAKE, FAKE, FAKE, t + 2, ell, None) == 3
    p.resp_len = FAKE + 2
    assert L.bgpo_elbo_fwd_noalloc(ctypes.byref(p), 0, FAKE, FAKE, FAKE, t, ell, None) == 3
    assert L.bgpo_sample_mask(ctypes.byref(p), 0, FAKE, L.bgpo_workspace_bytes(ctypes.byref(p)),
                              None, None, None) == 3


def test_workspace_too_small(L, bg):
    p = _prob(bg)
    ws = L.bgpo_workspace_bytes(ctypes.byref(p))
    assert L.bgpo_sample_mask(ctypes.byref(p), 0, FAKE, ws - 1, None, None, None) == 4
    assert L.bgpo_elbo_bwd_accumulate(ctypes.byref(p), 0, FAKE, FAKE, FAKE, FAKE, FAKE, 1024,
                                      FAKE, FAKE, None) == 4


def test_group_size_must_divide_batch(L, bg):
    p = _prob(bg, B=6, G=4)
    assert L.bgpo_group_advantage(ctypes.byref(p), FAKE, FAKE, None) == 2


def test_valid_call_without_gpu_reports_device(L, bg):
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    p = _prob(bg)
    ws = L.bgpo_workspace_bytes(ctypes.byref(p))
    assert L.bgpo_sample_mask(ctypes.byref(p), 0, FAKE, ws, None, None, None) == 6


def test_trace_api_without_events(L):
    assert L.bgpo_trace_create(0) is None
    assert L.bgpo_trace_count(None) == 0
    L.bgpo_trace_reset(None)
    L.bgpo_trace_destroy(None)
    kid = ctypes.c_int32(0)
    ms = ctypes.c_float(0)
    assert L.bgpo_trace_get(None, 0, ctypes.byref(kid), ctypes.byref(ms)) == 1


def test_binding_rejects_cpu_tensors(bg):
    import torch
    p = _prob(bg)
    with pytest.raises(ValueError):
        bg.sample_mask(p, 0, torch.zeros(16, dtype=torch.uint8))


def test_selftest_rejects_bad_arguments(L):
    assert L.bgpo_selftest_bounded_wait(None, 1024, 100, None) == 1
    assert L.bgpo_selftest_bounded_wait(FAKE + 8, 1024, 100, None) == 3
    assert L.bgpo_selftest_bounded_wait(FAKE, 1024, 0, None) == 1
    assert L.bgpo_selftest_bounded_wait(FAKE, 1024, 2000000, None) == 1


def test_checked_build_exports_the_same_abi():
    # the bounds-checked build (-DBGPO_CHECKED) is a drop-in for the normal one
    from paper_2510_11683_gb300 import _lib
    from tests.harness import ensure_built
    h = ctypes.CDLL(ensure_built(checked=True))
    for name, (res, args) in _lib.SIGNATURES.items():
        f = getattr(h, name)
        f.restype, f.argtypes = res, args
    assert h.bgpo_abi_version() == 3
    assert h.bgpo_status_string(9) == b"BGPO_ERR_BOUNDS"
