"""GB300-native BGPO masked-diffusion ELBO hot path (arxiv 2510.11683).

Thin PyTorch binding over the C ABI of ``include/bgpo.h``. Every step of the
path runs in the CUDA kernels of ``lib/libbgpo.so``; this module only checks
tensor dtypes/devices and passes raw pointers and the current CUDA stream.

Per MC sample j (Algorithm 1):

    sample_mask(prob, j, ws)                       # t_{b,j}, mask (Sec. 2.1)
    elbo_fwd(prob, j, X, W, Y, ws, ell[j])         # Eq. 4 through the LM head
    bound_coeffs(prob, j, ell[j], ell_old[j], A, coef, g, ws)   # Eq. 10, 13
    elbo_bwd_accumulate(prob, j, X, W, Y, coef, ws, dX, dW)     # dX, dW +=
"""
import ctypes

from . import _lib
from ._lib import BgpoError, BgpoProblem  # noqa: F401

T_IID = 0
T_STRATIFIED = 1
FLAG_KEEP_LOGITS = 1   # BGPO_FLAG_KEEP_LOGITS
FLAG_PAIR_DW = 2       # BGPO_FLAG_PAIR_DW


def _torch():
    import torch
    return torch


def problem(B, P, R, H, V, n_t, G, t_mode=T_IID, seed=0, loss_scale=None, trace=None,
            b_offset=0, resp_len=None, keep_logits=False, pair_dw=False, vocab_chunk=0):
    """Builds a ``bgpo_problem``; loss_scale defaults to 1/G (Algorithm 1).

    b_offset: global index of the first sequence (a data-parallel shard of a
    larger batch draws the same t and masks as the whole batch would).
    resp_len: optional int32 CUDA tensor [B] of real response lengths (padding
    positions are never masked); the tensor must outlive the calls.
    keep_logits: sets BGPO_FLAG_KEEP_LOGITS (the forward keeps the masked
    rows' fp32 logits in the workspace and the backward reads them instead of
    recomputing them; larger workspace, same results).
    pair_dw: sets BGPO_FLAG_PAIR_DW (samples 2k and 2k + 1 share one dW GEMM:
    dW is complete after every odd sample's backward and the last sample's,
    not in between; larger workspace, dW equal up to fp32 summation order).
    vocab_chunk: columns of the vocabulary the backward handles at a time (0 =
    the library's default; else a multiple of 256); sets the size of the
    workspace's dL/dz buffer."""
    p = BgpoProblem()
    p.B, p.P, p.R, p.H, p.V, p.n_t, p.G, p.t_mode = B, P, R, H, V, n_t, G, t_mode
    p.seed = seed
    p.loss_scale = (1.0 / G if G > 0 else 1.0) if loss_scale is None else loss_scale
    p.b_offset = b_offset
    p.resp_len = _ptr(resp_len, _torch().int32, "resp_len") if resp_len is not None else None
    p.trace = trace.handle if isinstance(trace, Trace) else trace
    p.flags = (FLAG_KEEP_LOGITS if keep_logits else 0) | (FLAG_PAIR_DW if pair_dw else 0)
    p.vocab_chunk = vocab_chunk
    return p


def problem_from(wl, trace=None, loss_scale=None, b_offset=0, resp_len=None,
                 keep_logits=False, pair_dw=False, vocab_chunk=0):
    """``bgpo_problem`` of a synthetic workload description (synth.Workload)."""
    return problem(wl.B, wl.P, wl.R, wl.H, wl.V, wl.n_t, wl.G, wl.t_mode, wl.seed,
                   loss_scale=loss_scale, trace=trace, b_offset=b_offset, resp_len=resp_len,
                   keep_logits=keep_logits, pair_dw=pair_dw, vocab_chunk=vocab_chunk)


def validate_problem(prob):
    return _lib.lib().bgpo_validate_problem(ctypes.byref(prob))


def workspace_bytes(prob):
    n = _lib.lib().bgpo_workspace_bytes(ctypes.byref(prob))
    if n == 0:
        raise BgpoError("bgpo_workspace_bytes", validate_problem(prob))
    return n


def alloc_workspace(prob, device="cuda"):
    """A uint8 device tensor of workspace_bytes(prob) (256-byte aligned by torch)
    with a cleared device error word and nothing pending (the rest is scratch
    the calls overwrite)."""
    torch = _torch()
    ws = torch.empty(workspace_bytes(prob), dtype=torch.uint8, device=device)
    assert ws.data_ptr() % 256 == 0
    with torch.cuda.device(ws.device):
        clear_device_error(ws)
    return ws


def _ptr(t, dtype=None, name="tensor"):
    if t is None:
        return None
    torch = _torch()
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch.Tensor")
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    # the library launches on the current device: a pointer into another
    # device's memory would be an illegal address there
    cur = torch.cuda.current_device()
    if t.device.index != cur:
        raise ValueError(f"{name} is on {t.device}, but the current CUDA device is cuda:{cur}")
    if dtype is not None and t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return t.data_ptr()


def _stream(stream):
    torch = _torch()
    s = torch.cuda.current_stream() if stream is None else stream
    return s.cuda_stream


def sample_mask(prob, j, ws, t_out=None, mask_out=None, stream=None):
    torch = _torch()
    st = _lib.lib().bgpo_sample_mask(
        ctypes.byref(prob), j, _ptr(ws, torch.uint8, "ws"), ws.numel(),
        _ptr(t_out, torch.float32, "t_out"), _ptr(mask_out, torch.uint8, "mask_out"),
        _stream(stream))
    _lib.check("bgpo_sample_mask", st)


def elbo_fwd(prob, j, X, W, Y, ws, ell_out, stream=None):
    torch = _torch()
    st = _lib.lib().bgpo_elbo_fwd(
        ctypes.byref(prob), j, _ptr(X, torch.bfloat16, "X"), _ptr(W, torch.bfloat16, "W"),
        _ptr(Y, torch.int32, "Y"), _ptr(ws, torch.uint8, "ws"), ws.numel(),
        _ptr(ell_out, torch.float32, "ell_out"), _stream(stream))
    _lib.check("bgpo_elbo_fwd", st)


def bound_coeffs(prob, j, ell, ell_old, A, coef_out, g_out, ws, stream=None):
    torch = _torch()
    f32 = torch.float32
    st = _lib.lib().bgpo_bound_coeffs(
        ctypes.byref(prob), j, _ptr(ell, f32, "ell"), _ptr(ell_old, f32, "ell_old"),
        _ptr(A, f32, "A"), _ptr(coef_out, f32, "coef_out"), _ptr(g_out, f32, "g_out"),
        _ptr(ws, torch.uint8, "ws"), ws.numel(), _stream(stream))
    _lib.check("bgpo_bound_coeffs", st)


def vrpo_coeffs(prob, ell, ell_old, A, coef_out, R_out, ws, stream=None):
    """Eq. 7 coefficients from all n_t samples' l ([n_t, B] tensors)."""
    torch = _torch()
    f32 = torch.float32
    st = _lib.lib().bgpo_vrpo_coeffs(
        ctypes.byref(prob), _ptr(ell, f32, "ell"), _ptr(ell_old, f32, "ell_old"),
        _ptr(A, f32, "A"), _ptr(coef_out, f32, "coef_out"), _ptr(R_out, f32, "R_out"),
        _ptr(ws, torch.uint8, "ws"), ws.numel(), _stream(stream))
    _lib.check("bgpo_vrpo_coeffs", st)


def elbo_bwd_accumulate(prob, j, X, W, Y, coef, ws, dX, dW, stream=None):
    torch = _torch()
    f32 = torch.float32
    st = _lib.lib().bgpo_elbo_bwd_accumulate(
        ctypes.byref(prob), j, _ptr(X, torch.bfloat16, "X"), _ptr(W, torch.bfloat16, "W"),
        _ptr(Y, torch.int32, "Y"), _ptr(coef, f32, "coef"), _ptr(ws, torch.uint8, "ws"),
        ws.numel(), _ptr(dX, f32, "dX"), _ptr(dW, f32, "dW"), _stream(stream))
    _lib.check("bgpo_elbo_bwd_accumulate", st)


def group_advantage(prob, rewards, A_out, stream=None):
    torch = _torch()
    st = _lib.lib().bgpo_group_advantage(
        ctypes.byref(prob), _ptr(rewards, torch.float32, "rewards"),
        _ptr(A_out, torch.float32, "A_out"), _stream(stream))
    _lib.check("bgpo_group_advantage", st)


def get_device_error(ws, stream=None):
    """(status, where) of the workspace's device error word (synchronises)."""
    torch = _torch()
    code = ctypes.c_int32(0)
    where = ctypes.c_int32(0)
    st = _lib.lib().bgpo_get_device_error(_ptr(ws, torch.uint8, "ws"), ws.numel(),
                                          ctypes.byref(code), ctypes.byref(where), _stream(stream))
    _lib.check("bgpo_get_device_error", st)
    return code.value, where.value


def clear_device_error(ws, stream=None):
    torch = _torch()
    st = _lib.lib().bgpo_clear_device_error(_ptr(ws, torch.uint8, "ws"), ws.numel(),
                                            _stream(stream))
    _lib.check("bgpo_clear_device_error", st)


def selftest_bounded_wait(ws, timeout_us=2000, stream=None):
    """Launches the bounded-wait self-test; read the result with get_device_error."""
    torch = _torch()
    st = _lib.lib().bgpo_selftest_bounded_wait(_ptr(ws, torch.uint8, "ws"), ws.numel(),
                                               timeout_us, _stream(stream))
    _lib.check("bgpo_selftest_bounded_wait", st)


def kernel_name(kid):
    return _lib.lib().bgpo_kernel_name(kid).decode()


class Trace:
    """Per-kernel CUDA-event timing: pass ``trace=`` to ``problem``."""

    def __init__(self, capacity):
        self.handle = _lib.lib().bgpo_trace_create(capacity)
        if not self.handle:
            raise BgpoError("bgpo_trace_create", 7)

    def reset(self):
        _lib.lib().bgpo_trace_reset(self.handle)

    def records(self):
        """[(kernel name, ms)] of the launches recorded since the last reset."""
        L = _lib.lib()
        out = []
        for i in range(L.bgpo_trace_count(self.handle)):
            kid = ctypes.c_int32(0)
            ms = ctypes.c_float(0)
            _lib.check("bgpo_trace_get", L.bgpo_trace_get(self.handle, i, ctypes.byref(kid),
                                                          ctypes.byref(ms)))
            out.append((kernel_name(kid.value), ms.value))
        return out

    def close(self):
        if self.handle:
            _lib.lib().bgpo_trace_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
