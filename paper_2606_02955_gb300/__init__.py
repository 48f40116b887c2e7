"""Python binding of libfdllm.so: Frechet profile commit-set selection on GB300 (sm_103a).

The functions carry the names of the C interface (include/fdllm.h) and only marshal
arguments: every step of the selection runs in the library's CUDA kernels.  PyTorch
supplies device memory and the current stream.  The first call loads the compiled library
and raises when it has not been built (``paper_2606_02955_gb300.build``); there is no
fallback implementation.
"""
from __future__ import annotations

import ctypes
import functools
import os

import torch

from .build import LIB_PATH

__all__ = [
    "BF16", "FP32", "FP16", "PROFILE", "FACTOR", "THRESHOLD", "ROW_NONFINITE", "ROW_DEVICE_ERROR",
    "FdllmError", "fdllm_select", "fdllm_select_ws", "fdllm_workspace_bytes",
    "fdllm_confidence", "fdllm_select_from_conf", "fdllm_device_status",
    "fdllm_workspace_status", "fdllm_static_status", "fdllm_release_workspace",
    "fdllm_status_string",
    "fdllm_version", "library_path", "fdllm_select_static", "fdllm_select_robust",
    "fdllm_profile_terms", "fdllm_check_bounded_wait", "fdllm_decode_loop", "FORWARD_FN",
    "fdllm_lmhead_select", "fdllm_lmhead_confidence", "fdllm_lmhead_logits",
    "fdllm_gather_masked_rows", "fdllm_decode_loop_lmhead", "fdllm_vocab_reduce",
    "fdllm_select_host",
]

BF16, FP32, FP16 = 0, 1, 2
PROFILE, FACTOR, THRESHOLD = 0, 1, 2
ROW_NONFINITE, ROW_DEVICE_ERROR = -1, -2
OK, ERR_ARG, ERR_ALIGN, ERR_NONFINITE, ERR_CUDA, ERR_WORKSPACE, ERR_DEVICE = range(7)
MODES = {"profile": PROFILE, "factor": FACTOR, "threshold": THRESHOLD}

_lib = None

# fdllm_forward_fn: (user, loop_state, block_mask, logits, stream) -> int
FORWARD_FN = ctypes.CFUNCTYPE(ctypes.c_int, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p,
                              ctypes.c_void_p, ctypes.c_void_p)


def _load():
    """Load libfdllm.so once; a missing library is an error, never a fallback."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise ImportError(
            "libfdllm.so is not built (%s); run paper_2606_02955_gb300.build.build_library() "
            "or __graft_entry__.build()" % LIB_PATH)
    lib = ctypes.CDLL(LIB_PATH)
    p, i, d, sz = ctypes.c_void_p, ctypes.c_int, ctypes.c_double, ctypes.c_size_t
    lib.fdllm_select.argtypes = [p, i, i, i, i, p, d, i, p, p, p, p]
    lib.fdllm_select.restype = i
    lib.fdllm_select_ws.argtypes = [p, i, i, i, i, p, d, i, p, p, p, p, sz, p]
    lib.fdllm_select_ws.restype = i
    lib.fdllm_select_robust.argtypes = [p, i, i, i, i, p, d, d, p, p, p, p, p]
    lib.fdllm_select_robust.restype = i
    lib.fdllm_select_static.argtypes = [p, i, i, i, i, p, d, i, p, p, p, p]
    lib.fdllm_select_static.restype = i
    lib.fdllm_workspace_bytes.argtypes = [i, i, i, i]
    lib.fdllm_workspace_bytes.restype = sz
    lib.fdllm_lmhead_select.argtypes = [p, p, i, i, i, i, p, d, i, p, p, p, p]
    lib.fdllm_lmhead_select.restype = i
    lib.fdllm_lmhead_confidence.argtypes = [p, p, i, i, i, i, p, p, p, p]
    lib.fdllm_lmhead_confidence.restype = i
    lib.fdllm_lmhead_logits.argtypes = [p, p, i, i, i, i, p, p, p]
    lib.fdllm_lmhead_logits.restype = i
    lib.fdllm_gather_masked_rows.argtypes = [p, p, i, i, i, i, p, p]
    lib.fdllm_gather_masked_rows.restype = i
    lib.fdllm_confidence.argtypes = [p, i, i, i, i, p, p, p, p]
    lib.fdllm_confidence.restype = i
    lib.fdllm_vocab_reduce.argtypes = [p, i, i, i, i, p, p]
    lib.fdllm_vocab_reduce.restype = i
    lib.fdllm_select_from_conf.argtypes = [p, p, i, i, p, d, i, p, p, p, p]
    lib.fdllm_select_from_conf.restype = i
    lib.fdllm_profile_terms.argtypes = [p, p, i, i, d, p, p, p, p, p, p]
    lib.fdllm_profile_terms.restype = i
    lib.fdllm_decode_loop.argtypes = [i, i, i, i, i, d, i, FORWARD_FN, p, p, p, p, i,
                                      ctypes.POINTER(ctypes.c_int), p]
    lib.fdllm_decode_loop.restype = i
    lib.fdllm_decode_loop_lmhead.argtypes = [i, i, i, i, i, p, d, i, FORWARD_FN, p, p, p, p, i,
                                             ctypes.POINTER(ctypes.c_int), p]
    lib.fdllm_decode_loop_lmhead.restype = i
    lib.fdllm_check_bounded_wait.argtypes = [d, p]
    lib.fdllm_check_bounded_wait.restype = i
    lib.fdllm_device_status.argtypes = [p]
    lib.fdllm_device_status.restype = i
    lib.fdllm_workspace_status.argtypes = [p, p]
    lib.fdllm_workspace_status.restype = i
    lib.fdllm_static_status.argtypes = [p]
    lib.fdllm_static_status.restype = i
    lib.fdllm_select_host.argtypes = [p, i, i, i, i, p, d, i, p, p, p, p]
    lib.fdllm_select_host.restype = i
    lib.fdllm_release_workspace.argtypes = []
    lib.fdllm_release_workspace.restype = None
    lib.fdllm_status_string.argtypes = [i]
    lib.fdllm_status_string.restype = ctypes.c_char_p
    lib.fdllm_version.argtypes = []
    lib.fdllm_version.restype = i
    _lib = lib
    return lib


class FdllmError(RuntimeError):
    def __init__(self, status: int, call: str):
        super().__init__("%s failed: status %d (%s)" % (call, status, fdllm_status_string(status)))
        self.status = status


def library_path() -> str:
    return LIB_PATH



def _on_device(fn):
    """Runs an entry point on the device of its CUDA tensor arguments (the library works on
    the current device: its workspace and launches), and rejects calls whose CUDA tensors
    live on different devices."""
    @functools.wraps(fn)
    def call(*args, **kwargs):
        cuda = [a for a in (*args, *kwargs.values()) if isinstance(a, torch.Tensor) and a.is_cuda]
        if not cuda:
            return fn(*args, **kwargs)
        dev = cuda[0].device
        for t in cuda[1:]:
            if t.device != dev:
                raise ValueError("the CUDA tensors of one call must share a device (%s, %s)"
                                 % (dev, t.device))
        with torch.cuda.device(dev):
            return fn(*args, **kwargs)
    return call


def fdllm_status_string(status: int) -> str:
    return _load().fdllm_status_string(int(status)).decode()


def fdllm_version() -> int:
    return _load().fdllm_version()


def _check(status: int, call: str):
    if status != 0:
        raise FdllmError(status, call)


def _mode(mode) -> int:
    return MODES[mode] if isinstance(mode, str) else int(mode)


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return BF16
    if t.dtype == torch.float32:
        return FP32
    if t.dtype == torch.float16:
        return FP16
    raise TypeError("logits must be bfloat16, float16 or float32, got %s" % t.dtype)


def _stream(stream) -> int:
    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)


def _dev(t: torch.Tensor, name: str, dtype=None, shape=None):
    if not t.is_cuda:
        raise ValueError("%s must be a CUDA tensor" % name)
    if not t.is_contiguous():
        raise ValueError("%s must be contiguous" % name)
    if dtype is not None and t.dtype != dtype:
        raise TypeError("%s must be %s, got %s" % (name, dtype, t.dtype))
    if shape is not None and tuple(t.shape) != tuple(shape):
        raise ValueError("%s must have shape %s, got %s" % (name, tuple(shape), tuple(t.shape)))
    return t.data_ptr()


def _outputs(B, L, device, out_tokens, out_commit, out_n):
    if out_tokens is None:
        out_tokens = torch.full((B, L), -1, dtype=torch.int32, device=device)
    if out_commit is None:
        out_commit = torch.empty((B, L), dtype=torch.uint8, device=device)
    if out_n is None:
        out_n = torch.empty((B,), dtype=torch.int32, device=device)
    return out_tokens, out_commit, out_n


@_on_device
def fdllm_select(logits: torch.Tensor, mask: torch.Tensor, param: float, mode=PROFILE,
                 out_tokens=None, out_commit=None, out_n=None, stream=None):
    """One selection step (fdllm_select).  ``logits`` [B, L, V] bf16/fp16/fp32, ``mask`` [B, L]
    uint8 (updated in place).  Returns (out_tokens, out_commit, out_n).

    Device tensors run asynchronously on ``stream`` (default: current stream).  With host
    tensors the call copies the inputs to the current CUDA device (pinned memory makes the
    copies asynchronous), runs the step, copies the outputs and the updated mask back and
    synchronises: the end-to-end form of the call."""
    if not logits.is_cuda:
        return _select_from_host(logits, mask, param, mode, out_tokens, out_commit, out_n)
    B, L, V = logits.shape
    lp = _dev(logits, "logits")
    mp = _dev(mask, "mask", torch.uint8, (B, L))
    out_tokens, out_commit, out_n = _outputs(B, L, logits.device, out_tokens, out_commit, out_n)
    st = _load().fdllm_select(lp, _dtype_code(logits), B, L, V, mp, float(param), _mode(mode),
                           _dev(out_tokens, "out_tokens", torch.int32, (B, L)),
                           _dev(out_commit, "out_commit", torch.uint8, (B, L)),
                           _dev(out_n, "out_n", torch.int32, (B,)), _stream(stream))
    _check(st, "fdllm_select")
    return out_tokens, out_commit, out_n


def _select_from_host(logits, mask, param, mode, out_tokens, out_commit, out_n):
    """fdllm_select_host: the whole step on host tensors in one library call (the GPU reads
    only the masked rows of page-locked logits; results and mask copied back)."""
    B, L, V = logits.shape
    if not logits.is_contiguous():
        raise FdllmError(1, "fdllm_select_host: contiguous logits required")
    pin = logits.is_pinned()

    def host(t, name, dtype, shape, fill=None):
        if t is None:
            t = torch.empty(shape, dtype=dtype, pin_memory=pin)
            if fill is not None:
                t.fill_(fill)
        if t.is_cuda or t.dtype != dtype or tuple(t.shape) != shape or not t.is_contiguous():
            raise FdllmError(1, "%s: contiguous host %s %s required" % (name, dtype, shape))
        return t

    mask = host(mask, "mask", torch.uint8, (B, L))
    out_tokens = host(out_tokens, "out_tokens", torch.int32, (B, L), -1)
    out_commit = host(out_commit, "out_commit", torch.uint8, (B, L))
    out_n = host(out_n, "out_n", torch.int32, (B,))
    st = _load().fdllm_select_host(logits.data_ptr(), _dtype_code(logits), B, L, V,
                                   mask.data_ptr(), float(param), _mode(mode),
                                   out_tokens.data_ptr(), out_commit.data_ptr(),
                                   out_n.data_ptr(), _stream(None))
    _check(st, "fdllm_select_host")
    return out_tokens, out_commit, out_n


@_on_device
def fdllm_select_robust(logits: torch.Tensor, mask: torch.Tensor, param: float, eta: float = 0.0,
                        eta_per_position=None, out_tokens=None, out_commit=None, out_n=None,
                        stream=None):
    """Calibration-robust profile selection (App. C): confidences lowered to
    max(0, c - eta) (``eta_per_position``: [B, L] fp32 CUDA tensor, else the uniform eta)
    before the profile rule.  Returns (out_tokens, out_commit, out_n)."""
    B, L, V = logits.shape
    out_tokens, out_commit, out_n = _outputs(B, L, logits.device, out_tokens, out_commit, out_n)
    ep = None if eta_per_position is None else _dev(eta_per_position, "eta_per_position",
                                                     torch.float32, (B, L))
    st = _load().fdllm_select_robust(_dev(logits, "logits"), _dtype_code(logits), B, L, V,
                                     _dev(mask, "mask", torch.uint8, (B, L)), float(param),
                                     float(eta), ep,
                                     _dev(out_tokens, "out_tokens", torch.int32, (B, L)),
                                     _dev(out_commit, "out_commit", torch.uint8, (B, L)),
                                     _dev(out_n, "out_n", torch.int32, (B,)), _stream(stream))
    _check(st, "fdllm_select_robust")
    return out_tokens, out_commit, out_n


@_on_device
def fdllm_select_static(logits: torch.Tensor, mask: torch.Tensor, param: float, mode=PROFILE,
                        out_tokens=None, out_commit=None, out_n=None, stream=None):
    """fdllm_select using the library's fixed device scratch array instead of an allocated
    workspace (for callers that cannot allocate while stepping).  Pass preallocated outputs
    to keep the call free of allocations on the Python side too."""
    B, L, V = logits.shape
    out_tokens, out_commit, out_n = _outputs(B, L, logits.device, out_tokens, out_commit, out_n)
    st = _load().fdllm_select_static(_dev(logits, "logits"), _dtype_code(logits), B, L, V,
                                     _dev(mask, "mask", torch.uint8, (B, L)), float(param),
                                     _mode(mode),
                                     _dev(out_tokens, "out_tokens", torch.int32, (B, L)),
                                     _dev(out_commit, "out_commit", torch.uint8, (B, L)),
                                     _dev(out_n, "out_n", torch.int32, (B,)), _stream(stream))
    _check(st, "fdllm_select_static")
    return out_tokens, out_commit, out_n


def fdllm_workspace_bytes(B: int, L: int, V: int, dtype=BF16) -> int:
    return int(_load().fdllm_workspace_bytes(B, L, V, dtype))


@_on_device
def fdllm_select_ws(logits: torch.Tensor, mask: torch.Tensor, param: float, mode,
                    workspace: torch.Tensor, out_tokens=None, out_commit=None, out_n=None,
                    stream=None):
    """fdllm_select with a caller workspace (a zero-filled uint8 CUDA tensor of at least
    fdllm_workspace_bytes bytes, 256-byte aligned as torch allocations are)."""
    B, L, V = logits.shape
    out_tokens, out_commit, out_n = _outputs(B, L, logits.device, out_tokens, out_commit, out_n)
    st = _load().fdllm_select_ws(_dev(logits, "logits"), _dtype_code(logits), B, L, V,
                              _dev(mask, "mask", torch.uint8, (B, L)), float(param), _mode(mode),
                              _dev(out_tokens, "out_tokens", torch.int32, (B, L)),
                              _dev(out_commit, "out_commit", torch.uint8, (B, L)),
                              _dev(out_n, "out_n", torch.int32, (B,)),
                              _dev(workspace, "workspace", torch.uint8),
                              workspace.numel(), _stream(stream))
    _check(st, "fdllm_select_ws")
    return out_tokens, out_commit, out_n


@_on_device
def fdllm_confidence(logits: torch.Tensor, mask: torch.Tensor, out_conf=None, out_argmax=None,
                     stream=None):
    """Step a1 alone: (conf fp32 [B, L], argmax int32 [B, L]) written at masked positions
    (unwritten positions of freshly allocated outputs hold NaN / -1)."""
    B, L, V = logits.shape
    if out_conf is None:
        out_conf = torch.full((B, L), float("nan"), dtype=torch.float32, device=logits.device)
    if out_argmax is None:
        out_argmax = torch.full((B, L), -1, dtype=torch.int32, device=logits.device)
    st = _load().fdllm_confidence(_dev(logits, "logits"), _dtype_code(logits), B, L, V,
                               _dev(mask, "mask", torch.uint8, (B, L)),
                               _dev(out_conf, "out_conf", torch.float32, (B, L)),
                               _dev(out_argmax, "out_argmax", torch.int32, (B, L)),
                               _stream(stream))
    _check(st, "fdllm_confidence")
    return out_conf, out_argmax


@_on_device
def fdllm_vocab_reduce(logits: torch.Tensor, mask: torch.Tensor, stream=None):
    """Step a1's vocabulary reduction alone (unit partials in the library workspace, not
    folded into confidences), for timing the reduction kernel by itself."""
    B, L, V = logits.shape
    st = _load().fdllm_vocab_reduce(_dev(logits, "logits"), _dtype_code(logits), B, L, V,
                                    _dev(mask, "mask", torch.uint8, (B, L)), _stream(stream))
    _check(st, "fdllm_vocab_reduce")


def _lmhead_shapes(hidden: torch.Tensor, w_vocab: torch.Tensor):
    B, L, H = hidden.shape
    V, H2 = w_vocab.shape
    if H2 != H:
        raise ValueError("w_vocab must be [V, %d], got %s" % (H, tuple(w_vocab.shape)))
    hp = _dev(hidden, "hidden", torch.bfloat16)
    wp = _dev(w_vocab, "w_vocab", torch.bfloat16)
    return B, L, H, V, hp, wp


@_on_device
def fdllm_lmhead_select(hidden: torch.Tensor, w_vocab: torch.Tensor, mask: torch.Tensor,
                        param: float, mode=PROFILE, out_tokens=None, out_commit=None, out_n=None,
                        stream=None):
    """One selection step with the logits computed and reduced inside the LM-head GEMM
    (fdllm_lmhead_select): ``hidden`` [B, L, H] bf16, ``w_vocab`` [V, H] bf16, ``mask``
    [B, L] uint8 (updated in place).  Returns (out_tokens, out_commit, out_n)."""
    B, L, H, V, hp, wp = _lmhead_shapes(hidden, w_vocab)
    out_tokens, out_commit, out_n = _outputs(B, L, hidden.device, out_tokens, out_commit, out_n)
    st = _load().fdllm_lmhead_select(hp, wp, B, L, H, V, _dev(mask, "mask", torch.uint8, (B, L)),
                                     float(param), _mode(mode),
                                     _dev(out_tokens, "out_tokens", torch.int32, (B, L)),
                                     _dev(out_commit, "out_commit", torch.uint8, (B, L)),
                                     _dev(out_n, "out_n", torch.int32, (B,)), _stream(stream))
    _check(st, "fdllm_lmhead_select")
    return out_tokens, out_commit, out_n


@_on_device
def fdllm_lmhead_confidence(hidden: torch.Tensor, w_vocab: torch.Tensor, mask: torch.Tensor,
                            out_conf=None, out_argmax=None, stream=None):
    """Step a1 on the LM head: (conf fp32 [B, L], argmax int32 [B, L]) at masked positions."""
    B, L, H, V, hp, wp = _lmhead_shapes(hidden, w_vocab)
    if out_conf is None:
        out_conf = torch.full((B, L), float("nan"), dtype=torch.float32, device=hidden.device)
    if out_argmax is None:
        out_argmax = torch.full((B, L), -1, dtype=torch.int32, device=hidden.device)
    st = _load().fdllm_lmhead_confidence(hp, wp, B, L, H, V,
                                         _dev(mask, "mask", torch.uint8, (B, L)),
                                         _dev(out_conf, "out_conf", torch.float32, (B, L)),
                                         _dev(out_argmax, "out_argmax", torch.int32, (B, L)),
                                         _stream(stream))
    _check(st, "fdllm_lmhead_confidence")
    return out_conf, out_argmax


@_on_device
def fdllm_lmhead_logits(hidden: torch.Tensor, w_vocab: torch.Tensor, mask: torch.Tensor,
                        out_logits=None, stream=None):
    """The LM-head GEMM's fp32 logits [B, L, V] at masked rows (other rows untouched; a
    freshly allocated output holds NaN there)."""
    B, L, H, V, hp, wp = _lmhead_shapes(hidden, w_vocab)
    if out_logits is None:
        out_logits = torch.full((B, L, V), float("nan"), dtype=torch.float32,
                                device=hidden.device)
    st = _load().fdllm_lmhead_logits(hp, wp, B, L, H, V, _dev(mask, "mask", torch.uint8, (B, L)),
                                     _dev(out_logits, "out_logits", torch.float32, (B, L, V)),
                                     _stream(stream))
    _check(st, "fdllm_lmhead_logits")
    return out_logits


@_on_device
def fdllm_select_from_conf(conf: torch.Tensor, argmax: torch.Tensor, mask: torch.Tensor,
                           param: float, mode=PROFILE, out_tokens=None, out_commit=None,
                           out_n=None, stream=None):
    """Steps a2-a5 alone on given confidences; returns (out_tokens, out_commit, out_n)."""
    B, L = conf.shape
    out_tokens, out_commit, out_n = _outputs(B, L, conf.device, out_tokens, out_commit, out_n)
    st = _load().fdllm_select_from_conf(_dev(conf, "conf", torch.float32, (B, L)),
                                     _dev(argmax, "argmax", torch.int32, (B, L)), B, L,
                                     _dev(mask, "mask", torch.uint8, (B, L)), float(param),
                                     _mode(mode),
                                     _dev(out_tokens, "out_tokens", torch.int32, (B, L)),
                                     _dev(out_commit, "out_commit", torch.uint8, (B, L)),
                                     _dev(out_n, "out_n", torch.int32, (B,)), _stream(stream))
    _check(st, "fdllm_select_from_conf")
    return out_tokens, out_commit, out_n


@_on_device
def fdllm_profile_terms(conf: torch.Tensor, mask: torch.Tensor, delta: float = 0.0,
                        stream=None):
    """Heterogeneity-bonus diagnostics by rank of each row's sorted masked profile:
    dict(G, F, B, f_eff) fp64 [B, L] (f_eff = 1 - delta + B, the effective factor of the
    profile rule with margin ``delta``) and order int32 [B, L] (NaN / -1 beyond the masked
    count)."""
    B, L = conf.shape
    dev = conf.device
    G, F, Bn, Fe = (torch.empty((B, L), dtype=torch.float64, device=dev) for _ in range(4))
    order = torch.empty((B, L), dtype=torch.int32, device=dev)
    st = _load().fdllm_profile_terms(_dev(conf, "conf", torch.float32, (B, L)),
                                     _dev(mask, "mask", torch.uint8, (B, L)), B, L,
                                     float(delta), G.data_ptr(), F.data_ptr(), Bn.data_ptr(),
                                     Fe.data_ptr(), order.data_ptr(), _stream(stream))
    _check(st, "fdllm_profile_terms")
    return dict(G=G, F=F, B=Bn, f_eff=Fe, order=order)


@_on_device
def fdllm_decode_loop(forward, logits: torch.Tensor, gen_len: int, param: float, mode=PROFILE,
                      max_steps: int | None = None, stream=None):
    """Algorithm 1's outer loop on the GPU (fdllm_decode_loop).  ``logits`` is the
    [B, block_len, V] buffer the forward pass fills; ``forward(loop_state_ptr,
    block_mask_ptr, logits_ptr, stream_ptr)`` receives raw device pointers and the capture
    stream and must only enqueue stream-ordered GPU work.  Returns (seq_tokens [B, gen_len]
    int32, nfe_per_block int32, total steps); synchronous."""
    B, Lb, V = logits.shape
    nblocks = gen_len // Lb
    dev = logits.device
    seq = torch.empty((B, gen_len), dtype=torch.int32, device=dev)
    nfe = torch.empty((nblocks,), dtype=torch.int32, device=dev)
    steps = ctypes.c_int(0)

    def trampoline(user, state, mask, out, strm):
        try:
            r = forward(state, mask, out, strm)
            return 0 if r is None else int(r)
        except Exception:  # the library reports it as FDLLM_ERR_ARG; keep the cause visible
            import traceback
            import warnings
            warnings.warn("forward pass raised during loop capture:\n" + traceback.format_exc())
            return 1

    cb = FORWARD_FN(trampoline)
    st = _load().fdllm_decode_loop(B, gen_len, Lb, V, _dtype_code(logits), float(param),
                                   _mode(mode), cb, None, _dev(logits, "logits"),
                                   seq.data_ptr(), nfe.data_ptr(),
                                   int(max_steps if max_steps is not None else gen_len + 1),
                                   ctypes.byref(steps), _stream(stream))
    _check(st, "fdllm_decode_loop")
    return seq, nfe, steps.value


@_on_device
def fdllm_gather_masked_rows(src: torch.Tensor, mask: torch.Tensor, dst=None, stream=None):
    """Copy the masked positions' rows of ``src`` [B, L, V] (a CUDA tensor or a pinned host
    tensor, read by the GPU directly) into ``dst`` (a CUDA tensor of the same shape and
    dtype; allocated when None).  Returns dst; its unmasked rows are not written."""
    if not src.is_cuda and not src.is_pinned():
        raise ValueError("src must be a CUDA tensor or a pinned host tensor")
    if not src.is_contiguous():
        raise ValueError("src must be contiguous")
    B, L, V = src.shape
    if dst is None:
        dst = torch.empty(src.shape, dtype=src.dtype, device=mask.device)
    _check(_load().fdllm_gather_masked_rows(src.data_ptr(),
                                            _dev(dst, "dst", src.dtype, (B, L, V)),
                                            _dtype_code(src), B, L, V,
                                            _dev(mask, "mask", torch.uint8, (B, L)),
                                            _stream(stream)), "fdllm_gather_masked_rows")
    return dst


@_on_device
def fdllm_decode_loop_lmhead(forward, hidden: torch.Tensor, w_vocab: torch.Tensor, gen_len: int,
                             param: float, mode=PROFILE, max_steps: int | None = None,
                             stream=None):
    """fdllm_decode_loop with the LM head in the loop: ``hidden`` is the [B, block_len, H]
    bf16 buffer the forward pass fills, ``w_vocab`` the [V, H] bf16 head.  Returns
    (seq_tokens [B, gen_len] int32, nfe_per_block int32, total steps); synchronous."""
    B, Lb, H = hidden.shape
    V, H2 = w_vocab.shape
    if H2 != H:
        raise ValueError("w_vocab must be [V, %d]" % H)
    nblocks = gen_len // Lb
    dev = hidden.device
    seq = torch.empty((B, gen_len), dtype=torch.int32, device=dev)
    nfe = torch.empty((nblocks,), dtype=torch.int32, device=dev)
    steps = ctypes.c_int(0)

    def trampoline(user, state, mask, out, strm):
        try:
            r = forward(state, mask, out, strm)
            return 0 if r is None else int(r)
        except Exception:  # the library reports it as FDLLM_ERR_ARG; keep the cause visible
            import traceback
            import warnings
            warnings.warn("forward pass raised during loop capture:\n" + traceback.format_exc())
            return 1

    cb = FORWARD_FN(trampoline)
    st = _load().fdllm_decode_loop_lmhead(
        B, gen_len, Lb, H, V, _dev(w_vocab, "w_vocab", torch.bfloat16), float(param),
        _mode(mode), cb, None, _dev(hidden, "hidden", torch.bfloat16), seq.data_ptr(),
        nfe.data_ptr(), int(max_steps if max_steps is not None else gen_len + 1),
        ctypes.byref(steps), _stream(stream))
    _check(st, "fdllm_decode_loop_lmhead")
    return seq, nfe, steps.value


def fdllm_check_bounded_wait(seconds: float = 0.01, stream=None) -> int:
    """Makes one kernel wait on a barrier nobody completes; returns the status code
    (FDLLM_ERR_DEVICE = 6 when the bounded wait ran out and was reported)."""
    return _load().fdllm_check_bounded_wait(float(seconds), _stream(stream))


def fdllm_device_status(stream=None) -> int:
    """Synchronises and returns (clearing it) the library workspace's sticky device status."""
    return _load().fdllm_device_status(_stream(stream))


@_on_device
def fdllm_workspace_status(workspace: torch.Tensor, stream=None) -> int:
    return _load().fdllm_workspace_status(_dev(workspace, "workspace", torch.uint8), _stream(stream))


def fdllm_static_status(stream=None) -> int:
    """Synchronises and returns (clearing it) the sticky device status of
    fdllm_select_static's fixed array on the current device."""
    return _load().fdllm_static_status(_stream(stream))


def fdllm_release_workspace() -> None:
    _load().fdllm_release_workspace()
