"""ctypes binding of libprorouter.so with the C ABI's call names.

Argument marshalling only: tensors are passed as raw pointers, every step of
the verifier runs in the library's CUDA kernels.  PyTorch provides device
memory and streams.  Importing this module raises if the library is missing:
there is no fallback.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np
import torch

from .build import LIB

PR_OK, PR_ERR_INVALID_ARG, PR_ERR_UNSUPPORTED, PR_ERR_CUDA, PR_ERR_NO_MEMORY = 0, -1, -2, -3, -4
PR_DTYPE_F32, PR_DTYPE_BF16 = 0, 1
PR_FLAG_NONFINITE, PR_FLAG_BAD_CHOSEN, PR_FLAG_EMPTY_REQ = 1, 2, 4
PR_FLAG_BAD_OFFSETS, PR_FLAG_BAD_SLOT, PR_FLAG_TIMEOUT = 8, 16, 32
PR_NFEAT, PR_NAGG, PR_MAX_TOPK = 8, 11, 32
PR_OPT_TOPK, PR_OPT_TOPK_RENORM, PR_OPT_SPLIT, PR_OPT_OVERLAP, PR_OPT_TIMING = 0, 1, 2, 3, 4
PR_NOALLOC_MAX_ROWS, PR_NOALLOC_MAX_REQUESTS = 16384, 1024
PR_HEAD_D, PR_HEAD_HEADS, PR_HEAD_FF, PR_HEAD_MAX_LAYERS = 64, 4, 128, 8
PR_QMLP_SUMMARY, PR_QMLP_PARAMS = 28, 6081
PR_LMHEAD_MAX_VOCAB = (1 << 31) - 256

# every symbol include/pro_router.h declares
EXPORTS = (
    "pr_ctx_create", "pr_ctx_destroy", "pr_ctx_reset", "pr_ctx_set_option", "pr_ctx_flags",
    "pr_token_features", "pr_aggregate_score", "pr_route", "pr_route_host", "pr_decode_step",
    "pr_state_export", "pr_state_import", "pr_status_string", "pr_last_cuda_error",
    "pr_launch_count", "pr_route_noalloc", "pr_head_param_count", "pr_head_score",
    "pr_ctx_kernel_times", "pr_selective_metrics", "pr_quantile_score", "pr_lmhead_features",
    "pr_selftest_wait", "pr_lmhead_decode_step", "pr_last_error", "pr_prescorer_fit",
    "pr_prescorer_destroy", "pr_prescorer_vocab_size", "pr_prescorer_term",
    "pr_prescorer_features", "pr_prescorer_score",
)

if not os.path.exists(LIB):
    raise ImportError("libprorouter.so has not been built (python -m paper_2608_28726_gb300.build)")

_P = ctypes.c_void_p
_I32, _I64, _F32, _SZ = ctypes.c_int32, ctypes.c_int64, ctypes.c_float, ctypes.c_size_t
_lib = ctypes.CDLL(LIB)
_SIGS = {
    "pr_ctx_create": [ctypes.POINTER(_P), ctypes.c_int, _I64, _I32],
    "pr_ctx_destroy": [_P],
    "pr_ctx_reset": [_P, _P],
    "pr_ctx_set_option": [_P, _I32, _I32],
    "pr_ctx_flags": [_P, _P, _I32, ctypes.POINTER(ctypes.c_uint32)],
    "pr_last_error": [_P, ctypes.POINTER(ctypes.c_uint32)],
    "pr_token_features": [_P, _P, ctypes.c_int, _I64, _I64, _I64, _P, _I32, _P, _I32, _P, _P, _P,
                          _P],
    "pr_aggregate_score": [_P, _P, _P, _I64, _P, _I32, _P, _F32, _F32, _P, _P, _P, _P, _P],
    "pr_route": [_P, _P, ctypes.c_int, _I64, _I64, _I64, _I64, _P, _P, _I32, _P, _F32, _F32, _P, _P,
                 _P, _P, _P],
    "pr_route_host": [_P, _P, ctypes.c_int, _I64, _I64, _I64, _P, _P, _I32, _P, _F32, _F32, _I64,
                      _P, _P, _P, _P, _P],
    "pr_decode_step": [_P, _P, ctypes.c_int, _I32, _I64, _I64, _P, _P, _P, _P, _F32, _F32, _P, _P,
                       _P, _P, _P],
    "pr_route_noalloc": [_P, ctypes.c_int, _I64, _I64, _I64, _P, _P, _I32, _P, _F32, _F32, _P, _P,
                         _P, _P, _P],
    "pr_ctx_kernel_times": [_P, _P, _I32, ctypes.POINTER(_I32)],
    "pr_lmhead_features": [_P, _P, _P, _I64, _I64, _I64, _P, _I32, _P, _I32, _P, _P, _P, _P],
    "pr_selftest_wait": [_P, _I64, ctypes.POINTER(_I32)],
    "pr_lmhead_decode_step": [_P, _P, _P, _I32, _I64, _I64, _P, _P, _P, _P, _F32, _F32, _P, _P,
                              _P, _P, _P],
    "pr_quantile_score": [_P, _P, _P, _I64, _P, _I32, _P, _F32, _P, _P, _P, _P, _P],
    "pr_selective_metrics": [_P, _P, _P, _I64, ctypes.c_double, _P, _P],
    "pr_head_score": [_P, _P, _P, _I64, _P, _I32, _P, _I32, _F32, _P, _P, _P, _P],
    "pr_state_export": [_P, _P, ctypes.POINTER(_SZ)],
    "pr_state_import": [_P, _P, _SZ],
    "pr_prescorer_fit": [_P, _I32, _I32, ctypes.POINTER(_P)],
    "pr_prescorer_features": [_P, ctypes.c_char_p, _I32, _P, _P, ctypes.POINTER(_I32),
                              ctypes.POINTER(_I64)],
    "pr_prescorer_score": [_P, _P, _P, _I32, _P, _F32, _I32, _P, _P],
}
for _name, _args in _SIGS.items():
    _fn = getattr(_lib, _name)
    _fn.argtypes = _args
    _fn.restype = ctypes.c_int
_lib.pr_status_string.argtypes = [ctypes.c_int]
_lib.pr_status_string.restype = ctypes.c_char_p
_lib.pr_last_cuda_error.argtypes = []
_lib.pr_last_cuda_error.restype = ctypes.c_char_p
_lib.pr_launch_count.argtypes = []
_lib.pr_launch_count.restype = ctypes.c_uint64
_lib.pr_head_param_count.argtypes = [_I32]
_lib.pr_head_param_count.restype = _I64
_lib.pr_prescorer_destroy.argtypes = [_P]
_lib.pr_prescorer_destroy.restype = None
_lib.pr_prescorer_vocab_size.argtypes = [_P]
_lib.pr_prescorer_vocab_size.restype = _I64
_lib.pr_prescorer_term.argtypes = [_P, _I64]
_lib.pr_prescorer_term.restype = ctypes.c_char_p


class PRError(RuntimeError):
    def __init__(self, status: int, call: str, detail: str | None = None):
        msg = _lib.pr_status_string(status).decode()
        if status == PR_ERR_CUDA:
            msg += " (" + _lib.pr_last_cuda_error().decode() + ")"
        if detail:
            msg += " (" + detail + ")"
        super().__init__("%s: %s" % (call, msg))
        self.status = status


def _check(st: int, call: str):
    if st != PR_OK:
        raise PRError(st, call)


# ---- argument checks before any pointer reaches the library -------------------------
#
# The C ABI cannot tell a host pointer from a device pointer, nor a buffer's
# size, without a driver query per call; a CPU tensor, a tensor on another GPU
# or a short output buffer would reach a kernel as a bad address.  So every
# tensor meant for device memory is checked here: a CUDA tensor on the
# device of the context (or the current device for the context-free call),
# of the expected dtype, contiguous, and at least as large as the call needs.

_CTX_DEVICE = {}  # context handle value -> CUDA device index

_I32_T = (torch.int32,)
_U8_T = (torch.uint8, torch.bool)
_F32_T = (torch.float32,)
_I64_T = (torch.int64,)


def _ctx_device(ctx) -> int:
    h = getattr(ctx, "value", ctx)
    if h in _CTX_DEVICE:
        return _CTX_DEVICE[h]
    return torch.cuda.current_device() if torch.cuda.is_available() else 0


def _dev(call: str, dev: int, name: str, t, dtypes=None, numel: int | None = None,
         optional: bool = False, contiguous: bool = True):
    # the common case in one expression (this runs on every call of a hot loop)
    try:
        if (t.is_cuda and t.get_device() == dev and (dtypes is None or t.dtype in dtypes)
                and (not contiguous or t.is_contiguous()) and (numel is None or t.numel() >= numel)):
            return
    except AttributeError:
        pass
    _dev_refuse(call, dev, name, t, dtypes, numel, optional, contiguous)


def _dev_refuse(call, dev, name, t, dtypes, numel, optional, contiguous):
    if t is None:
        if optional:
            return
        raise PRError(PR_ERR_INVALID_ARG, call, "%s is required" % name)
    if not isinstance(t, torch.Tensor) or not t.is_cuda or t.device.index != dev:
        where = t.device if isinstance(t, torch.Tensor) else type(t).__name__
        raise PRError(PR_ERR_INVALID_ARG, call,
                      "%s must be a CUDA tensor on cuda:%d, got %s" % (name, dev, where))
    if dtypes is not None and t.dtype not in dtypes:
        raise PRError(PR_ERR_INVALID_ARG, call, "%s has dtype %s, expected %s" % (
            name, t.dtype, " or ".join(str(d) for d in dtypes)))
    if contiguous and not t.is_contiguous():
        raise PRError(PR_ERR_INVALID_ARG, call, "%s must be contiguous" % name)
    if numel is not None and t.numel() < numel:
        raise PRError(PR_ERR_INVALID_ARG, call, "%s holds %d elements, the call needs %d" % (
            name, t.numel(), numel))


def _host(call: str, name: str, t, optional: bool = False):
    if t is None:
        if optional:
            return
        raise PRError(PR_ERR_INVALID_ARG, call, "%s is required" % name)
    if isinstance(t, torch.Tensor):
        if t.is_cuda:
            raise PRError(PR_ERR_INVALID_ARG, call, "%s must be in host memory" % name)
        if not t.is_contiguous():
            raise PRError(PR_ERR_INVALID_ARG, call, "%s must be contiguous" % name)
    elif not isinstance(t, np.ndarray):
        raise PRError(PR_ERR_INVALID_ARG, call, "%s must be a host tensor" % name)


def _logits(call: str, dev: int, logits):
    if not isinstance(logits, torch.Tensor) or not logits.is_cuda or logits.device.index != dev:
        _dev(call, dev, "logits", logits)


def _ptr(t):
    if t is None:
        return None
    if isinstance(t, torch.Tensor):
        return t.data_ptr()  # an int: ctypes converts it for a c_void_p argument
    if isinstance(t, np.ndarray):
        return t.ctypes.data_as(ctypes.c_void_p)
    raise TypeError(type(t))


def _stream(stream):
    if stream is None:
        return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    if isinstance(stream, torch.cuda.Stream):
        return ctypes.c_void_p(stream.cuda_stream)
    return ctypes.c_void_p(int(stream))


def _dtype(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return PR_DTYPE_BF16
    if t.dtype == torch.float32:
        return PR_DTYPE_F32
    raise TypeError("logits must be bfloat16 or float32")


def _rows(logits: torch.Tensor, vocab):
    if logits.dim() != 2 or (logits.size(1) > 1 and logits.stride(1) != 1):
        raise ValueError("logits must be 2-D with unit stride along the vocabulary")
    stride = logits.stride(0) if logits.size(0) > 1 else logits.size(1)
    V = logits.size(1) if vocab is None else int(vocab)
    return V, max(stride, V)


def launch_count() -> int:
    return int(_lib.pr_launch_count())


def pr_status_string(status: int) -> str:
    return _lib.pr_status_string(status).decode()


# ---- context ---------------------------------------------------------------------

def pr_ctx_create(device: int = 0, max_rows: int = 0, max_requests: int = 0):
    h = ctypes.c_void_p()
    _check(_lib.pr_ctx_create(ctypes.byref(h), int(device), int(max_rows), int(max_requests)),
           "pr_ctx_create")
    _CTX_DEVICE[h.value] = int(device)
    return h


def pr_ctx_destroy(ctx):
    _check(_lib.pr_ctx_destroy(ctx), "pr_ctx_destroy")
    _CTX_DEVICE.pop(getattr(ctx, "value", ctx), None)


def pr_ctx_reset(ctx, stream=None):
    _check(_lib.pr_ctx_reset(ctx, _stream(stream)), "pr_ctx_reset")


def pr_ctx_set_option(ctx, option: int, value: int):
    _check(_lib.pr_ctx_set_option(ctx, int(option), int(value)), "pr_ctx_set_option")


def pr_ctx_kernel_times(ctx, cap: int = 32) -> list:
    """Per-kernel times (ms) of the last call made with PR_OPT_TIMING = 1."""
    buf = (ctypes.c_float * cap)()
    n = _I32(0)
    _check(_lib.pr_ctx_kernel_times(ctx, buf, cap, ctypes.byref(n)), "pr_ctx_kernel_times")
    return [float(buf[i]) for i in range(min(n.value, cap))]


def pr_ctx_flags(ctx, stream=None, clear: bool = False) -> int:
    v = ctypes.c_uint32(0)
    _check(_lib.pr_ctx_flags(ctx, _stream(stream), int(bool(clear)), ctypes.byref(v)),
           "pr_ctx_flags")
    return int(v.value)


def pr_last_error(ctx) -> int:
    """The context's flag word after all work on its device has finished."""
    v = ctypes.c_uint32(0)
    _check(_lib.pr_last_error(ctx, ctypes.byref(v)), "pr_last_error")
    return int(v.value)


# ---- verifier calls ------------------------------------------------------------------

_FLAG_T = (torch.int32,) + ((torch.uint32,) if hasattr(torch, "uint32") else ())


def pr_token_features(ctx, logits, chosen, topk: int = 20, offsets=None, feat=None, top2=None,
                      row_flags=None, vocab=None, stream=None):
    call = "pr_token_features"
    dev = _ctx_device(ctx)
    _logits(call, dev, logits)
    n = logits.size(0)
    V, stride = _rows(logits, vocab)
    d = logits.device
    feat = torch.empty(n, PR_NFEAT, dtype=torch.float32, device=d) if feat is None else feat
    top2 = torch.empty(n, 2, dtype=torch.int32, device=d) if top2 is None else top2
    row_flags = torch.empty(n, dtype=torch.int32, device=d) if row_flags is None else row_flags
    n_req = 0 if offsets is None else offsets.numel() - 1
    _dev(call, dev, "chosen", chosen, _I32_T, n)
    _dev(call, dev, "offsets", offsets, _I64_T, optional=True)
    _dev(call, dev, "feat", feat, _F32_T, n * PR_NFEAT)
    _dev(call, dev, "top2", top2, _I32_T, 2 * n)
    _dev(call, dev, "row_flags", row_flags, _FLAG_T, n)
    _check(_lib.pr_token_features(ctx, _ptr(logits), _dtype(logits), n, V, stride, _ptr(chosen),
                                  int(topk), _ptr(offsets), n_req, _ptr(feat), _ptr(top2),
                                  _ptr(row_flags), _stream(stream)), call)
    return feat, top2, row_flags


def _request_outputs(call, dev, n_req, score, ship, req_flags, agg=None, want_agg=False):
    d = torch.device("cuda", dev)
    score = torch.empty(n_req, dtype=torch.float32, device=d) if score is None else score
    ship = torch.empty(n_req, dtype=torch.uint8, device=d) if ship is None else ship
    req_flags = torch.empty(n_req, dtype=torch.int32, device=d) if req_flags is None else req_flags
    if agg is None and want_agg:
        agg = torch.empty(n_req, PR_NAGG, dtype=torch.float32, device=d)
    _dev(call, dev, "score", score, _F32_T, n_req)
    _dev(call, dev, "ship", ship, _U8_T, n_req)
    _dev(call, dev, "req_flags", req_flags, _FLAG_T, n_req)
    _dev(call, dev, "agg", agg, _F32_T, n_req * PR_NAGG, optional=True)
    return score, ship, req_flags, agg


def _offsets_and_w(call, dev, offsets, w, n_w=PR_NAGG):
    _dev(call, dev, "offsets", offsets, _I64_T)
    _dev(call, dev, "w", w, _F32_T, n_w)
    return offsets.numel() - 1


def pr_aggregate_score(ctx, feat, offsets, w, b: float, tau: float, row_flags=None, agg=None,
                       score=None, ship=None, req_flags=None, stream=None):
    call = "pr_aggregate_score"
    dev = _ctx_device(ctx)
    n_req = _offsets_and_w(call, dev, offsets, w)
    _dev(call, dev, "feat", feat, _F32_T)
    n_rows = feat.size(0) if feat.dim() > 0 else 0
    _dev(call, dev, "feat", feat, _F32_T, n_rows * PR_NFEAT)
    _dev(call, dev, "row_flags", row_flags, _FLAG_T, n_rows, optional=True)
    score, ship, req_flags, agg = _request_outputs(call, dev, n_req, score, ship, req_flags, agg,
                                                   want_agg=True)
    _check(_lib.pr_aggregate_score(ctx, _ptr(feat), _ptr(row_flags), n_rows, _ptr(offsets),
                                   n_req, _ptr(w), float(b), float(tau), _ptr(agg), _ptr(score),
                                   _ptr(ship), _ptr(req_flags), _stream(stream)), call)
    return agg, score, ship, req_flags


def pr_route(ctx, logits, chosen, offsets, w, b: float, tau: float, row_base: int = 0, score=None,
             ship=None, req_flags=None, agg=None, vocab=None, stream=None, want_agg: bool = True):
    call = "pr_route"
    dev = _ctx_device(ctx)
    _logits(call, dev, logits)
    n = logits.size(0)
    V, stride = _rows(logits, vocab)
    n_req = _offsets_and_w(call, dev, offsets, w)
    _dev(call, dev, "chosen", chosen, _I32_T, n)
    score, ship, req_flags, agg = _request_outputs(call, dev, n_req, score, ship, req_flags, agg,
                                                   want_agg)
    _check(_lib.pr_route(ctx, _ptr(logits), _dtype(logits), int(row_base), n, V, stride,
                         _ptr(chosen), _ptr(offsets), n_req, _ptr(w), float(b), float(tau),
                         _ptr(score), _ptr(ship), _ptr(req_flags), _ptr(agg), _stream(stream)),
           call)
    return score, ship, req_flags, agg


def pr_route_host(ctx, logits, chosen, offsets, w, b: float, tau: float, chunk_rows: int = 8192,
                  score=None, ship=None, req_flags=None, agg=None, vocab=None, stream=None):
    """Host tensors in, host tensors out (pinned host memory copies fastest)."""
    call = "pr_route_host"
    _host(call, "logits", logits)
    n = logits.size(0)
    V, stride = _rows(logits, vocab)
    n_req = offsets.numel() - 1
    score = torch.empty(n_req, dtype=torch.float32) if score is None else score
    ship = torch.empty(n_req, dtype=torch.uint8) if ship is None else ship
    req_flags = torch.empty(n_req, dtype=torch.int32) if req_flags is None else req_flags
    for name, t in (("chosen", chosen), ("offsets", offsets), ("w", w), ("score", score),
                    ("ship", ship), ("req_flags", req_flags)):
        _host(call, name, t)
    _host(call, "agg", agg, optional=True)
    _check(_lib.pr_route_host(ctx, _ptr(logits), _dtype(logits), n, V, stride, _ptr(chosen),
                              _ptr(offsets), n_req, _ptr(w), float(b), float(tau), int(chunk_rows),
                              _ptr(score), _ptr(ship), _ptr(req_flags), _ptr(agg),
                              _stream(stream)), call)
    return score, ship, req_flags, agg


def pr_route_noalloc(logits, chosen, offsets, w, b: float, tau: float, score, ship, req_flags,
                     agg=None, vocab=None, stream=None):
    """pr_route for callers that cannot allocate: no context, the library's
    fixed scratch, every output buffer supplied by the caller (CUDA tensors on
    the current device; anything else raises PRError before the library is
    called).  Batches above PR_NOALLOC_MAX_ROWS rows or PR_NOALLOC_MAX_REQUESTS
    requests raise PRError (invalid argument).  The offsets must cover the
    batch: when offsets[n_req] < n_rows the last request is reported with
    PR_FLAG_BAD_OFFSETS and a NaN score, and the rows after offsets[n_req] are
    not verified."""
    call = "pr_route_noalloc"
    if not torch.cuda.is_available():
        raise PRError(PR_ERR_UNSUPPORTED, call, "no CUDA device")
    dev = torch.cuda.current_device()
    _logits(call, dev, logits)
    n = logits.size(0)
    V, stride = _rows(logits, vocab)
    n_req = _offsets_and_w(call, dev, offsets, w)
    _dev(call, dev, "chosen", chosen, _I32_T, n)
    _request_outputs(call, dev, n_req, score, ship, req_flags, agg)
    _check(_lib.pr_route_noalloc(_ptr(logits), _dtype(logits), n, V, stride, _ptr(chosen),
                                 _ptr(offsets), n_req, _ptr(w), float(b), float(tau), _ptr(score),
                                 _ptr(ship), _ptr(req_flags), _ptr(agg), _stream(stream)), call)
    return score, ship, req_flags, agg


def pr_decode_step(ctx, logits, slot, chosen, eos, w, b: float, tau: float, score_out, ship_out,
                   slot_flags, agg_out=None, vocab=None, stream=None):
    """One decode step: row i belongs to slot[i].  The outputs are indexed by
    slot, so they must hold an entry for every slot index passed."""
    call = "pr_decode_step"
    dev = _ctx_device(ctx)
    _logits(call, dev, logits)
    n = logits.size(0)
    V, stride = _rows(logits, vocab)
    _dev(call, dev, "slot", slot, _I32_T, n)
    _dev(call, dev, "chosen", chosen, _I32_T, n)
    _dev(call, dev, "eos", eos, _U8_T, n)
    _dev(call, dev, "w", w, _F32_T, PR_NAGG)
    _dev(call, dev, "score_out", score_out, _F32_T)
    _dev(call, dev, "ship_out", ship_out, _U8_T)
    _dev(call, dev, "slot_flags", slot_flags, _FLAG_T)
    _dev(call, dev, "agg_out", agg_out, _F32_T, optional=True)
    _check(_lib.pr_decode_step(ctx, _ptr(logits), _dtype(logits), n, V, stride, _ptr(slot),
                               _ptr(chosen), _ptr(eos), _ptr(w), float(b), float(tau),
                               _ptr(score_out), _ptr(ship_out), _ptr(slot_flags), _ptr(agg_out),
                               _stream(stream)), call)


def pr_state_export(ctx) -> bytes:
    size = ctypes.c_size_t(0)
    _check(_lib.pr_state_export(ctx, None, ctypes.byref(size)), "pr_state_export")
    buf = ctypes.create_string_buffer(size.value)
    _check(_lib.pr_state_export(ctx, buf, ctypes.byref(size)), "pr_state_export")
    return buf.raw[:size.value]


def pr_state_import(ctx, state: bytes):
    buf = ctypes.create_string_buffer(state, len(state))
    _check(_lib.pr_state_import(ctx, buf, len(state)), "pr_state_import")


# ---- transformer scorer head ------------------------------------------------------------

def pr_head_param_count(n_layers: int) -> int:
    return int(_lib.pr_head_param_count(int(n_layers)))


def pr_head_score(ctx, feat, offsets, w, n_layers: int, tau: float, row_flags=None, score=None,
                  ship=None, req_flags=None, stream=None):
    call = "pr_head_score"
    dev = _ctx_device(ctx)
    n_w = pr_head_param_count(n_layers)
    n_req = _offsets_and_w(call, dev, offsets, w, max(n_w, 0))
    _dev(call, dev, "feat", feat, _F32_T)
    n_rows = feat.size(0) if feat.dim() > 0 else 0
    _dev(call, dev, "feat", feat, _F32_T, n_rows * PR_NFEAT)
    _dev(call, dev, "row_flags", row_flags, _FLAG_T, n_rows, optional=True)
    score, ship, req_flags, _ = _request_outputs(call, dev, n_req, score, ship, req_flags)
    _check(_lib.pr_head_score(ctx, _ptr(feat), _ptr(row_flags), n_rows, _ptr(offsets), n_req,
                              _ptr(w), int(n_layers), float(tau), _ptr(score), _ptr(ship),
                              _ptr(req_flags), _stream(stream)), call)
    return score, ship, req_flags


# ---- operating point and selective-prediction metrics ----------------------------------------

class PrSelective(ctypes.Structure):
    _fields_ = [("tau", ctypes.c_float), ("reserved", ctypes.c_int32), ("n_finite", _I64),
                ("k", _I64), ("n_ship", _I64), ("n_pos", _I64), ("auroc", ctypes.c_double),
                ("auarc", ctypes.c_double), ("acc_shipped", ctypes.c_double)]


def pr_selective_metrics(ctx, scores, q: float, labels=None, stream=None) -> dict:
    """Calibrate tau for ship fraction q on device scores; with device labels
    (uint8, non-zero = correct) also AUROC, AUARC and the shipped accuracy."""
    call = "pr_selective_metrics"
    dev = _ctx_device(ctx)
    _dev(call, dev, "scores", scores, _F32_T)
    _dev(call, dev, "labels", labels, _U8_T, scores.numel(), optional=True)
    res = PrSelective()
    _check(_lib.pr_selective_metrics(ctx, _ptr(scores), _ptr(labels), scores.numel(), float(q),
                                     ctypes.byref(res), _stream(stream)), "pr_selective_metrics")
    return {name: getattr(res, name) for name, _ in PrSelective._fields_ if name != "reserved"}


# ---- quantile-summary + MLP aggregator ----------------------------------------------------------

def pr_quantile_score(ctx, feat, offsets, w, tau: float, row_flags=None, summary=None, score=None,
                      ship=None, req_flags=None, want_summary: bool = True, stream=None):
    call = "pr_quantile_score"
    dev = _ctx_device(ctx)
    n_req = _offsets_and_w(call, dev, offsets, w, PR_QMLP_PARAMS)
    _dev(call, dev, "feat", feat, _F32_T)
    n_rows = feat.size(0) if feat.dim() > 0 else 0
    _dev(call, dev, "feat", feat, _F32_T, n_rows * PR_NFEAT)
    _dev(call, dev, "row_flags", row_flags, _FLAG_T, n_rows, optional=True)
    if summary is None and want_summary:
        summary = torch.empty(n_req, PR_QMLP_SUMMARY, dtype=torch.float32, device=feat.device)
    _dev(call, dev, "summary", summary, _F32_T, n_req * PR_QMLP_SUMMARY, optional=True)
    score, ship, req_flags, _ = _request_outputs(call, dev, n_req, score, ship, req_flags)
    _check(_lib.pr_quantile_score(ctx, _ptr(feat), _ptr(row_flags), n_rows, _ptr(offsets),
                                  n_req, _ptr(w), float(tau), _ptr(summary), _ptr(score),
                                  _ptr(ship), _ptr(req_flags), _stream(stream)), call)
    return score, ship, req_flags, summary


# ---- LM head fused with the row reduction ---------------------------------------------------

def pr_lmhead_features(ctx, hidden, weight, chosen, topk: int = 20, offsets=None, feat=None,
                       top2=None, row_flags=None, stream=None):
    """Row records of the logits weight @ hidden[r] (bf16 [n][d] and [V][d])
    without materialising the logits."""
    if hidden.dtype != torch.bfloat16 or weight.dtype != torch.bfloat16:
        raise TypeError("hidden and weight must be bfloat16")
    if not (hidden.is_contiguous() and weight.is_contiguous()) or hidden.size(1) != weight.size(1):
        raise ValueError("hidden [n][d] and weight [V][d] must be contiguous with the same d")
    call = "pr_lmhead_features"
    dev = _ctx_device(ctx)
    _dev(call, dev, "hidden", hidden)
    _dev(call, dev, "weight", weight)
    n, d = hidden.shape
    V = weight.size(0)
    feat = torch.empty(n, PR_NFEAT, dtype=torch.float32, device=hidden.device) if feat is None else feat
    top2 = torch.empty(n, 2, dtype=torch.int32, device=hidden.device) if top2 is None else top2
    row_flags = (torch.empty(n, dtype=torch.int32, device=hidden.device) if row_flags is None
                 else row_flags)
    n_req = 0 if offsets is None else offsets.numel() - 1
    _dev(call, dev, "chosen", chosen, _I32_T, n)
    _dev(call, dev, "offsets", offsets, _I64_T, optional=True)
    _dev(call, dev, "feat", feat, _F32_T, n * PR_NFEAT)
    _dev(call, dev, "top2", top2, _I32_T, 2 * n)
    _dev(call, dev, "row_flags", row_flags, _FLAG_T, n)
    _check(_lib.pr_lmhead_features(ctx, _ptr(hidden), _ptr(weight), n, d, V, _ptr(chosen),
                                   int(topk), _ptr(offsets), n_req, _ptr(feat), _ptr(top2),
                                   _ptr(row_flags), _stream(stream)), "pr_lmhead_features")
    return feat, top2, row_flags


def pr_lmhead_decode_step(ctx, hidden, weight, slot, chosen, eos, w, b: float, tau: float,
                          score_out, ship_out, slot_flags, agg_out=None, stream=None):
    """One decode step from the live slots' bf16 hidden states [n][d] and the
    bf16 LM head [V][d]: the logits stay on chip, each row's features are
    folded into its slot (outputs as pr_decode_step)."""
    if hidden.dtype != torch.bfloat16 or weight.dtype != torch.bfloat16:
        raise TypeError("hidden and weight must be bfloat16")
    if not (hidden.is_contiguous() and weight.is_contiguous()) or hidden.size(1) != weight.size(1):
        raise ValueError("hidden [n][d] and weight [V][d] must be contiguous with the same d")
    call = "pr_lmhead_decode_step"
    dev = _ctx_device(ctx)
    _dev(call, dev, "hidden", hidden)
    _dev(call, dev, "weight", weight)
    n, d = hidden.shape
    _dev(call, dev, "slot", slot, _I32_T, n)
    _dev(call, dev, "chosen", chosen, _I32_T, n)
    _dev(call, dev, "eos", eos, _U8_T, n)
    _dev(call, dev, "w", w, _F32_T, PR_NAGG)
    _dev(call, dev, "score_out", score_out, _F32_T)
    _dev(call, dev, "ship_out", ship_out, _U8_T)
    _dev(call, dev, "slot_flags", slot_flags, _FLAG_T)
    _dev(call, dev, "agg_out", agg_out, _F32_T, optional=True)
    _check(_lib.pr_lmhead_decode_step(ctx, _ptr(hidden), _ptr(weight), n, d, weight.size(0),
                                      _ptr(slot), _ptr(chosen), _ptr(eos), _ptr(w), float(b),
                                      float(tau), _ptr(score_out), _ptr(ship_out),
                                      _ptr(slot_flags), _ptr(agg_out), _stream(stream)),
           "pr_lmhead_decode_step")


def pr_selftest_wait(ctx, limit_ns: int) -> bool:
    """The library's bounded device wait on an mbarrier nothing completes;
    returns whether it completed (False: it ran out and raised PR_FLAG_TIMEOUT)."""
    done = _I32(-1)
    _check(_lib.pr_selftest_wait(ctx, int(limit_ns), ctypes.byref(done)), "pr_selftest_wait")
    return done.value == 1


# ---- the prompt pre-scorer (host CPU; Section 3.1, Eq. 2) ---------------------------------

def _texts(texts):
    """(buffer, pointers, n): the n texts as NUL-terminated byte strings side
    by side in one host buffer, and a uint64 array of their addresses (the C
    call's `const char* const*`).  The caller keeps both alive for the call."""
    texts = list(texts)
    n = len(texts)
    if n == 0:
        return b"", np.zeros(1, np.uint64), 0
    if all(isinstance(t, str) for t in texts):
        buf = ("\0".join(texts) + "\0").encode()
    else:
        buf = b"\0".join(t.encode() if isinstance(t, str) else bytes(t) for t in texts) + b"\0"
    a = np.frombuffer(buf, np.uint8)
    ends = np.flatnonzero(a == 0)
    if ends.size != n:
        raise PRError(PR_ERR_INVALID_ARG, "prescorer", "a text holds a NUL byte")
    ptrs = np.empty(n, np.uint64)
    ptrs[0] = 0
    ptrs[1:] = ends[:-1] + 1
    ptrs += np.uint64(a.ctypes.data)
    return buf, ptrs, n


def pr_prescorer_fit(docs, min_df: int = 1):
    """Vocabulary and smoothed idf of a corpus (str or bytes texts)."""
    buf, ptrs, n = _texts(docs)
    out = _P()
    _check(_lib.pr_prescorer_fit(ptrs.ctypes.data, n, int(min_df), ctypes.byref(out)),
           "pr_prescorer_fit")
    return out.value


def pr_prescorer_destroy(ps):
    _lib.pr_prescorer_destroy(ps)


def pr_prescorer_vocab_size(ps) -> int:
    return int(_lib.pr_prescorer_vocab_size(ps))


def pr_prescorer_term(ps, column: int):
    return _lib.pr_prescorer_term(ps, int(column))


def pr_prescorer_features(ps, prompt, cap: int = 4096):
    """(columns int32, values float32, token count) of one prompt."""
    p = prompt.encode() if isinstance(prompt, str) else bytes(prompt)
    cols = np.empty(max(1, cap), np.int32)
    vals = np.empty(max(1, cap), np.float32)
    nnz, length = _I32(), _I64()
    _check(_lib.pr_prescorer_features(ps, p, int(cap), cols.ctypes.data, vals.ctypes.data,
                                      ctypes.byref(nnz), ctypes.byref(length)),
           "pr_prescorer_features")
    return cols[:nnz.value].copy(), vals[:nnz.value].copy(), int(length.value)


def pr_prescorer_score(ps, prompts, n_images, w, b: float, n_threads: int = 0):
    """(p_pre float32 [n], logit float32 [n]) on the host; w: float32 [V + 2]."""
    buf, ptrs, n = _texts(prompts)
    img = np.ascontiguousarray(n_images, np.int32)
    wv = np.ascontiguousarray(w, np.float32)
    if img.shape != (n,) or wv.shape != (pr_prescorer_vocab_size(ps) + 2,):
        raise PRError(PR_ERR_INVALID_ARG, "pr_prescorer_score", "n_images or w has the wrong size")
    score = np.empty(max(1, n), np.float32)
    logit = np.empty(max(1, n), np.float32)
    _check(_lib.pr_prescorer_score(ps, ptrs.ctypes.data, img.ctypes.data, n, wv.ctypes.data,
                                   float(b), int(n_threads), score.ctypes.data, logit.ctypes.data),
           "pr_prescorer_score")
    return score[:n], logit[:n]
