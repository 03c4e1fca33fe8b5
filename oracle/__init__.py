"""Float64 CPU oracle of the token-aware verifier (Pro-Router, Section 3.1, Eq. 3).

TEST INFRASTRUCTURE ONLY: the tests, the smoke check and the benchmark's CPU
baseline leg may use this module; the product path never imports it.  It wraps
``pr_oracle.c`` (plain C, double precision) through ctypes and shares no code
with the CUDA library.

Parity status of each function (what pins it is in ``tests/test_oracle_pins.py``):
  row_features   pinned: closed forms (uniform, one-hot, two-way tie), brute
                 force against scipy/sorted() on tiny rows, invariances.
  request_score  pinned: T = 1, mean position fraction (T+1)/(2T), zero and
                 one-hot weights, threshold equality, permutation invariance.
  route          pinned: equals row_features + request_score composed by hand
                 on ragged batches; thread count does not change any output.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "pr_oracle.c")
LIB = os.path.join(HERE, "_build", "liboracle.so")

DTYPE_F32 = 0
DTYPE_BF16 = 1

FLAG_NONFINITE = 1
FLAG_BAD_CHOSEN = 2
FLAG_EMPTY_REQ = 4
FLAG_BAD_OFFSETS = 8

NFEAT = 8
NAGG = 11
# feature slots of a row record
LOGP, MAXP, MARGIN, ENT, TOPK, RHO, LSE, X1 = range(8)

_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (IEEE semantics: no fast-math, no FMA contraction)."""
    os.makedirs(os.path.dirname(LIB), exist_ok=True)
    if force or not os.path.exists(LIB) or os.path.getmtime(LIB) < os.path.getmtime(SRC):
        tmp = LIB + ".tmp%d" % os.getpid()
        subprocess.check_call([
            "gcc", "-std=c11", "-O2", "-ffp-contract=off", "-fno-fast-math", "-fPIC",
            "-shared", "-o", tmp, SRC, "-lm", "-lpthread"])
        os.replace(tmp, LIB)
    return LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            build()
            lib = ctypes.CDLL(LIB)
            P = ctypes.c_void_p
            i32, i64, f64 = ctypes.c_int32, ctypes.c_int64, ctypes.c_double
            lib.oracle_row_features.argtypes = [P, ctypes.c_int, i64, i32, i32, i32, P, P, P]
            lib.oracle_row_features.restype = ctypes.c_int
            lib.oracle_request_score.argtypes = [P, i64, P, P, f64, f64, P, P, P, P]
            lib.oracle_request_score.restype = ctypes.c_int
            lib.oracle_route.argtypes = [P, ctypes.c_int, i64, i64, i64, P, P, i32, i32, i32,
                                         P, f64, f64, i32, P, P, P, P, P, P, P]
            lib.oracle_route.restype = ctypes.c_int
            _lib = lib
    return _lib


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def _as_row_bytes(logits: np.ndarray):
    """Return (contiguous array, dtype code). bf16 rows arrive as uint16 bit patterns."""
    if logits.dtype == np.float32:
        return np.ascontiguousarray(logits), DTYPE_F32
    if logits.dtype == np.uint16:
        return np.ascontiguousarray(logits), DTYPE_BF16
    raise TypeError("logits must be float32 or uint16 (bfloat16 bit patterns)")


def row_features(row: np.ndarray, chosen: int, K: int = 20, renorm: bool = False):
    """Eq. 3 features of one logit row.

    Returns (feat[8] float64, idx[2] int32, flags) with feat slots
    [l, m, margin, H, h, rho(=0 here), LSE, x1] and idx = (i1, i2).
    """
    lib = _load()
    row, dt = _as_row_bytes(np.asarray(row).reshape(-1))
    feat = np.empty(NFEAT, np.float64)
    idx = np.empty(2, np.int32)
    flags = np.zeros(1, np.uint32)
    st = lib.oracle_row_features(_ptr(row), dt, row.size, int(chosen), int(K), int(bool(renorm)),
                                 _ptr(feat), _ptr(idx), _ptr(flags))
    if st != 0:
        raise ValueError("oracle_row_features failed with status %d" % st)
    return feat, idx, int(flags[0])


def request_score(feat: np.ndarray, row_flags, w, b: float, tau: float):
    """Pool T row records (T x 8, float64), score and threshold one request.

    Returns (agg[11], score, ship, flags).
    """
    lib = _load()
    feat = np.ascontiguousarray(feat, np.float64).reshape(-1, NFEAT)
    T = feat.shape[0]
    rf = np.ascontiguousarray(np.asarray(row_flags, np.uint32).reshape(-1))
    if rf.size != T:
        raise ValueError("row_flags must have one entry per row")
    w = np.ascontiguousarray(w, np.float64)
    agg = np.empty(NAGG, np.float64)
    score = np.empty(1, np.float64)
    ship = np.empty(1, np.uint8)
    flags = np.zeros(1, np.uint32)
    lib.oracle_request_score(_ptr(feat), T, _ptr(rf), _ptr(w), float(b), float(tau),
                             _ptr(agg), _ptr(score), _ptr(ship), _ptr(flags))
    return agg, float(score[0]), int(ship[0]), int(flags[0])


def route(logits: np.ndarray, chosen, offsets, w, b: float, tau: float, K: int = 20,
          renorm: bool = False, n_threads: int = 1, vocab: int | None = None):
    """Full-response verification of a ragged batch.

    ``logits`` is [n_rows, row_stride] float32 or uint16 (bf16 bits); the first
    ``vocab`` columns of each row (all of them by default) are the distribution.
    Returns a dict with feat, idx, row_flags, agg, score, ship, req_flags.
    """
    lib = _load()
    logits, dt = _as_row_bytes(np.asarray(logits))
    if logits.ndim != 2:
        raise ValueError("logits must be 2-D")
    n_rows, stride = logits.shape
    V = stride if vocab is None else int(vocab)
    if not 0 < V <= stride:
        raise ValueError("vocab must be in (0, row_stride]")
    chosen = np.ascontiguousarray(chosen, np.int32)
    offsets = np.ascontiguousarray(offsets, np.int64)
    n_req = offsets.size - 1
    w = np.ascontiguousarray(w, np.float64)
    out = dict(
        feat=np.empty((n_rows, NFEAT), np.float64),
        idx=np.empty((n_rows, 2), np.int32),
        row_flags=np.zeros(n_rows, np.uint32),
        agg=np.empty((n_req, NAGG), np.float64),
        score=np.empty(n_req, np.float64),
        ship=np.empty(n_req, np.uint8),
        req_flags=np.zeros(n_req, np.uint32),
    )
    st = lib.oracle_route(_ptr(logits), dt, n_rows, V, stride, _ptr(chosen), _ptr(offsets),
                          n_req, int(K), int(bool(renorm)), _ptr(w), float(b), float(tau),
                          int(n_threads), _ptr(out["feat"]), _ptr(out["idx"]),
                          _ptr(out["row_flags"]), _ptr(out["agg"]), _ptr(out["score"]),
                          _ptr(out["ship"]), _ptr(out["req_flags"]))
    if st != 0:
        raise ValueError("oracle_route failed with status %d" % st)
    return out
