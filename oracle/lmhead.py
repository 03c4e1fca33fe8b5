"""Float64 oracle of the LM head fused with the verifier's row features
(Pro-Router, Section 3.1: the per-token features need nothing beyond what the
small model's decoding already computes; its logits are x = W h).

TEST INFRASTRUCTURE ONLY: used by the tests and the benchmark's CPU baseline;
the product path never imports it.  The definition written out: the logits of
a row are the exact products of the bf16 hidden state with the bf16 LM-head
rows, summed in float64 (a float64 matrix product); the row's Eq. 3 features
are then the pinned float64 feature oracle (oracle.route / row_features) on
those logits, rounded to float32 at the hand-over.

Parity status: pinned by one-hot hidden states (the logits are a column of W:
a transposed operand fails), by linearity in h, and by the chosen token's
logit equal to its dot product; the features inherit the feature oracle's pins.
"""
from __future__ import annotations

import numpy as np

import oracle


def bf16_to_f64(bits) -> np.ndarray:
    """bf16 bit patterns (uint16) -> float64."""
    b = np.asarray(bits, np.uint16).astype(np.uint32) << 16
    return b.view(np.float32).astype(np.float64)


def logits(hidden_bits, weight_bits) -> np.ndarray:
    """x[r][v] = sum_k weight[v][k] hidden[r][k], exactly in float64 ([n_rows][V])."""
    H = bf16_to_f64(hidden_bits)
    W = bf16_to_f64(weight_bits)
    return H @ W.T


def features(hidden_bits, weight_bits, chosen, K: int = 20, offsets=None, n_threads: int = 1):
    """The verifier's feature records of the rows' logits: dict with feat,
    idx (top-2 indices), row_flags and the float64 logits."""
    x = logits(hidden_bits, weight_bits)
    n = x.shape[0]
    off = np.array([0, n], np.int64) if offsets is None else np.asarray(offsets, np.int64)
    o = oracle.route(x.astype(np.float32), chosen, off, np.zeros(11), 0.0, 0.5, K=K,
                     n_threads=n_threads)
    o["logits"] = x
    if offsets is None:
        o["feat"][:, 5] = 0.0  # no request layout: rho is not defined (the library writes 0)
    return o
