"""Float64 oracle of the quantile-summary + MLP aggregator (Pro-Router,
Section 4.2, Table 2: the verifier-architecture ablation's alternative to the
transformer head).

TEST INFRASTRUCTURE ONLY: used by the tests, the smoke check and the
benchmark's CPU baseline; the product path never imports it.

The paper names the variant only.  Readings (no figure or text gives more):

* Summary: for each of the four Eq. 3 features of a request, x_t in (l_t,
  m_t, h_t, rho_t) over its T rows, seven quantiles at the levels p = a / b in
  LEVELS; 4 x 7 = 28 numbers, feature-major.
* Quantile: the linear interpolation between order statistics (the textbook
  definition numpy and R call "linear" / type 7): with x_(0) <= ... <= x_(T-1),
  h = p (T - 1), q = x_(floor h) + (h - floor h) (x_(floor h + 1) - x_(floor h)).
  With p = a / b, floor h and the fraction come from the integer division of
  a (T - 1) by b, so both sides of a parity test take the same order
  statistics.
* MLP: 28 -> 64 -> 64 -> 1, ReLU after the two hidden layers; score =
  sigmoid(z), ship iff score >= tau.
* Flags and edge cases follow the other scorers: a row flagged non-finite or
  bad-token escalates its request (score NaN), an empty request scores 0.

Weights are one flat array (y = W x + b):
  W1[64][28] b1[64] W2[64][64] b2[64] w3[64] b3

Parity status: the summary is pinned against numpy.quantile(method="linear")
and closed forms (T = 1, arithmetic progressions, permutation invariance); the
MLP against torch.nn layers in float64 and the zero-weight case.
"""
from __future__ import annotations

import numpy as np

LEVELS = ((0, 1), (1, 10), (1, 4), (1, 2), (3, 4), (9, 10), (1, 1))
FEATS = (0, 1, 4, 5)  # record slots of l, m, h, rho
NQ = len(LEVELS)
NS = 4 * NQ           # summary length
H = 64                # hidden width


def n_params() -> int:
    return H * NS + H + H * H + H + H + 1


def unpack(w):
    w = np.asarray(w, np.float64).reshape(-1)
    if w.size != n_params():
        raise ValueError("expected %d weights, got %d" % (n_params(), w.size))
    o = 0

    def take(*shape):
        nonlocal o
        n = int(np.prod(shape))
        out = w[o:o + n].reshape(shape)
        o += n
        return out

    return dict(W1=take(H, NS), b1=take(H), W2=take(H, H), b2=take(H), w3=take(H),
                b3=take(1)[0])


def quantile(x, a: int, b: int) -> float:
    """Quantile at level a / b of the values x (linear interpolation)."""
    xs = np.sort(np.asarray(x, np.float64))
    T = xs.size
    lo, rem = divmod(a * (T - 1), b)
    if rem == 0:
        return float(xs[lo])
    hi = min(lo + 1, T - 1)
    return float(xs[lo] + (rem / b) * (xs[hi] - xs[lo]))


def summary(X) -> np.ndarray:
    """28-number summary of a request's T x 4 features (feature-major)."""
    X = np.asarray(X, np.float64).reshape(-1, 4)
    return np.array([quantile(X[:, f], a, b) for f in range(4) for (a, b) in LEVELS])


def mlp_logit(s, w) -> float:
    p = unpack(w)
    h1 = np.maximum(p["W1"] @ np.asarray(s, np.float64) + p["b1"], 0.0)
    h2 = np.maximum(p["W2"] @ h1 + p["b2"], 0.0)
    return float(p["w3"] @ h2 + p["b3"])


def quantile_score(feat, row_flags, offsets, w, tau: float):
    """Requests of a batch of row records (n_rows x 8): returns
    (score, ship, req_flags, summaries [n_req][28])."""
    feat = np.asarray(feat, np.float64)
    row_flags = np.asarray(row_flags, np.uint32)
    offsets = np.asarray(offsets, np.int64)
    n_req = offsets.size - 1
    score = np.zeros(n_req)
    ship = np.zeros(n_req, np.uint8)
    flags = np.zeros(n_req, np.uint32)
    summ = np.full((n_req, NS), np.nan)
    for r in range(n_req):
        lo, hi = offsets[r], offsets[r + 1]
        if hi == lo:
            flags[r] = 4
            continue
        fl = int(np.bitwise_or.reduce(row_flags[lo:hi]))
        flags[r] = fl
        if fl & 3:
            score[r] = np.nan
            continue
        s = summary(feat[lo:hi][:, FEATS])
        summ[r] = s
        z = mlp_logit(s, w)
        score[r] = 1.0 / (1.0 + np.exp(-z))
        ship[r] = 1 if score[r] >= tau else 0
    return score, ship, flags, summ
