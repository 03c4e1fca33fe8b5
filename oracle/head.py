"""Float64 oracle of the verifier's scorer head (Pro-Router, Section 3.1).

TEST INFRASTRUCTURE ONLY: used by the tests, the smoke check and the
benchmark's CPU baseline; the product path never imports it.  Plain numpy,
one request at a time, written from the description in Section 3.1: the
T x 4 feature sequence x_t = (l_t, m_t, h_t, rho_t) of a request goes through a
linear projection with positional encoding, a transformer encoder, a mean pool
over t and a sigmoid layer that outputs the shipping confidence.

Readings where the paper is silent (its figure with the head's sizes is not
available): d = 64, 4 heads, feed-forward width 128, post-norm encoder layers
(residual, then LayerNorm with eps 1e-5), ReLU, sinusoidal positional encoding
of the 0-based position t, L = 2 layers (1 and 4 in the paper's ablation).
These sizes give 67,329 parameters for L = 2, matching the paper's figure of
about 67 thousand (Section 4.2).

Weights are one flat float array in this order (y = x W^T + b convention):
  W_in[64][4] b_in[64]
  per layer: W_qkv[192][64] (rows: q, k, v) b_qkv[192] W_o[64][64] b_o[64]
             g1[64] be1[64] W_1[128][64] b_1[128] W_2[64][128] b_2[64] g2[64] be2[64]
  w_out[64] b_out[1]

Parity status: pinned against torch.nn.TransformerEncoderLayer in float64
(tests/test_head_oracle.py), against closed forms (T = 1, where attention
returns the value projection; zero encoder weights) and by permutation
properties of the encoder without positional encoding.
"""
from __future__ import annotations

import numpy as np

D, HEADS, DFF, DIN = 64, 4, 128, 4
DH = D // HEADS
LN_EPS = 1e-5
FEATS = (0, 1, 4, 5)  # record slots of l, m, h, rho


def layer_size() -> int:
    return 3 * D * D + 3 * D + D * D + D + 2 * D + DFF * D + DFF + D * DFF + D + 2 * D


def n_params(n_layers: int) -> int:
    return D * DIN + D + n_layers * layer_size() + D + 1


def unpack(w: np.ndarray, n_layers: int) -> dict:
    """Split the flat weight array into named float64 arrays."""
    w = np.asarray(w, np.float64).reshape(-1)
    if w.size != n_params(n_layers):
        raise ValueError("expected %d weights, got %d" % (n_params(n_layers), w.size))
    pos = 0

    def take(*shape):
        nonlocal pos
        n = int(np.prod(shape))
        out = w[pos:pos + n].reshape(shape)
        pos += n
        return out

    p = {"W_in": take(D, DIN), "b_in": take(D), "layers": []}
    for _ in range(n_layers):
        p["layers"].append(dict(
            W_qkv=take(3 * D, D), b_qkv=take(3 * D), W_o=take(D, D), b_o=take(D),
            g1=take(D), be1=take(D), W_1=take(DFF, D), b_1=take(DFF), W_2=take(D, DFF),
            b_2=take(D), g2=take(D), be2=take(D)))
    p["w_out"] = take(D)
    p["b_out"] = take(1)[0]
    return p


def positional_encoding(T: int) -> np.ndarray:
    """Sinusoidal encoding: PE[t, 2i] = sin(t / 10000^(2i/D)), PE[t, 2i+1] = cos(same)."""
    pe = np.zeros((T, D))
    t = np.arange(T, dtype=np.float64)[:, None]
    freq = 10000.0 ** (-np.arange(0, D, 2, dtype=np.float64) / D)
    pe[:, 0::2] = np.sin(t * freq)
    pe[:, 1::2] = np.cos(t * freq)
    return pe


def layer_norm(x, g, b):
    mu = x.mean(axis=-1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)
    return (x - mu) / np.sqrt(var + LN_EPS) * g + b


def softmax_rows(s):
    s = s - s.max(axis=-1, keepdims=True)
    e = np.exp(s)
    return e / e.sum(axis=-1, keepdims=True)


def encoder_layer(x, L):
    """One post-norm transformer encoder layer on a T x D sequence."""
    T = x.shape[0]
    qkv = x @ L["W_qkv"].T + L["b_qkv"]
    q, k, v = qkv[:, :D], qkv[:, D:2 * D], qkv[:, 2 * D:]
    heads = []
    for h in range(HEADS):
        sl = slice(h * DH, (h + 1) * DH)
        att = softmax_rows((q[:, sl] @ k[:, sl].T) / np.sqrt(DH))
        heads.append(att @ v[:, sl])
    a = np.concatenate(heads, axis=1) @ L["W_o"].T + L["b_o"]
    x = layer_norm(x + a, L["g1"], L["be1"])
    f = np.maximum(x @ L["W_1"].T + L["b_1"], 0.0) @ L["W_2"].T + L["b_2"]
    return layer_norm(x + f, L["g2"], L["be2"])


def head_logit(X: np.ndarray, w: np.ndarray, n_layers: int, pe: bool = True) -> float:
    """z for one request: X is T x 4 (l, m, h, rho); score = sigmoid(z)."""
    p = unpack(w, n_layers)
    X = np.asarray(X, np.float64).reshape(-1, DIN)
    x = X @ p["W_in"].T + p["b_in"]
    if pe:
        x = x + positional_encoding(X.shape[0])
    for L in p["layers"]:
        x = encoder_layer(x, L)
    return float(x.mean(axis=0) @ p["w_out"] + p["b_out"])


def head_score(feat: np.ndarray, row_flags, offsets, w, n_layers: int, tau: float):
    """Requests of a batch of row records (n_rows x 8, slots as the verifier's):
    returns (score, ship, req_flags) with the same conventions as the linear
    scorer (flagged rows escalate with NaN score; empty requests score 0)."""
    feat = np.asarray(feat, np.float64)
    row_flags = np.asarray(row_flags, np.uint32)
    offsets = np.asarray(offsets, np.int64)
    n_req = offsets.size - 1
    score = np.zeros(n_req)
    ship = np.zeros(n_req, np.uint8)
    flags = np.zeros(n_req, np.uint32)
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
        z = head_logit(feat[lo:hi][:, FEATS], w, n_layers)
        s = 1.0 / (1.0 + np.exp(-z))
        score[r] = s
        ship[r] = 1 if s >= tau else 0
    return score, ship, flags
