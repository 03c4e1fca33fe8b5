"""Pins for the scorer-head oracle (CPU only): PyTorch's own encoder layer in
float64 with the same weights, closed forms, and permutation properties."""
import math

import numpy as np
import pytest
import torch

from oracle import head as H
from paper_2608_28726_gb300 import workloads as W


def test_parameter_count_matches_the_paper():
    """The experiments (Section 4.2) report a head of about 67k parameters."""
    assert H.n_params(2) == W.head_param_count(2) == 67329
    assert H.n_params(1) == 33857 and H.n_params(4) == 134273


def _torch_layer(L):
    layer = torch.nn.TransformerEncoderLayer(d_model=64, nhead=4, dim_feedforward=128,
                                             dropout=0.0, activation="relu", batch_first=True,
                                             norm_first=False, layer_norm_eps=1e-5,
                                             dtype=torch.float64)
    with torch.no_grad():
        layer.self_attn.in_proj_weight.copy_(torch.from_numpy(L["W_qkv"]))
        layer.self_attn.in_proj_bias.copy_(torch.from_numpy(L["b_qkv"]))
        layer.self_attn.out_proj.weight.copy_(torch.from_numpy(L["W_o"]))
        layer.self_attn.out_proj.bias.copy_(torch.from_numpy(L["b_o"]))
        layer.norm1.weight.copy_(torch.from_numpy(L["g1"]))
        layer.norm1.bias.copy_(torch.from_numpy(L["be1"]))
        layer.linear1.weight.copy_(torch.from_numpy(L["W_1"]))
        layer.linear1.bias.copy_(torch.from_numpy(L["b_1"]))
        layer.linear2.weight.copy_(torch.from_numpy(L["W_2"]))
        layer.linear2.bias.copy_(torch.from_numpy(L["b_2"]))
        layer.norm2.weight.copy_(torch.from_numpy(L["g2"]))
        layer.norm2.bias.copy_(torch.from_numpy(L["be2"]))
    return layer.eval()


@pytest.mark.parametrize("n_layers", [1, 2, 4])
@pytest.mark.parametrize("T", [1, 2, 17, 130])
def test_against_torch_encoder(n_layers, T):
    w = W.head_weights(n_layers, seed=7 + n_layers)
    p = H.unpack(w, n_layers)
    g = np.random.default_rng(T)
    X = np.stack([-g.exponential(2.0, T), g.uniform(0, 1, T), -g.uniform(0, 3, T),
                  np.arange(1, T + 1) / T], axis=1)
    x = X @ p["W_in"].T + p["b_in"] + H.positional_encoding(T)
    xt = torch.from_numpy(x)[None]
    with torch.no_grad():
        for L in p["layers"]:
            xt = _torch_layer(L)(xt)
    z_ref = float(xt[0].mean(0).numpy() @ p["w_out"] + p["b_out"])
    assert H.head_logit(X, w, n_layers) == pytest.approx(z_ref, abs=1e-11)


def test_positional_encoding_closed_form():
    pe = H.positional_encoding(50)
    assert np.allclose(pe[0, 0::2], 0.0) and np.allclose(pe[0, 1::2], 1.0)
    for t in (1, 7, 49):
        assert pe[t, 0] == pytest.approx(math.sin(t)) and pe[t, 1] == pytest.approx(math.cos(t))
        assert pe[t, 62] == pytest.approx(math.sin(t / 10000 ** (62 / 64)))
        assert pe[t, 63] == pytest.approx(math.cos(t / 10000 ** (62 / 64)))


def test_no_layers_is_linear():
    """With no encoder layer the logit is linear in the mean feature vector."""
    w = W.head_weights(0, seed=3)
    p = H.unpack(w, 0)
    g = np.random.default_rng(1)
    X = g.standard_normal((23, 4))
    z = H.head_logit(X, w, 0)
    pooled = p["W_in"] @ X.mean(0) + p["b_in"] + H.positional_encoding(23).mean(0)
    assert z == pytest.approx(float(pooled @ p["w_out"] + p["b_out"]), abs=1e-12)


def test_single_token_attention_returns_the_value():
    """T = 1: the softmax over one key is 1, so attention = the value projection."""
    w = W.head_weights(1, seed=5)
    p = H.unpack(w, 1)
    L = p["layers"][0]
    x = np.random.default_rng(2).standard_normal((1, 64))
    v = x @ L["W_qkv"][128:].T + L["b_qkv"][128:]
    a = v @ L["W_o"].T + L["b_o"]
    h = H.layer_norm(x + a, L["g1"], L["be1"])
    f = np.maximum(h @ L["W_1"].T + L["b_1"], 0) @ L["W_2"].T + L["b_2"]
    assert np.allclose(H.encoder_layer(x, L), H.layer_norm(h + f, L["g2"], L["be2"]), atol=1e-12)


def test_encoder_without_position_is_permutation_invariant():
    """Without positional encoding the encoder is permutation-equivariant and
    the mean pool invariant: a causal mask or a mixed-up head would break it."""
    w = W.head_weights(2, seed=9)
    g = np.random.default_rng(4)
    X = g.standard_normal((31, 4))
    perm = g.permutation(31)
    a = H.head_logit(X, w, 2, pe=False)
    b = H.head_logit(X[perm], w, 2, pe=False)
    assert a == pytest.approx(b, abs=1e-11)
    assert abs(H.head_logit(X, w, 2) - H.head_logit(X[perm], w, 2)) > 1e-6


def test_head_score_conventions():
    w = W.head_weights(2)
    g = np.random.default_rng(0)
    feat = g.standard_normal((10, 8))
    flags = np.zeros(10, np.uint32)
    flags[7] = 1
    off = np.array([0, 4, 4, 10])
    s, ship, fl = H.head_score(feat, flags, off, w, 2, 0.5)
    assert fl.tolist() == [0, 4, 1] and s[1] == 0.0 and ship[1] == 0
    assert np.isnan(s[2]) and ship[2] == 0
    z = H.head_logit(feat[0:4][:, list(H.FEATS)], w, 2)
    assert s[0] == pytest.approx(1 / (1 + math.exp(-z)), abs=1e-15)
    assert ship[0] == (1 if s[0] >= 0.5 else 0)
