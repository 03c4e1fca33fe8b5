"""Pins of the quantile-summary + MLP oracle (oracle/quantile.py, Section 4.2
Table 2): numpy's own quantile routine, closed forms, permutation invariance,
and torch's linear layers in float64."""
import numpy as np
import pytest

from oracle import quantile as oq


@pytest.mark.parametrize("T", [1, 2, 3, 10, 11, 31, 257, 1000])
def test_quantile_matches_numpy_linear(T):
    g = np.random.Generator(np.random.PCG64(T))
    x = g.normal(size=T)
    x[::5] = np.round(x[::5], 1)  # some ties
    for a, b in oq.LEVELS:
        assert oq.quantile(x, a, b) == pytest.approx(np.quantile(x, a / b, method="linear"),
                                                     abs=1e-12)


def test_quantile_closed_forms():
    assert [oq.quantile([3.5], a, b) for a, b in oq.LEVELS] == [3.5] * oq.NQ  # T = 1
    x = 2.0 + 0.5 * np.arange(21)  # arithmetic progression: q(p) = x0 + p (T - 1) step
    for a, b in oq.LEVELS:
        assert oq.quantile(x[::-1], a, b) == pytest.approx(2.0 + (a / b) * 20 * 0.5, abs=1e-12)
    assert oq.quantile([1.0, 5.0], 1, 4) == 2.0


def test_summary_layout_and_permutation_invariance():
    g = np.random.Generator(np.random.PCG64(7))
    X = g.normal(size=(40, 4))
    s = oq.summary(X)
    assert s.shape == (oq.NS,)
    assert np.array_equal(s, oq.summary(X[g.permutation(40)]))
    # feature-major: block f holds the quantiles of column f, min first, max last
    for f in range(4):
        assert s[f * oq.NQ] == X[:, f].min() and s[f * oq.NQ + oq.NQ - 1] == X[:, f].max()


def test_mlp_matches_torch():
    torch = pytest.importorskip("torch")
    g = np.random.Generator(np.random.PCG64(8))
    w = g.normal(size=oq.n_params()) * 0.2
    p = oq.unpack(w)
    net = torch.nn.Sequential(torch.nn.Linear(oq.NS, oq.H), torch.nn.ReLU(),
                              torch.nn.Linear(oq.H, oq.H), torch.nn.ReLU(),
                              torch.nn.Linear(oq.H, 1)).double()
    with torch.no_grad():
        net[0].weight.copy_(torch.from_numpy(p["W1"]))
        net[0].bias.copy_(torch.from_numpy(p["b1"]))
        net[2].weight.copy_(torch.from_numpy(p["W2"]))
        net[2].bias.copy_(torch.from_numpy(p["b2"]))
        net[4].weight.copy_(torch.from_numpy(p["w3"][None, :]))
        net[4].bias.fill_(p["b3"])
        for _ in range(5):
            s = g.normal(size=oq.NS)
            assert oq.mlp_logit(s, w) == pytest.approx(
                float(net(torch.from_numpy(s)[None, :])[0, 0]), abs=1e-12)


def test_mlp_zero_weights_and_score_conventions():
    w = np.zeros(oq.n_params())
    w[-1] = 0.75
    assert oq.mlp_logit(np.ones(oq.NS), w) == 0.75
    feat = np.zeros((6, 8))
    offsets = np.array([0, 3, 3, 6])
    flags = np.array([0, 0, 0, 0, 1, 0], np.uint32)
    score, ship, fl, summ = oq.quantile_score(feat, flags, offsets, w, 0.5)
    assert score[0] == pytest.approx(1 / (1 + np.exp(-0.75))) and ship[0] == 1
    assert score[1] == 0 and fl[1] == 4 and ship[1] == 0   # empty
    assert np.isnan(score[2]) and fl[2] == 1 and ship[2] == 0  # flagged row
