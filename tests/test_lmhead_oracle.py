"""Pins of the LM-head + features oracle (oracle/lmhead.py, Section 3.1)."""
import numpy as np
import pytest

from oracle import lmhead


def bf16_bits(x):
    """float32 -> bf16 bit patterns by round-to-nearest-even (test helper)."""
    u = np.asarray(x, np.float32).view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return u.astype(np.uint16)


def test_bf16_decoding():
    bits = np.array([0x3F80, 0xC000, 0x7F80, 0x0000, 0x3E20], np.uint16)
    assert list(lmhead.bf16_to_f64(bits)) == [1.0, -2.0, np.inf, 0.0, 0.15625]


def test_one_hot_hidden_selects_a_weight_column():
    g = np.random.Generator(np.random.PCG64(1))
    W = bf16_bits(g.normal(size=(50, 16)))
    H = np.zeros((3, 16), np.uint16)
    for r, j in enumerate((0, 7, 15)):
        H[r, j] = 0x3F80  # 1.0
    x = lmhead.logits(H, W)
    for r, j in enumerate((0, 7, 15)):
        assert np.array_equal(x[r], lmhead.bf16_to_f64(W[:, j]))


def test_linear_in_the_hidden_state():
    g = np.random.Generator(np.random.PCG64(2))
    W = bf16_bits(g.normal(size=(40, 24)))
    h = g.normal(size=(2, 24)).astype(np.float32)
    x1 = lmhead.logits(bf16_bits(h), W)
    x2 = lmhead.logits(bf16_bits(2 * lmhead.bf16_to_f64(bf16_bits(h))), W)
    assert np.array_equal(x2, 2 * x1)


def test_features_of_the_logits():
    scipy_special = pytest.importorskip("scipy.special")
    g = np.random.Generator(np.random.PCG64(3))
    W = bf16_bits(g.normal(size=(300, 32)) * 0.3)
    H = bf16_bits(g.normal(size=(5, 32)))
    chosen = np.array([0, 17, 299, 5, 120], np.int32)
    o = lmhead.features(H, W, chosen, K=20)
    x = lmhead.logits(H, W)
    for r in range(5):
        lse = scipy_special.logsumexp(x[r])
        assert o["feat"][r, 0] == pytest.approx(x[r, chosen[r]] - lse, abs=1e-5)  # l = log p(y)
        assert o["feat"][r, 6] == pytest.approx(lse, abs=1e-5)
        assert o["idx"][r, 0] == int(np.argmax(x[r]))
    assert np.all(o["feat"][:, 5] == 0.0)
