"""GPU parity of pr_selective_metrics (coverage calibration, AUROC, AUARC;
Section 3.1 and Section 4.1) against the float64 oracle in oracle/selective.py.

Counts, the threshold and the AUROC numerator are integers or copied scores:
exact.  AUROC divides an exact integer by P N in double: 1e-12.  AUARC sums n
double terms C_k / k in a different order than numpy: the rounding is below
n * 2^-53 relative, 1e-9 here."""
import numpy as np
import pytest
import torch

from oracle import selective as sel

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def B():
    from paper_2608_28726_gb300 import binding
    return binding


@pytest.fixture(scope="module")
def ctx(B):
    c = B.pr_ctx_create(0, 16, 4)
    yield c
    B.pr_ctx_destroy(c)


def make(n, seed, levels=0, nan_frac=0.0, neg_zero=False):
    """float32 scores (continuous, or `levels` values with many ties) and labels
    whose rate of correct answers rises with the score."""
    g = np.random.Generator(np.random.PCG64(seed))
    if levels:
        s = (np.floor(g.random(n) * levels) / levels).astype(np.float32)
    else:
        s = g.random(n).astype(np.float32)
    y = (g.random(n) < 0.2 + 0.6 * s).astype(np.uint8)
    if nan_frac:
        bad = g.random(n) < nan_frac
        s[bad] = np.where(g.random(bad.sum()) < 0.5, np.nan, np.inf).astype(np.float32)
    if neg_zero:
        s[::7] = np.float32(-0.0)
        s[3::7] = np.float32(0.0)
    return s, y


def run(B, ctx, s, y, q):
    ds = torch.from_numpy(s).cuda()
    dy = None if y is None else torch.from_numpy(y).cuda()
    return B.pr_selective_metrics(ctx, ds, q, labels=dy)


def check(g, s, y, q):
    o = sel.selective_metrics(s, y, q)
    assert g["n_finite"] == o["n_finite"]
    assert g["k"] == o["k"]
    assert g["n_ship"] == o["n_ship"]
    assert np.float32(g["tau"]) == np.float32(o["tau"])
    if y is None:
        assert np.isnan(g["auroc"]) and np.isnan(g["auarc"]) and g["n_pos"] == 0
        return
    assert g["n_pos"] == o["n_pos"]
    for name, tol in (("auroc", 1e-12), ("auarc", 1e-9), ("acc_shipped", 1e-12)):
        a, b = g[name], o[name]
        assert (np.isnan(a) and np.isnan(b)) or abs(a - b) <= tol, (name, a, b)


@pytest.mark.parametrize("n", [1, 2, 31, 2047, 2048, 2049, 4095, 4096, 4097, 12289, 100003])
def test_selective_matches_oracle_sizes(B, ctx, n):
    # tile edges (2,048 items per tile) and ragged tails
    s, y = make(n, seed=n, levels=97, nan_frac=0.03)
    # q * n + 1/2 lands on an integer for some of these: the rounding of q itself
    # must be the oracle's (double)
    for q in (0.0, 0.05, 0.1, 0.3, 0.5, 0.7, 0.77, 0.9, 1.0):
        check(run(B, ctx, s, y, q), s, y, q)


@pytest.mark.parametrize("kind", ["continuous", "few_levels", "one_level", "signed_zero"])
def test_selective_tie_structures(B, ctx, kind):
    n = 30000
    if kind == "continuous":
        s, y = make(n, 1)
    elif kind == "few_levels":
        s, y = make(n, 2, levels=3)
    elif kind == "one_level":
        s, y = make(n, 3)
        s[:] = np.float32(0.625)
    else:
        s, y = make(n, 4, neg_zero=True)
    for q in (0.1, 0.5, 0.9):
        check(run(B, ctx, s, y, q), s, y, q)


def test_selective_degenerate_pools(B, ctx):
    s, y = make(5000, 5)
    check(run(B, ctx, s, None, 0.4), s, None, 0.4)          # calibration only
    ones = np.ones_like(y)
    check(run(B, ctx, s, ones, 0.4), s, ones, 0.4)           # no incorrect answer: AUROC NaN
    bad = np.full(1000, np.nan, np.float32)
    g = run(B, ctx, bad, y[:1000], 0.5)
    assert g["n_finite"] == 0 and g["k"] == 0 and g["tau"] == np.inf and np.isnan(g["auarc"])
    g = B.pr_selective_metrics(ctx, torch.empty(0, device="cuda"), 0.5)
    assert g["n_finite"] == 0 and g["tau"] == np.inf
    with pytest.raises(B.PRError):
        run(B, ctx, s, y, 1.5)


def test_selective_is_deterministic(B, ctx):
    s, y = make(200000, 6, levels=1000)
    a = run(B, ctx, s, y, 0.3)
    b = run(B, ctx, s, y, 0.3)
    assert a == b


def test_selective_full_pool(B, ctx):
    """2^24 scores (the benchmark's pool), continuous with a few repeated values."""
    n = 1 << 24
    s, y = make(n, 7)
    s[::1000] = np.float32(0.5)
    check(run(B, ctx, s, y, 0.7), s, y, 0.7)

