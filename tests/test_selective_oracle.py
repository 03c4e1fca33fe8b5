"""Pins of the calibration / selective-metrics oracle (oracle/selective.py)
against facts that do not come from its own formulas: brute-force counting,
scikit-learn's AUROC, exhaustive averaging over the orders of tied groups, and
closed forms (Section 3.1 calibration, Section 4.1 metrics)."""
import itertools

import numpy as np
import pytest

from oracle import selective as sel


def tied_scores(n, seed, levels=20, nan_frac=0.0):
    g = np.random.Generator(np.random.PCG64(seed))
    s = np.round(g.random(n) * levels) / levels  # many exact ties
    y = g.random(n) < 0.3 + 0.4 * s             # correctness rises with the score
    if nan_frac:
        s[g.random(n) < nan_frac] = np.nan
    return s, y.astype(np.uint8)


@pytest.mark.parametrize("seed", [1, 2, 3])
def test_auroc_rank_formula_equals_pair_counting(seed):
    s, y = tied_scores(400, seed, nan_frac=0.05)
    assert sel.auroc_ranks(s, y) == pytest.approx(sel.auroc_pairs(s, y), abs=1e-12)
    assert sel.auroc(s, y) == pytest.approx(sel.auroc_pairs(s, y), abs=1e-12)


@pytest.mark.parametrize("seed", [11, 12])
def test_array_forms_equal_loop_forms(seed):
    s, y = tied_scores(20000, seed, levels=300, nan_frac=0.02)
    assert sel.auroc(s, y) == pytest.approx(sel.auroc_ranks(s, y), abs=1e-12)
    assert sel.auarc(s, y) == pytest.approx(sel.auarc_loop(s, y), abs=1e-12)


def test_auroc_matches_scikit_learn():
    metrics = pytest.importorskip("sklearn.metrics")
    for seed in (4, 5):
        s, y = tied_scores(1000, seed)
        assert sel.auroc(s, y) == pytest.approx(metrics.roc_auc_score(y, s), abs=1e-12)


def test_auroc_closed_forms():
    s = np.arange(10, dtype=float)
    assert sel.auroc(s, s >= 5) == 1.0      # every correct answer above every incorrect one
    assert sel.auroc(s, s < 5) == 0.0
    assert sel.auroc(np.ones(10), s >= 5) == 0.5  # all tied: chance
    assert np.isnan(sel.auroc(s, np.ones(10)))    # no incorrect answer


def brute_auarc(s, y):
    """Average of the plain AUARC over every order of each tied group."""
    s = np.asarray(s, float)
    y = np.asarray(y, float)
    levels = sorted(set(s.tolist()), reverse=True)
    groups = [list(np.flatnonzero(s == v)) for v in levels]
    total, count = 0.0, 0
    for perm in itertools.product(*[list(itertools.permutations(g)) for g in groups]):
        order = [i for grp in perm for i in grp]
        c = np.cumsum(y[order])
        total += np.mean(c / np.arange(1, len(order) + 1))
        count += 1
    return total / count


@pytest.mark.parametrize("seed", range(6))
def test_auarc_equals_average_over_tie_orders(seed):
    g = np.random.Generator(np.random.PCG64(100 + seed))
    n = 7
    s = g.integers(0, 3, size=n).astype(float)  # three levels: large tie groups
    y = g.integers(0, 2, size=n)
    assert sel.auarc_loop(s, y) == pytest.approx(brute_auarc(s, y), abs=1e-12)
    assert sel.auarc(s, y) == pytest.approx(brute_auarc(s, y), abs=1e-12)


def test_auarc_closed_forms():
    n, P = 50, 20
    s = np.arange(n, 0, -1, dtype=float)
    y = np.zeros(n)
    y[:P] = 1  # perfect ranking: the first P shipped are all correct
    expect = (P + sum(P / k for k in range(P + 1, n + 1))) / n
    assert sel.auarc(s, y) == pytest.approx(expect, abs=1e-12)
    assert sel.auarc(np.ones(n), y) == pytest.approx(P / n, abs=1e-12)  # no ranking: base rate
    assert sel.auarc(s, np.ones(n)) == 1.0


@pytest.mark.parametrize("q", [0.0, 0.05, 0.3, 0.5, 0.77, 1.0])
def test_calibration_ships_the_fraction(q):
    s, _ = tied_scores(500, 9, nan_frac=0.1)
    tau, k, n_ship = sel.calibrate(s, q)
    fin = s[np.isfinite(s)]
    assert k == min(int(np.floor(q * s.size + 0.5)), fin.size)
    if k == 0:
        assert tau == np.inf and n_ship == 0
        return
    assert n_ship == np.count_nonzero(fin >= tau) >= k   # ties at tau ship too
    assert np.count_nonzero(fin > tau) < k               # tau is the k-th largest
    assert tau in fin


def test_calibration_caps_at_the_finite_scores():
    s = np.array([0.9, np.nan, 0.2, np.nan])
    tau, k, n_ship = sel.calibrate(s, 1.0)
    assert (tau, k, n_ship) == (0.2, 2, 2)  # flagged requests never ship


def test_accuracy_at_threshold():
    s = np.array([0.1, 0.5, 0.5, 0.9, np.nan])
    y = np.array([0, 1, 0, 1, 1])
    rate, acc = sel.accuracy_at(s, y, 0.5)
    assert rate == pytest.approx(3 / 5) and acc == pytest.approx(2 / 3)
