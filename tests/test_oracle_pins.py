"""Pins for the float64 oracle (CPU only).

The oracle is checked against facts that do not come from itself: closed forms
of the Eq. 3 features on rows whose distribution is known exactly, brute force
through library routines (scipy's logsumexp / entropy, Python's sorted) on tiny
rows with many ties, and invariances of the definitions.  Each test is chosen
so that a plausible slip in the oracle (a dropped term, a sign, the tie rule,
raw vs renormalised top-K, the >= of the ship rule) fails at least one of them.
"""
import itertools
import math

import numpy as np
import pytest
import scipy.special
import scipy.stats

import oracle
from oracle import ENT, LOGP, LSE, MARGIN, MAXP, RHO, TOPK, X1

NEG_INF = np.float32(-np.inf)


def bf16_bits(x):
    """Round-to-nearest-even float32 -> bfloat16 bit patterns (test helper)."""
    u = np.asarray(x, np.float32).view(np.uint32).astype(np.uint64)
    r = ((u + 0x7FFF + ((u >> 16) & 1)) >> 16).astype(np.uint16)
    return r


def bf16_value(bits):
    return (bits.astype(np.uint32) << 16).view(np.float32)


# ---- closed forms ------------------------------------------------------------

@pytest.mark.parametrize("V", [1, 2, 7, 20, 21, 1000, 32000])
@pytest.mark.parametrize("c", [0.0, -3.5, 17.25])
@pytest.mark.parametrize("K", [1, 20])
def test_uniform_row(V, c, K):
    """All logits equal: p = 1/V, H = ln V, m = 1/V, l = -ln V, margin = 0,
    h = -(min(K,V)/V) ln V, LSE = c + ln V, i1 = 0, i2 = 1."""
    row = np.full(V, c, np.float32)
    f, idx, fl = oracle.row_features(row, chosen=V // 2, K=K)
    assert fl == 0
    lnV = math.log(V)
    assert f[ENT] == pytest.approx(lnV, abs=1e-12)
    assert f[MAXP] == pytest.approx(1.0 / V, rel=1e-12)
    assert f[LOGP] == pytest.approx(-lnV, abs=1e-12)
    assert f[MARGIN] == (1.0 if V == 1 else 0.0)
    assert f[TOPK] == pytest.approx(-(min(K, V) / V) * lnV, abs=1e-12)
    assert f[LSE] == pytest.approx(c + lnV, abs=1e-12)
    assert f[X1] == c
    assert idx[0] == 0
    assert idx[1] == (1 if V >= 2 else -1)


@pytest.mark.parametrize("V,K", [(5, 3), (20, 20), (100, 20), (100, 7)])
def test_uniform_row_renormalised(V, K):
    """Renormalised top-K of a uniform row is uniform over K tokens: entropy ln K."""
    row = np.zeros(V, np.float32)
    f, _, _ = oracle.row_features(row, 0, K=K, renorm=True)
    assert f[TOPK] == pytest.approx(-math.log(min(K, V)), abs=1e-12)


@pytest.mark.parametrize("V,spike", [(1, 0), (2, 1), (9, 0), (9, 8), (1000, 517)])
def test_one_hot_masked(V, spike):
    """One finite token, the rest -inf (masked): H = 0, m = 1, l(spike) = 0,
    margin = 1, h = 0; i2 is the lowest index other than the spike."""
    row = np.full(V, NEG_INF)
    row[spike] = 3.0
    f, idx, fl = oracle.row_features(row, chosen=spike)
    assert fl == 0
    assert f[ENT] == 0.0 and f[MAXP] == 1.0 and f[LOGP] == 0.0
    assert f[MARGIN] == 1.0 and f[TOPK] == 0.0 and f[LSE] == 3.0
    assert idx[0] == spike
    assert idx[1] == (-1 if V == 1 else (1 if spike == 0 else 0))
    if V > 1:
        other = 1 if spike == 0 else 0
        f2, _, _ = oracle.row_features(row, chosen=other)
        assert f2[LOGP] == -np.inf


def test_one_hot_by_gap():
    """A gap of 200 in float32 is a one-hot row to double precision."""
    row = np.full(4096, -200.0, np.float32)
    row[1234] = 0.0
    f, idx, _ = oracle.row_features(row, chosen=1234)
    assert f[MAXP] == pytest.approx(1.0, abs=1e-80)
    assert f[ENT] == pytest.approx(0.0, abs=1e-80)
    assert f[LOGP] == pytest.approx(0.0, abs=1e-80)
    assert idx[0] == 1234 and idx[1] == 0


@pytest.mark.parametrize("i,j", [(0, 1), (3, 10), (10, 3)])
def test_two_way_tie(i, j):
    """Two equal finite logits, rest masked: H = ln 2, m = 1/2, margin = 0,
    h = -ln 2 (K >= 2) and the lower index comes first."""
    row = np.full(16, NEG_INF)
    row[i] = row[j] = -1.5
    f, idx, _ = oracle.row_features(row, chosen=j)
    assert f[ENT] == pytest.approx(math.log(2), abs=1e-15)
    assert f[MAXP] == 0.5 and f[MARGIN] == 0.0
    assert f[TOPK] == pytest.approx(-math.log(2), abs=1e-15)
    assert f[LOGP] == pytest.approx(-math.log(2), abs=1e-15)
    assert list(idx) == [min(i, j), max(i, j)]


def test_known_probabilities():
    """x = ln p for p = (0.1, 0.2, 0.3, 0.4): every feature is a closed form of p.
    K = 2 keeps only 0.4 and 0.3, which pins the top-K cut and the sign of h."""
    p = np.array([0.1, 0.2, 0.3, 0.4])
    row = np.log(p).astype(np.float32)
    # the float32 rounding of ln p moves p by < 1e-7 relative
    f, idx, _ = oracle.row_features(row, chosen=0, K=2)
    assert f[LOGP] == pytest.approx(math.log(0.1), abs=1e-6)
    assert f[MAXP] == pytest.approx(0.4, abs=1e-7)
    assert f[MARGIN] == pytest.approx(0.1, abs=1e-7)
    assert f[ENT] == pytest.approx(-sum(q * math.log(q) for q in p), abs=1e-6)
    assert f[TOPK] == pytest.approx(0.4 * math.log(0.4) + 0.3 * math.log(0.3), abs=1e-6)
    assert f[LSE] == pytest.approx(0.0, abs=1e-6)
    assert list(idx) == [3, 2]
    fr, _, _ = oracle.row_features(row, chosen=0, K=2, renorm=True)
    q = np.array([0.4, 0.3]) / 0.7
    assert fr[TOPK] == pytest.approx(float(np.sum(q * np.log(q))), abs=1e-6)


# ---- brute force through library routines -------------------------------------

def _library_features(x, chosen, K, renorm=False):
    """Independent statement through scipy and sorted() (no oracle code)."""
    x = np.asarray(x, np.float64)
    V = x.size
    lse = scipy.special.logsumexp(x)
    p = scipy.special.softmax(x)
    H = scipy.stats.entropy(p)
    order = sorted(range(V), key=lambda v: (-x[v], v))
    top = [p[v] for v in order[:K]]
    if renorm:
        top = list(np.array(top) / np.sum(top))
    h = -scipy.stats.entropy(top) if renorm else float(sum(q * math.log(q) for q in top if q > 0))
    i2 = order[1] if V > 1 else -1
    return dict(logp=math.log(p[chosen]), maxp=p[order[0]],
                margin=p[order[0]] - (p[i2] if V > 1 else 0.0), ent=H, topk=h, lse=lse,
                x1=x[order[0]], i1=order[0], i2=i2)


@pytest.mark.parametrize("V,K", [(1, 20), (2, 1), (3, 2), (4, 2), (4, 20), (5, 3)])
def test_exhaustive_small_integer_rows(V, K):
    """Every row in {-2..2}^V (ties everywhere) against the library statement."""
    vals = [-2.0, -1.0, 0.0, 1.0, 2.0]
    for tup in itertools.product(vals, repeat=V):
        row = np.array(tup, np.float32)
        for chosen in range(V):
            f, idx, fl = oracle.row_features(row, chosen, K=K)
            ref = _library_features(row, chosen, K)
            assert fl == 0
            assert idx[0] == ref["i1"] and idx[1] == ref["i2"], tup
            assert f[LOGP] == pytest.approx(ref["logp"], abs=1e-12)
            assert f[MAXP] == pytest.approx(ref["maxp"], abs=1e-12)
            assert f[MARGIN] == pytest.approx(ref["margin"], abs=1e-12)
            assert f[ENT] == pytest.approx(ref["ent"], abs=1e-12)
            assert f[TOPK] == pytest.approx(ref["topk"], abs=1e-12)
            assert f[LSE] == pytest.approx(ref["lse"], abs=1e-12)
            assert f[X1] == ref["x1"]


@pytest.mark.parametrize("seed", range(6))
@pytest.mark.parametrize("renorm", [False, True])
def test_random_rows_against_library(seed, renorm):
    g = np.random.default_rng(seed)
    V = int(g.integers(2, 400))
    K = int(g.integers(1, 25))
    row = (g.standard_normal(V) * g.uniform(0.5, 6)).astype(np.float32)
    if seed % 2:
        row[g.integers(0, V, size=3)] = row.max()  # ties at the top
    chosen = int(g.integers(0, V))
    f, idx, _ = oracle.row_features(row, chosen, K=K, renorm=renorm)
    ref = _library_features(row, chosen, K, renorm)
    assert (idx[0], idx[1]) == (ref["i1"], ref["i2"])
    for k, slot in [("logp", LOGP), ("maxp", MAXP), ("margin", MARGIN), ("ent", ENT),
                    ("topk", TOPK), ("lse", LSE)]:
        assert f[slot] == pytest.approx(ref[k], rel=1e-10, abs=1e-12), k


# ---- invariances ---------------------------------------------------------------

def test_bf16_upcast_is_exact():
    g = np.random.default_rng(7)
    bits = bf16_bits(g.standard_normal(3000) * 3)
    vals = bf16_value(bits)
    fa, ia, _ = oracle.row_features(bits, 11)
    fb, ib, _ = oracle.row_features(vals, 11)
    assert np.array_equal(fa, fb, equal_nan=True) and np.array_equal(ia, ib)


def test_shift_invariance():
    """Adding an exactly representable constant shifts only LSE and x1."""
    g = np.random.default_rng(3)
    row = np.round(g.standard_normal(5000) * 64) / 64  # exact in float32 after +1024
    a = row.astype(np.float32)
    b = (row + 1024.0).astype(np.float32)
    fa, ia, _ = oracle.row_features(a, 42)
    fb, ib, _ = oracle.row_features(b, 42)
    for s in (LOGP, MAXP, MARGIN, ENT, TOPK):
        assert fb[s] == pytest.approx(fa[s], abs=1e-11)
    assert fb[LSE] - fa[LSE] == pytest.approx(1024.0, abs=1e-9)
    assert list(ia) == list(ib)


def test_permutation_moves_indices():
    g = np.random.default_rng(5)
    row = g.permutation(np.arange(2000, dtype=np.float32) / 97.0)  # distinct values
    perm = g.permutation(2000)
    f, idx, _ = oracle.row_features(row, 17)
    fp, idxp, _ = oracle.row_features(row[perm], int(np.where(perm == 17)[0][0]))
    inv = np.argsort(perm)
    assert list(idxp) == [inv[idx[0]], inv[idx[1]]]
    for s in (LOGP, MAXP, MARGIN, ENT, TOPK, LSE):
        assert fp[s] == pytest.approx(f[s], abs=1e-12)


def test_masked_tokens_equal_removed_tokens():
    """-inf tokens behave as if absent (p = 0, 0 log 0 = 0); indices remap."""
    g = np.random.default_rng(9)
    row = g.standard_normal(300).astype(np.float32)
    mask = g.random(300) < 0.4
    masked = row.copy()
    masked[mask] = -np.inf
    keep = np.where(~mask)[0]
    c = int(keep[5])
    fm, im, _ = oracle.row_features(masked, c)
    fr, ir, _ = oracle.row_features(row[keep], 5)
    for s in (LOGP, MAXP, MARGIN, ENT, TOPK, LSE):
        assert fm[s] == pytest.approx(fr[s], abs=1e-12)
    assert list(im) == [keep[ir[0]], keep[ir[1]]]


@pytest.mark.parametrize("bad", [np.nan, np.inf])
def test_nonfinite_row(bad):
    row = np.zeros(50, np.float32)
    row[7] = bad
    f, idx, fl = oracle.row_features(row, 3)
    assert fl & oracle.FLAG_NONFINITE
    assert np.all(np.isnan(f)) and list(idx) == [-1, -1]


def test_all_masked_row_is_nonfinite():
    f, idx, fl = oracle.row_features(np.full(10, NEG_INF), 0)
    assert fl == oracle.FLAG_NONFINITE and np.all(np.isnan(f))


@pytest.mark.parametrize("chosen", [-1, 64, 1 << 30])
def test_bad_chosen(chosen):
    row = np.linspace(-1, 1, 64).astype(np.float32)
    f, idx, fl = oracle.row_features(row, chosen)
    ok, _, _ = oracle.row_features(row, 0)
    assert fl == oracle.FLAG_BAD_CHOSEN and math.isnan(f[LOGP])
    assert np.array_equal(f[1:], ok[1:])


# ---- requests ------------------------------------------------------------------

def _rand_feats(g, T):
    f = np.zeros((T, 8))
    f[:, LOGP] = -g.exponential(2.0, T)
    f[:, MAXP] = g.uniform(0, 1, T)
    f[:, MARGIN] = g.uniform(0, 1, T) * f[:, MAXP]
    f[:, ENT] = g.uniform(0, 8, T)
    f[:, TOPK] = -g.uniform(0, 3, T)
    f[:, RHO] = np.arange(1, T + 1) / T
    return f


def test_single_row_request_equals_row():
    g = np.random.default_rng(0)
    f = _rand_feats(g, 1)
    agg, s, ship, fl = oracle.request_score(f, [0], np.zeros(11), 0.0, 0.5)
    r = f[0]
    expect = [r[LOGP], r[LOGP], r[MAXP], r[MAXP], r[MARGIN], r[MARGIN], -r[ENT], -r[ENT],
              r[TOPK], r[TOPK], 1.0]
    assert np.allclose(agg, expect, rtol=0, atol=1e-15)


@pytest.mark.parametrize("T", [1, 2, 3, 10, 64, 1000])
def test_mean_position_fraction(T):
    """mean over t of t/T is (T+1)/(2T)."""
    g = np.random.default_rng(T)
    agg, _, _, _ = oracle.request_score(_rand_feats(g, T), np.zeros(T), np.zeros(11), 0.0, 0.5)
    assert agg[10] == pytest.approx((T + 1) / (2 * T), abs=1e-14)


def test_pool_against_numpy():
    g = np.random.default_rng(1)
    f = _rand_feats(g, 37)
    agg, _, _, _ = oracle.request_score(f, np.zeros(37), np.zeros(11), 0.0, 0.5)
    cols = [f[:, LOGP], f[:, MAXP], f[:, MARGIN], -f[:, ENT], f[:, TOPK]]
    for k, c in enumerate(cols):
        assert agg[2 * k] == pytest.approx(np.mean(c), abs=1e-13)
        assert agg[2 * k + 1] == np.min(c)


def test_zero_scorer_ships_at_half():
    """z = 0 gives score 0.5, and the ship rule is score >= tau (Section 3.1)."""
    g = np.random.default_rng(2)
    f = _rand_feats(g, 5)
    _, s, ship, _ = oracle.request_score(f, np.zeros(5), np.zeros(11), 0.0, 0.5)
    assert s == 0.5 and ship == 1
    _, s, ship, _ = oracle.request_score(f, np.zeros(5), np.zeros(11), 0.0, 0.5 + 1e-12)
    assert ship == 0


@pytest.mark.parametrize("j", range(11))
def test_one_hot_weight_selects_aggregate(j):
    g = np.random.default_rng(10 + j)
    f = _rand_feats(g, 9)
    w = np.zeros(11)
    w[j] = 1.0
    agg, s, _, _ = oracle.request_score(f, np.zeros(9), w, 0.25, 0.5)
    assert s == pytest.approx(scipy.special.expit(agg[j] + 0.25), abs=1e-15)


def test_flagged_rows_escalate():
    g = np.random.default_rng(4)
    f = _rand_feats(g, 4)
    for flag in (oracle.FLAG_NONFINITE, oracle.FLAG_BAD_CHOSEN):
        agg, s, ship, fl = oracle.request_score(f, [0, flag, 0, 0], np.ones(11), 5.0, 0.1)
        assert ship == 0 and math.isnan(s) and np.all(np.isnan(agg)) and fl == flag


# ---- batches -------------------------------------------------------------------

def _batch(seed, lengths, V=257, dtype="f32"):
    g = np.random.default_rng(seed)
    n = int(np.sum(lengths))
    x = (g.standard_normal((n, V)) * 2).astype(np.float32)
    if dtype == "bf16":
        x = bf16_bits(x)
    chosen = g.integers(0, V, n).astype(np.int32)
    off = np.concatenate([[0], np.cumsum(lengths)]).astype(np.int64)
    w = (g.standard_normal(11) * 0.1).astype(np.float32).astype(np.float64)
    return x, chosen, off, w


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_route_is_composition(dtype):
    lengths = [3, 0, 1, 7, 2]
    x, chosen, off, w = _batch(11, lengths, dtype=dtype)
    out = oracle.route(x, chosen, off, w, 0.05, 0.5, n_threads=3)
    for r in range(len(lengths)):
        lo, hi = off[r], off[r + 1]
        feats, flags = [], []
        for t, row in enumerate(range(lo, hi), start=1):
            f, idx, fl = oracle.row_features(x[row], chosen[row])
            f[RHO] = t / (hi - lo)
            assert np.array_equal(out["feat"][row], f)
            assert list(out["idx"][row]) == list(idx)
            feats.append(f)
            flags.append(fl)
        if hi == lo:
            assert out["req_flags"][r] == oracle.FLAG_EMPTY_REQ
            assert out["score"][r] == 0.0 and out["ship"][r] == 0
            continue
        agg, s, ship, fl = oracle.request_score(np.array(feats), flags, w, 0.05, 0.5)
        assert np.array_equal(out["agg"][r], agg) and out["score"][r] == s
        assert out["ship"][r] == ship and out["req_flags"][r] == fl


def test_route_thread_count_invariant():
    x, chosen, off, w = _batch(12, [5, 9, 1, 30, 4])
    a = oracle.route(x, chosen, off, w, 0.0, 0.5, n_threads=1)
    b = oracle.route(x, chosen, off, w, 0.0, 0.5, n_threads=7)
    for k in a:
        assert np.array_equal(a[k], b[k], equal_nan=True), k


def test_route_request_permutation_invariant():
    """Reordering whole requests reorders the per-request results only."""
    lengths = [4, 6, 2, 5]
    x, chosen, off, w = _batch(13, lengths)
    a = oracle.route(x, chosen, off, w, 0.0, 0.5)
    perm = [2, 0, 3, 1]
    rows = np.concatenate([np.arange(off[r], off[r + 1]) for r in perm])
    off2 = np.concatenate([[0], np.cumsum([lengths[r] for r in perm])])
    b = oracle.route(x[rows], chosen[rows], off2, w, 0.0, 0.5)
    for i, r in enumerate(perm):
        assert np.array_equal(b["agg"][i], a["agg"][r]) and b["ship"][i] == a["ship"][r]


def test_route_bad_offsets_flagged():
    x, chosen, off, w = _batch(14, [2, 2])
    off = np.array([0, 3, 2], np.int64)
    out = oracle.route(x, chosen, off, w, 0.0, 0.5)
    assert out["req_flags"][1] == oracle.FLAG_BAD_OFFSETS and out["ship"][1] == 0


def test_route_vocab_narrower_than_stride():
    x, chosen, off, w = _batch(15, [3, 2], V=64)
    chosen = chosen % 50
    a = oracle.route(x, chosen, off, w, 0.0, 0.5, vocab=50)
    b = oracle.route(np.ascontiguousarray(x[:, :50]), chosen, off, w, 0.0, 0.5)
    for k in a:
        assert np.array_equal(a[k], b[k], equal_nan=True), k
