"""GPU parity of pr_quantile_score (quantile summary + MLP, Section 4.2 Table 2)
against the float64 oracle in oracle/quantile.py.

Tolerance: order statistics are exact (the same rank on both sides); an
interpolated quantile is formed in fp32 from two fp32 values (error a few
ulp of its magnitude): 1e-6 absolute + 1e-6 relative.  The MLP sums 28 and 64
products of unit-scale terms in fp32 (~1e-6), so the score (slope <= 1/4) is
compared at 1e-5."""
import numpy as np
import pytest
import torch

from oracle import quantile as oq
from paper_2608_28726_gb300 import workloads
from tests._util import assert_close, assert_ship

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def B():
    from paper_2608_28726_gb300 import binding
    return binding


@pytest.fixture(scope="module")
def ctx(B):
    c = B.pr_ctx_create(0, 16, 16)
    yield c
    B.pr_ctx_destroy(c)


def run(B, ctx, feat, offsets, w, tau=0.5, row_flags=None):
    dev = torch.device("cuda")
    f = torch.from_numpy(np.ascontiguousarray(feat, np.float32)).to(dev)
    o = torch.from_numpy(np.ascontiguousarray(offsets, np.int64)).to(dev)
    wt = torch.from_numpy(np.ascontiguousarray(w, np.float32)).to(dev)
    rf = None if row_flags is None else torch.from_numpy(
        np.ascontiguousarray(row_flags, np.uint32).view(np.int32)).to(dev)
    score, ship, fl, summ = B.pr_quantile_score(ctx, f, o, wt, tau, row_flags=rf)
    torch.cuda.synchronize()
    return (score.cpu().numpy(), ship.cpu().numpy(), fl.cpu().numpy().view(np.uint32),
            summ.cpu().numpy())


def check(B, ctx, feat, offsets, tau=0.5, row_flags=None, seed=6001):
    w = workloads.qmlp_weights(seed)
    sg, pg, fg, mg = run(B, ctx, feat, offsets, w, tau, row_flags)
    rf = np.zeros(int(offsets[-1]), np.uint32) if row_flags is None else row_flags
    so, po, fo, mo = oq.quantile_score(feat.astype(np.float64), rf, offsets, w.astype(np.float64),
                                       tau)
    ok = ~np.isnan(mo[:, 0])
    assert_close(mg[ok], mo[ok], "summary", rtol=1e-6, atol=1e-6)
    assert_close(sg, so, "score", rtol=0.0, atol=1e-5)
    assert_ship(pg, po, so, tau)
    assert (fg == fo).all()
    return sg, so


def test_quantile_lengths_both_paths(B, ctx):
    # 1 .. 2,048 rows sort in shared memory; 2,049 and 5,000 use radix selection
    lengths = [1, 2, 3, 10, 11, 31, 32, 33, 257, 1000, 2048, 2049, 5000]
    feat, offsets = workloads.head_features(lengths, 7100)
    check(B, ctx, feat, offsets)


def test_quantile_ties_and_levels(B, ctx):
    lengths = [40, 41, 100, 3000]
    feat, offsets = workloads.head_features(lengths, 7200)
    feat[:, [0, 1, 4]] = np.round(feat[:, [0, 1, 4]] * 4) / 4  # heavy ties
    feat[offsets[1]:offsets[2], 1] = 0.5                        # one constant column
    for tau in (0.2, 0.5, 0.8):
        check(B, ctx, feat, offsets, tau=tau)


def test_quantile_full_response_and_ragged_layouts(B, ctx):
    wl = workloads.make("full")
    feat, offsets = workloads.head_features(wl.lengths, 7300)
    check(B, ctx, feat, offsets)
    wl = workloads.make("ragged")
    feat, offsets = workloads.head_features(wl.lengths, 7301)
    check(B, ctx, feat, offsets)


def test_quantile_flags_empty_and_bad_offsets(B, ctx):
    lengths = [5, 0, 7, 3, 0, 9]
    feat, offsets = workloads.head_features(lengths, 7400)
    rf = np.zeros(int(offsets[-1]), np.uint32)
    rf[offsets[2] + 1] = 1
    rf[offsets[3]] = 2
    rf[offsets[5] + 4] = 32
    w = workloads.qmlp_weights()
    sg, pg, fg, _ = run(B, ctx, feat, offsets, w, row_flags=rf)
    so, po, fo, _ = oq.quantile_score(feat.astype(np.float64), rf, offsets, w.astype(np.float64),
                                      0.5)
    assert_close(sg, so, "score", rtol=0.0, atol=1e-5)
    assert list(fg) == list(fo) == [0, 4, 1, 2, 4, 32]
    assert np.isnan(sg[2]) and np.isnan(sg[3]) and sg[1] == 0 and sg[4] == 0
    bad = offsets.copy()
    bad[-1] = offsets[-1] + 5
    sg, pg, fg, _ = run(B, ctx, feat, bad, w, row_flags=rf)
    assert fg[-1] == 8 and np.isnan(sg[-1]) and pg[-1] == 0


def test_quantile_is_deterministic(B, ctx):
    feat, offsets = workloads.head_features([50, 700, 2100], 7500)
    w = workloads.qmlp_weights()
    a = run(B, ctx, feat, offsets, w)
    b = run(B, ctx, feat, offsets, w)
    for x, y in zip(a, b):
        assert np.array_equal(x, y, equal_nan=True)
