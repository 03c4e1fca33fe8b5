"""GPU parity of the transformer scorer head (Section 3.1) against the float64
oracle in oracle/head.py, through the C ABI (pr_head_score).

Tolerance: the kernel computes in fp32 with fixed-order sums.  Each linear
layer sums at most 128 products of O(1) terms (relative rounding ~6e-8 per
term, so ~1e-6 per output in the worst case), LayerNorm rescales by ~1/sigma
of its unit-scale input, the softmax sums at most T positive terms; the
pre-sigmoid logit therefore carries an absolute error of at most ~1e-5 per
layer, and the score (sigmoid slope <= 1/4) is compared with
|score_gpu - score_oracle| <= 1e-5 for up to 4 layers.
"""
import numpy as np
import pytest
import torch

from oracle import head as ohead
from paper_2608_28726_gb300 import workloads
from tests._util import assert_close, assert_ship

pytestmark = pytest.mark.gpu

SCORE_ATOL = 1e-5


@pytest.fixture(scope="module")
def B():
    from paper_2608_28726_gb300 import binding
    return binding


@pytest.fixture(scope="module")
def ctx(B):
    c = B.pr_ctx_create(0, 1 << 16, 4096)
    yield c
    B.pr_ctx_destroy(c)


def run_head(B, ctx, feat, offsets, w, n_layers, tau=0.5, row_flags=None):
    dev = torch.device("cuda")
    f = torch.from_numpy(np.ascontiguousarray(feat, np.float32)).to(dev)
    o = torch.from_numpy(np.ascontiguousarray(offsets, np.int64)).to(dev)
    wt = torch.from_numpy(np.ascontiguousarray(w, np.float32)).to(dev)
    rf = None if row_flags is None else torch.from_numpy(
        np.ascontiguousarray(row_flags, np.uint32).view(np.int32)).to(dev)
    score, ship, fl = B.pr_head_score(ctx, f, o, wt, n_layers, tau, row_flags=rf)
    torch.cuda.synchronize()
    return score.cpu().numpy(), ship.cpu().numpy(), fl.cpu().numpy().view(np.uint32)


def oracle_head(feat, offsets, w, n_layers, tau=0.5, row_flags=None):
    n = offsets[-1]
    rf = np.zeros(n, np.uint32) if row_flags is None else row_flags
    return ohead.head_score(feat.astype(np.float64), rf, offsets, w.astype(np.float64), n_layers,
                            tau)


def check(B, ctx, lengths, n_layers, seed, tau=0.5, row_flags=None):
    feat, offsets = workloads.head_features(lengths, seed)
    w = workloads.head_weights(n_layers, seed=3001 + n_layers)
    sg, pg, fg = run_head(B, ctx, feat, offsets, w, n_layers, tau, row_flags)
    so, po, fo = oracle_head(feat, offsets, w, n_layers, tau, row_flags)
    assert_close(sg, so, "score", rtol=0.0, atol=SCORE_ATOL)
    assert_ship(pg, po, so, tau)
    assert (fg == fo).all()
    return sg, so


@pytest.mark.parametrize("n_layers", [1, 2, 4])
def test_head_matches_oracle_across_tiles(B, ctx, n_layers):
    # T = 1, exact chunk multiples, ragged tails, and several 32-row chunks
    lengths = [1, 2, 31, 32, 33, 64, 65, 100, 129, 257]
    check(B, ctx, lengths, n_layers, seed=4100 + n_layers)


def test_head_full_response_shapes(B, ctx):
    """64 requests of T ~ U{32..256}, the full-response batch's request mix."""
    g = np.random.Generator(np.random.PCG64(1002))
    lengths = g.integers(32, 256, size=64, endpoint=True)
    sg, so = check(B, ctx, lengths, 2, seed=4200)
    print("max |score err| = %.3g" % np.max(np.abs(sg - so)))


def test_head_long_requests(B, ctx):
    """The longest requests of the ragged batch (T = 1,024) and a 1,000-token decode request."""
    check(B, ctx, [1024, 1000, 513], 2, seed=4300)


def test_head_requests_past_one_round_of_query_blocks(B, ctx):
    """T = 2,100 and 1,300: more 128-query blocks than CTAs per (request,
    head), so a CTA takes a second block; 17 key chunks with a ragged last one."""
    check(B, ctx, [2100, 1, 1300, 128], 2, seed=4350)


def test_head_more_row_tiles_than_sms(B, ctx):
    """About 30,000 rows: more 128-row tiles than SMs, so the row kernels run
    in more than one wave of CTAs (each holds a whole SM's TMEM)."""
    g = np.random.Generator(np.random.PCG64(4400))
    lengths = g.integers(100, 200, size=200, endpoint=True)
    assert lengths.sum() > 128 * 160
    check(B, ctx, lengths, 2, seed=4401)


def test_head_thresholds(B, ctx):
    g = np.random.Generator(np.random.PCG64(7))
    lengths = g.integers(1, 80, size=40, endpoint=True)
    for tau in (0.05, 0.3, 0.5, 0.9, 0.999):
        check(B, ctx, lengths, 2, seed=4400, tau=tau)


def test_head_flags_empty_and_bad_offsets(B, ctx):
    lengths = [5, 0, 7, 3, 0, 9]
    feat, offsets = workloads.head_features(lengths, 4500)
    n = int(offsets[-1])
    rf = np.zeros(n, np.uint32)
    rf[offsets[2] + 1] = 1  # non-finite row in request 2
    rf[offsets[3]] = 2      # bad token id in request 3
    rf[offsets[5] + 4] = 32  # an unknown bit is passed through without escalating
    w = workloads.head_weights(2)
    sg, pg, fg = run_head(B, ctx, feat, offsets, w, 2, row_flags=rf)
    so, po, fo = oracle_head(feat, offsets, w, 2, row_flags=rf)
    assert_close(sg, so, "score", rtol=0.0, atol=SCORE_ATOL)
    assert list(fg) == list(fo) == [0, 4, 1, 2, 4, 32]
    assert np.isnan(sg[2]) and np.isnan(sg[3]) and sg[1] == 0 and sg[4] == 0
    assert pg[1] == pg[2] == pg[3] == pg[4] == 0
    # a request reaching past n_rows
    bad = offsets.copy()
    bad[-1] = n + 5
    sg, pg, fg = run_head(B, ctx, feat, bad, w, 2, row_flags=rf)
    assert fg[-1] == 8 and np.isnan(sg[-1]) and pg[-1] == 0
    assert_close(sg[:-1], so[:-1], "score", rtol=0.0, atol=SCORE_ATOL)


def test_head_is_deterministic_and_ignores_other_slots(B, ctx):
    lengths = [50, 77, 128]
    feat, offsets = workloads.head_features(lengths, 4600)
    w = workloads.head_weights(2)
    s1, _, _ = run_head(B, ctx, feat, offsets, w, 2)
    s2, _, _ = run_head(B, ctx, feat, offsets, w, 2)
    assert np.array_equal(s1, s2)
    other = feat.copy()
    other[:, [2, 3, 6, 7]] = 123.0
    s3, _, _ = run_head(B, ctx, other, offsets, w, 2)
    assert np.array_equal(s1, s3)


def test_head_chain_from_logits(B, ctx):
    """Logits -> Eq. 3 features -> head, GPU chain against oracle chain (tiny batch)."""
    import oracle
    wl = workloads.make("tiny", n_req=4, max_len=40)
    logits, chosen = workloads.rows(wl, 0, wl.n_rows)
    offs = torch.from_numpy(wl.offsets).cuda()
    feat, _, rf = B.pr_token_features(ctx, logits, chosen, 20, offsets=offs)
    w = workloads.head_weights(2)
    wt = torch.from_numpy(w).cuda()
    sg, pg, fg = B.pr_head_score(ctx, feat, offs, wt, 2, 0.5, row_flags=rf)
    torch.cuda.synchronize()
    ref = oracle.route(workloads.to_oracle_array(logits), chosen.cpu().numpy(), wl.offsets,
                       wl.w, wl.b, wl.tau)
    so, po, fo = ohead.head_score(ref["feat"], ref["row_flags"], wl.offsets, w.astype(np.float64),
                                  2, 0.5)
    assert_close(sg.cpu().numpy(), so, "score", rtol=0.0, atol=SCORE_ATOL)
    assert_ship(pg.cpu().numpy(), po, so, 0.5)


def test_head_rejects_bad_arguments(B, ctx):
    feat, offsets = workloads.head_features([4], 1)
    f = torch.from_numpy(feat).cuda()
    o = torch.from_numpy(offsets).cuda()
    w = torch.from_numpy(workloads.head_weights(2)).cuda()
    for nl in (0, 9):
        with pytest.raises(B.PRError):
            B.pr_head_score(ctx, f, o, w, nl, 0.5)
    with pytest.raises(B.PRError):
        B.pr_head_score(ctx, f, o, w[1:], 2, 0.5)  # weights not 16-byte aligned


def test_head_kernel_timing_option(B, ctx):
    """PR_OPT_TIMING reports one positive duration per kernel (2 L + 3) and
    leaves the results unchanged."""
    lengths = [40, 90, 200]
    feat, offsets = workloads.head_features(lengths, 4700)
    w = workloads.head_weights(2)
    s0, _, _ = run_head(B, ctx, feat, offsets, w, 2)
    B.pr_ctx_set_option(ctx, B.PR_OPT_TIMING, 1)
    try:
        s1, _, _ = run_head(B, ctx, feat, offsets, w, 2)
        times = B.pr_ctx_kernel_times(ctx)
    finally:
        B.pr_ctx_set_option(ctx, B.PR_OPT_TIMING, 0)
    assert np.array_equal(s0, s1)
    assert len(times) == 2 * 2 + 3 and all(t > 0 for t in times)
