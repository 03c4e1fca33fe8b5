"""GPU parity of pr_lmhead_features (tcgen05 LM head with the row reduction in
its epilogue; Section 3.1) against the float64 oracle in oracle/lmhead.py.

Tolerance: each logit is a sum of d exact bf16 x bf16 products accumulated in
fp32 by the tensor cores; its error is below d * 2^-24 * sum |products| and
typically sqrt(d) times an ulp of the partial sums, ~1e-5 to 1e-4 for the
unit-scale logits here.  Features that are smooth in the logits (log p,
probabilities, entropies, LSE, x1) are compared at 1e-4 absolute + 1e-4
relative.  Top-2 indices are compared where the oracle's gaps between the
first three logits exceed 1e-3 (far above the logit error); elsewhere the
kernel's choice must be one of the tied tokens within that band."""
import numpy as np
import pytest
import torch

from oracle import lmhead
from tests._util import assert_close

pytestmark = pytest.mark.gpu

TOL = 1e-4


@pytest.fixture(scope="module")
def B():
    from paper_2608_28726_gb300 import binding
    return binding


@pytest.fixture(scope="module")
def ctx(B):
    c = B.pr_ctx_create(0, 16, 16)
    yield c
    B.pr_ctx_destroy(c)


def make(n, d, V, seed, wscale=None):
    """bf16 hidden states (row scale ~ U(0.5, 2)) and LM-head weights with
    N(0, (2 / sqrt(d))^2) entries: logits of a few units, as in the verifier's
    workloads."""
    g = torch.Generator().manual_seed(seed)
    h = torch.randn(n, d, generator=g) * (0.5 + 1.5 * torch.rand(n, 1, generator=g))
    w = torch.randn(V, d, generator=g) * (wscale if wscale else 2.0 / d ** 0.5)
    chosen = torch.randint(0, V, (n,), generator=g, dtype=torch.int32)
    return h.to(torch.bfloat16), w.to(torch.bfloat16), chosen


def bits(t):
    return t.contiguous().view(torch.int16).numpy().view(np.uint16)


def check(B, ctx, n, d, V, seed, topk=20, offsets=None, chosen_override=None):
    h, w, chosen = make(n, d, V, seed)
    if chosen_override is not None:
        chosen = chosen_override
    off_d = None if offsets is None else torch.from_numpy(np.asarray(offsets, np.int64)).cuda()
    feat, top2, rf = B.pr_lmhead_features(ctx, h.cuda(), w.cuda(), chosen.cuda(), topk,
                                          offsets=off_d)
    torch.cuda.synchronize()
    assert (B.pr_ctx_flags(ctx) & B.PR_FLAG_TIMEOUT) == 0
    o = lmhead.features(bits(h), bits(w), chosen.numpy(), K=topk, offsets=offsets)
    fg = feat.cpu().numpy()
    assert_close(fg, o["feat"], "features", rtol=TOL, atol=TOL)
    assert np.array_equal(rf.cpu().numpy().view(np.uint32), o["row_flags"])
    x = o["logits"]
    tg = top2.cpu().numpy()
    srt = -np.sort(-x, axis=1)
    for r in range(n):
        if V >= 3 and srt[r, 0] - srt[r, 1] > 1e-3 and srt[r, 1] - srt[r, 2] > 1e-3:
            assert list(tg[r]) == list(o["idx"][r]), r
        else:
            assert x[r, tg[r, 0]] >= srt[r, 0] - 1e-3
    if V == 1:
        assert (tg[:, 1] == -1).all()
    return fg, o


def test_lmhead_one_tile(B, ctx):
    check(B, ctx, 128, 64, 256, seed=1)


@pytest.mark.parametrize("n,d,V", [(1, 64, 256), (130, 128, 1000), (257, 192, 4097),
                                   (300, 520, 2304)])
def test_lmhead_ragged_shapes(B, ctx, n, d, V):
    # row tiles of 128 (CTA pairs of 256; n = 300 leaves one CTA without rows), vocabulary
    # tiles of 256 and K blocks of 128 (two boxes of 64) with ragged tails
    check(B, ctx, n, d, V, seed=n + d + V)


@pytest.mark.parametrize("topk", [1, 2, 20, 32])
def test_lmhead_topk(B, ctx, topk):
    check(B, ctx, 64, 256, 3000, seed=10 + topk, topk=topk)


def test_lmhead_flags_and_rho(B, ctx):
    n = 40
    chosen = torch.arange(n, dtype=torch.int32) * 37
    chosen[3] = -1
    chosen[7] = 10 ** 6  # outside the vocabulary
    fg, o = check(B, ctx, n, 128, 1500, seed=5, offsets=[0, 10, 10, 40], chosen_override=chosen)
    assert np.isnan(fg[3, 0]) and np.isnan(fg[7, 0])


def test_lmhead_large_vocab_and_hidden(B, ctx):
    """d = 3,584 (the small model's hidden size) and V = 151,936 on a few rows
    (on 152 SMs: 76 splits of 8 vocabulary tiles, the last split empty)."""
    check(B, ctx, 8, 3584, 151936, seed=7)


def test_lmhead_splits_without_tiles(B, ctx):
    """16 rows x V = 32,000: a small batch takes as many splits as fill one
    wave (76 on 152 SMs) of 2 of the 125 vocabulary tiles each, so the last 13
    splits hold no tile.  Their states stay empty and must leave the merge
    unchanged."""
    check(B, ctx, 16, 128, 32000, seed=21)


@pytest.mark.parametrize("n,d,V", [(3, 64, 1), (5, 64, 5), (7, 128, 17)])
def test_lmhead_vocab_below_k(B, ctx, n, d, V):
    """V < K = 20: the top-K sums run over the whole vocabulary, so the
    top-K entropy equals the full entropy; the lists' unused entries stay
    empty; V = 1 gives i2 = -1 and a margin p1 - p2 of 1."""
    fg, _ = check(B, ctx, n, d, V, seed=V)
    assert np.allclose(-fg[:, 4], fg[:, 3], rtol=TOL, atol=TOL)
    if V == 1:
        assert np.allclose(fg[:, 1:3], 1.0, atol=TOL)


def test_lmhead_is_deterministic(B, ctx):
    h, w, chosen = make(200, 256, 5000, 9)
    a = B.pr_lmhead_features(ctx, h.cuda(), w.cuda(), chosen.cuda())
    b = B.pr_lmhead_features(ctx, h.cuda(), w.cuda(), chosen.cuda())
    torch.cuda.synchronize()
    for x, y in zip(a, b):
        assert torch.equal(x.view(torch.int32), y.view(torch.int32))


def test_lmhead_full_batch_sampled_rows(B, ctx):
    """The benchmark's batch in its launch configuration (8,847 rows x d =
    3,584 x V = 151,936: 13 vocabulary splits, row pairs in bands of 18):
    rows at tile, pair and band boundaries and the last rows against the
    oracle, computed row by row."""
    from paper_2608_28726_gb300 import workloads as W
    n, d, V = 8847, 3584, 151936
    h, w, chosen = W.lmhead_inputs(n, d, V, device="cpu")
    feat, top2, rf = B.pr_lmhead_features(ctx, h.cuda(), w.cuda(), chosen.cuda(), 20)
    torch.cuda.synchronize()
    assert (B.pr_ctx_flags(ctx) & B.PR_FLAG_TIMEOUT) == 0
    rows = np.array([0, 1, 127, 128, 255, 256, 4607, 4608, 8703, 8704, 8845, 8846])
    o = lmhead.features(bits(h[rows]), bits(w), chosen.numpy()[rows], K=20)
    assert_close(feat.cpu().numpy()[rows], o["feat"], "features", rtol=TOL, atol=TOL)
    assert np.array_equal(rf.cpu().numpy()[rows].view(np.uint32), o["row_flags"])
    x = o["logits"]
    srt = -np.sort(-x, axis=1)
    tg = top2.cpu().numpy()[rows]
    for i in range(len(rows)):
        if srt[i, 0] - srt[i, 1] > 1e-3 and srt[i, 1] - srt[i, 2] > 1e-3:
            assert list(tg[i]) == list(o["idx"][i]), rows[i]
        else:
            assert x[i, tg[i, 0]] >= srt[i, 0] - 1e-3


def test_bounded_wait_runs_out_and_flags(B, ctx):
    """Failure detection without a stall: the kernels' bounded mbarrier wait,
    run on a barrier nothing completes with a 1 ms limit, gives up, raises
    PR_FLAG_TIMEOUT in the context flag word, and the context keeps working."""
    B.pr_ctx_flags(ctx, clear=True)
    assert B.pr_selftest_wait(ctx, 1_000_000) is False
    assert B.pr_ctx_flags(ctx, clear=True) & B.PR_FLAG_TIMEOUT
    assert B.pr_ctx_flags(ctx) == 0
    check(B, ctx, 130, 128, 1000, seed=77)  # asserts the flag stays clear
    with pytest.raises(B.PRError):
        B.pr_selftest_wait(ctx, -1)


def test_lmhead_exact_ties_across_splits(B, ctx):
    """A weight row duplicated at two far indices (other tiles, splits and
    column halves) and hidden states along it: the three logits are equal bit
    for bit (same products in the same order), so the top-2 must be the two
    lowest indices and the margin exactly 0, as in the oracle's (value desc,
    index asc) order."""
    n, d, V = 6, 256, 20000
    h, w, chosen = make(n, d, V, seed=91)
    w[7368] = w[17]  # column half 1 of its tile; 17 and 19999 are in half 0
    w[19999] = w[17]
    h[:3] = (w[17].float() * 4.0).to(torch.bfloat16)  # logit |w17|^2 * 4: far above the rest
    feat, top2, rf = B.pr_lmhead_features(ctx, h.cuda(), w.cuda(), chosen.cuda(), 20)
    torch.cuda.synchronize()
    o = lmhead.features(bits(h), bits(w), chosen.numpy(), K=20)
    assert_close(feat.cpu().numpy(), o["feat"], "features", rtol=TOL, atol=TOL)
    tg = top2.cpu().numpy()
    for r in range(3):
        assert list(tg[r]) == [17, 7368], tg[r]
        assert list(o["idx"][r]) == [17, 7368]
        assert feat[r, 2].item() == 0.0  # margin p1 - p2


def test_lmhead_decode_steps_match_oracle(B):
    """pr_lmhead_decode_step over a 40-step trace of 6 slots (requests of 1..14
    tokens, a new request when one ends): every finished request's
    aggregates, score, ship decision and flags against the float64 oracle of
    the request's rows (exact products of its hidden states and the head)."""
    import oracle
    n_slots, steps, d, V = 6, 40, 128, 3000
    g = np.random.default_rng(21)
    eos = np.zeros((steps, n_slots), np.uint8)
    reqs = []
    for s in range(n_slots):
        t = 0
        while t < steps:
            L = int(g.integers(1, 15))
            reqs.append((s, t, L))
            if t + L - 1 < steps:
                eos[t + L - 1, s] = 1
            t += L
    _, w_lm, _ = make(1, d, V, seed=301)
    hs = [make(n_slots, d, 8, seed=400 + t)[0] for t in range(steps)]
    ch = [torch.from_numpy(g.integers(0, V, n_slots).astype(np.int32)) for _ in range(steps)]
    w = (g.standard_normal(11) * 0.1).astype(np.float32)
    b = float(np.float32(g.standard_normal() * 0.1))
    ctx = B.pr_ctx_create(0, max_rows=16, max_requests=n_slots)
    try:
        slot = torch.arange(n_slots, dtype=torch.int32, device="cuda")
        dw, wd = torch.from_numpy(w).cuda(), w_lm.cuda()
        score = torch.full((n_slots,), -1.0, device="cuda")
        ship = torch.zeros(n_slots, dtype=torch.uint8, device="cuda")
        fl = torch.zeros(n_slots, dtype=torch.int32, device="cuda")
        agg = torch.zeros(n_slots, 11, device="cuda")
        B.pr_ctx_reset(ctx)
        ends = {}
        for t in range(steps):
            B.pr_lmhead_decode_step(ctx, hs[t].cuda(), wd, slot, ch[t].cuda(),
                                    torch.from_numpy(eos[t]).cuda(), dw, b, 0.5, score, ship, fl,
                                    agg_out=agg)
            for s in np.nonzero(eos[t])[0]:
                ends[(int(s), t)] = (score[s].item(), ship[s].item(), fl[s].item(),
                                     agg[s].cpu().numpy().copy())
        assert (B.pr_ctx_flags(ctx) & B.PR_FLAG_TIMEOUT) == 0
    finally:
        B.pr_ctx_destroy(ctx)
    wb = bits(w_lm)
    checked = 0
    for (s, t0, L) in reqs:
        if t0 + L > steps:
            continue
        hb = np.stack([bits(hs[t][s:s + 1])[0] for t in range(t0, t0 + L)])
        X = lmhead.logits(hb, wb).astype(np.float32)  # rounded at the hand-over, as lmhead.features
        C = np.array([int(ch[t][s]) for t in range(t0, t0 + L)], np.int32)
        o = oracle.route(X, C, np.array([0, L]), w.astype(np.float64), b, 0.5)
        sc, sh, f, ag = ends[(s, t0 + L - 1)]
        assert f == o["req_flags"][0]
        assert_close(ag, o["agg"][0], "decode agg", rtol=TOL, atol=TOL)
        assert_close(sc, o["score"][0], "decode score", rtol=TOL, atol=TOL)
        assert sh == o["ship"][0] or abs(o["score"][0] - 0.5) < 1e-4
        checked += 1
    assert checked >= 15


def test_lmhead_decode_step_arguments_and_bad_slot(B):
    """Host checks (hidden size not a multiple of 8, more live rows than
    slots) and a slot id outside the context flagged on the device."""
    ctx = B.pr_ctx_create(0, max_rows=16, max_requests=4)
    try:
        w11 = torch.zeros(11, device="cuda")
        out = (torch.zeros(4, device="cuda"), torch.zeros(4, dtype=torch.uint8, device="cuda"),
               torch.zeros(4, dtype=torch.int32, device="cuda"))
        h, w, chosen = make(2, 64, 300, seed=5)
        slot = torch.tensor([0, 9], dtype=torch.int32, device="cuda")
        eos = torch.ones(2, dtype=torch.uint8, device="cuda")
        B.pr_ctx_flags(ctx, clear=True)
        B.pr_lmhead_decode_step(ctx, h.cuda(), w.cuda(), slot, chosen.cuda(), eos, w11, 0.0, 0.5,
                                *out)
        torch.cuda.synchronize()
        assert B.pr_ctx_flags(ctx, clear=True) & B.PR_FLAG_BAD_SLOT
        h20 = torch.zeros(2, 20, dtype=torch.bfloat16, device="cuda")
        w20 = torch.zeros(300, 20, dtype=torch.bfloat16, device="cuda")
        with pytest.raises(B.PRError) as e:
            B.pr_lmhead_decode_step(ctx, h20, w20, slot, chosen.cuda(), eos, w11, 0.0, 0.5, *out)
        assert e.value.status == B.PR_ERR_INVALID_ARG
        h6, _, c6 = make(6, 64, 300, seed=6)
        with pytest.raises(B.PRError):
            B.pr_lmhead_decode_step(ctx, h6.cuda(), w.cuda(),
                                    torch.arange(6, dtype=torch.int32, device="cuda"), c6.cuda(),
                                    torch.zeros(6, dtype=torch.uint8, device="cuda"), w11, 0.0,
                                    0.5, *out)
    finally:
        B.pr_ctx_destroy(ctx)


@pytest.mark.parametrize("vocab", [(1 << 31) - 255, (1 << 31) - 1])
def test_lmhead_rejects_vocab_above_its_limit(B, ctx, vocab):
    """A vocabulary above PR_LMHEAD_MAX_VOCAB (2^31 - 256, where the last
    tile's 32-bit column arithmetic would pass 2^31) is refused by both calls
    before anything is queued; the pointers are valid but never read."""
    h, w, chosen = make(2, 64, 300, seed=3)
    h, w, chosen = h.cuda(), w.cuda(), chosen.cuda()
    feat = torch.zeros(2, 8, device="cuda")
    top2 = torch.zeros(2, 2, dtype=torch.int32, device="cuda")
    rf = torch.zeros(2, dtype=torch.int32, device="cuda")
    n0 = B.launch_count()
    st = B._lib.pr_lmhead_features(ctx, h.data_ptr(), w.data_ptr(), 2, 64, vocab,
                                   chosen.data_ptr(), 20, None, 0, feat.data_ptr(),
                                   top2.data_ptr(), rf.data_ptr(), None)
    assert st == B.PR_ERR_INVALID_ARG
    slot = torch.arange(2, dtype=torch.int32, device="cuda")
    eos = torch.zeros(2, dtype=torch.uint8, device="cuda")
    w11 = torch.zeros(11, device="cuda")
    st = B._lib.pr_lmhead_decode_step(ctx, h.data_ptr(), w.data_ptr(), 2, 64, vocab,
                                      slot.data_ptr(), chosen.data_ptr(), eos.data_ptr(),
                                      w11.data_ptr(), 0.0, 0.5, feat.data_ptr(), eos.data_ptr(),
                                      rf.data_ptr(), None, None)
    assert st == B.PR_ERR_INVALID_ARG
    assert B.launch_count() == n0
    assert B.PR_LMHEAD_MAX_VOCAB == (1 << 31) - 256
