"""GPU parity of the three verifier calls against the float64 oracle, on
small inputs that still span several tiles and a ragged tail, plus the edge
cases: odd and tiny vocabularies, unaligned rows, every K, masked / tied /
non-finite rows, bad ids and offsets, row splits, chunking, decode steps,
checkpoints, the host-memory path and buffer guards.  Everything goes
through the C ABI (ctypes binding)."""
import numpy as np
import pytest
import torch

import oracle
from _util import as_oracle, assert_close, assert_ship, random_rows

pytestmark = pytest.mark.gpu

B = None  # the binding, imported once a GPU is known to be present


@pytest.fixture(scope="module")
def ctx():
    global B
    assert torch.cuda.is_available(), "the GPU tests need a CUDA device"
    from paper_2608_28726_gb300 import build
    build.build()
    from paper_2608_28726_gb300 import binding
    B = binding
    h = B.pr_ctx_create(0, max_rows=1 << 16, max_requests=1024)
    yield h
    B.pr_ctx_destroy(h)


def _set(ctx, split=0, renorm=0, topk=20):
    B.pr_ctx_set_option(ctx, B.PR_OPT_SPLIT, split)
    B.pr_ctx_set_option(ctx, B.PR_OPT_TOPK_RENORM, renorm)
    B.pr_ctx_set_option(ctx, B.PR_OPT_TOPK, topk)


def _oracle_rows(x, chosen, K=20, renorm=False, vocab=None):
    xs = as_oracle(x)
    ch = chosen.cpu().numpy()
    feats, idxs, flags = [], [], []
    for r in range(xs.shape[0]):
        row = xs[r] if vocab is None else xs[r, :vocab]
        f, i, fl = oracle.row_features(row, int(ch[r]), K=K, renorm=renorm)
        feats.append(f)
        idxs.append(i)
        flags.append(fl)
    return np.array(feats), np.array(idxs), np.array(flags)


def _check_features(feat, top2, rflags, of, oi, ofl, what):
    feat = feat.cpu().numpy()
    top2 = top2.cpu().numpy()
    rflags = rflags.cpu().numpy().astype(np.uint32)
    assert np.array_equal(rflags, ofl), "%s flags %s vs %s" % (what, rflags, ofl)
    assert np.array_equal(top2, oi), "%s top2 differ at rows %s" % (
        what, np.argwhere((top2 != oi).any(1)).ravel()[:8])
    for s in (oracle.LOGP, oracle.MAXP, oracle.MARGIN, oracle.ENT, oracle.TOPK, oracle.LSE,
              oracle.X1):
        assert_close(feat[:, s], of[:, s], "%s feature %d" % (what, s))


# ---- per-token features ----------------------------------------------------------------

# split 0 lets the library choose (a cluster per row for these small batches);
# split 1 forces the persistent warp-specialised kernel
@pytest.mark.parametrize("split", [0, 1])
@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("V", [1, 2, 7, 8, 9, 31, 160, 1000, 4097, 32000, 70001])
def test_features_vocab_sizes(ctx, dtype, V, split):
    _set(ctx, split=split)
    x, ch = random_rows(24, V, dtype, seed=V)
    feat, top2, rf = B.pr_token_features(ctx, x, ch, topk=20)
    of, oi, ofl = _oracle_rows(x, ch)
    _check_features(feat, top2, rf, of, oi, ofl, "V=%d" % V)


@pytest.mark.parametrize("split", [0, 1])
@pytest.mark.parametrize("K", [1, 2, 3, 19, 20, 21, 32])
@pytest.mark.parametrize("renorm", [0, 1])
def test_features_topk(ctx, K, renorm, split):
    _set(ctx, renorm=renorm, split=split)
    x, ch = random_rows(16, 3001, torch.bfloat16, seed=100 + K)
    feat, top2, rf = B.pr_token_features(ctx, x, ch, topk=K)
    of, oi, ofl = _oracle_rows(x, ch, K=K, renorm=bool(renorm))
    _check_features(feat, top2, rf, of, oi, ofl, "K=%d renorm=%d" % (K, renorm))
    _set(ctx)


@pytest.mark.parametrize("split", [0, 1])
@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("shift", [1, 3])
def test_features_unaligned_rows(ctx, dtype, shift, split):
    """Row starts off the 16-byte grid take the element-load path."""
    _set(ctx, split=split)
    V = 2053
    base, ch = random_rows(12, V + shift + 5, dtype, seed=7 + shift)
    x = base[:, shift:shift + V]  # row stride V + shift + 5, start offset `shift` elements
    assert x.stride(0) == V + shift + 5
    feat, top2, rf = B.pr_token_features(ctx, x, ch % V, topk=20)
    of, oi, ofl = _oracle_rows(x.contiguous(), ch % V)
    _check_features(feat, top2, rf, of, oi, ofl, "unaligned")
    _set(ctx)


def test_features_vocab_narrower_than_stride(ctx):
    x, ch = random_rows(10, 5000, torch.float32, seed=3)
    V = 4321
    feat, top2, rf = B.pr_token_features(ctx, x, ch % V, topk=20, vocab=V)
    of, oi, ofl = _oracle_rows(x, ch % V, vocab=V)
    _check_features(feat, top2, rf, of, oi, ofl, "vocab<stride")


def _special_rows(V, dtype):
    rows, chosen = [], []
    neg = float("-inf")
    r = torch.full((V,), 1.25)                      # uniform
    rows.append(r); chosen.append(3)
    r = torch.full((V,), neg); r[V // 3] = 2.0      # one-hot by masking
    rows.append(r); chosen.append(V // 3)
    r = torch.full((V,), neg); r[5] = r[V - 2] = -1.0  # two-way tie, rest masked
    rows.append(r); chosen.append(V - 2)
    r = torch.randn(V); r[torch.rand(V) < 0.5] = neg   # half masked
    rows.append(r); chosen.append(int(torch.nonzero(r > neg)[0]))
    r = torch.randn(V); r[17] = float("nan")        # NaN
    rows.append(r); chosen.append(0)
    r = torch.randn(V); r[V - 1] = float("inf")     # +inf
    rows.append(r); chosen.append(0)
    rows.append(torch.full((V,), neg)); chosen.append(0)  # nothing finite
    r = torch.randn(V); rows.append(r); chosen.append(-1)  # bad chosen
    r = torch.randn(V); rows.append(r); chosen.append(V)   # bad chosen
    r = torch.randn(V); m = r.max(); r[[2, 9, 200, V - 1]] = m  # 4-way tie at the top
    rows.append(r); chosen.append(9)
    r = torch.zeros(V); r[0] = -200.0               # one low outlier
    rows.append(r); chosen.append(0)
    r = torch.randn(V) * 30; rows.append(r); chosen.append(1)  # very peaked
    r = torch.randn(V) + 1000.0; rows.append(r); chosen.append(4)  # large offset
    r = torch.randn(V); r[3] = neg; rows.append(r); chosen.append(3)  # chosen is masked
    x = torch.stack(rows).to(dtype)
    return x.cuda(), torch.tensor(chosen, dtype=torch.int32).cuda()


@pytest.mark.parametrize("split", [0, 1])
@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("V", [257, 4096])
def test_features_special_rows(ctx, dtype, V, split):
    _set(ctx, split=split)
    x, ch = _special_rows(V, dtype)
    feat, top2, rf = B.pr_token_features(ctx, x, ch, topk=20)
    of, oi, ofl = _oracle_rows(x, ch)
    _check_features(feat, top2, rf, of, oi, ofl, "special V=%d" % V)


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_split_factor_invariance(ctx, dtype):
    """1, 2, 4 or 8 CTAs per row: same indices and flags, features to tolerance."""
    x, ch = random_rows(20, 151936 if dtype == torch.bfloat16 else 65536, dtype, seed=11)
    of, oi, ofl = _oracle_rows(x, ch)
    for split in (1, 2, 4, 8):
        _set(ctx, split=split)
        feat, top2, rf = B.pr_token_features(ctx, x, ch, topk=20)
        _check_features(feat, top2, rf, of, oi, ofl, "split=%d" % split)
    _set(ctx)


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_persistent_many_rows_per_cta(ctx, dtype):
    """3,000 rows: each persistent CTA carries several rows through both shared
    buffers; special rows (masked, NaN, ties, constant) sit among them."""
    _set(ctx, split=1)
    V = 4097
    x, ch = random_rows(3000, V, dtype, seed=77)
    sx, sch = _special_rows(V, dtype)
    for j in range(sx.size(0)):
        x[97 * j + 5] = sx[j]
        ch[97 * j + 5] = sch[j]
    feat, top2, rf = B.pr_token_features(ctx, x, ch, topk=20)
    of, oi, ofl = _oracle_rows(x, ch)
    _check_features(feat, top2, rf, of, oi, ofl, "persistent")
    _set(ctx)


def _tile_pattern_rows(V, dtype, seed):
    """Rows whose largest values sit where the persistent kernel's candidate
    tiles come from different places.  Group g of a row belongs to tile
    g // 1024 and thread g % 256 (four groups of 16 bytes per thread per
    tile); a thread's best tile is read back from shared memory, its other
    candidate tiles from the row."""
    vec = 8 if dtype == torch.bfloat16 else 4
    nt, unr = 256, 4
    tile = nt * unr
    ntiles = -(-(V // vec) // tile)
    g = torch.Generator().manual_seed(seed)

    def at(t, tid, k, e):
        return ((t * tile + k * nt + tid) * vec + e)

    rows = []
    # one thread holds the top values in five tiles: a third tile >= theta1,
    # so every tile of that thread is a candidate
    r = torch.randn(V, generator=g)
    for j, t in enumerate(range(0, ntiles, max(1, ntiles // 5))):
        for k in range(unr):
            v = at(t, 7, k, (j + k) % vec)
            if v < V:
                r[v] = 10.0 + j + 0.125 * k
    rows.append(r)
    # 24 threads with two strong tiles each: second-best tiles as candidates
    r = torch.randn(V, generator=g)
    for i in range(24):
        for j, t in enumerate((1 + i % 3, ntiles - 2 - i % 4)):
            v = at(t, 9 * i + 3, i % unr, i % vec)
            if v < V:
                r[v] = 8.0 + 0.0625 * i + 0.5 * j
    rows.append(r)
    # rising along the row: every tile beats its thread's best so far
    rows.append(torch.linspace(-3.0, 3.0, V) + 0.01 * torch.randn(V, generator=g))
    # falling: each thread's best tile is its first and must outlast the row
    rows.append(torch.linspace(3.0, -3.0, V) + 0.01 * torch.randn(V, generator=g))
    # the two largest values, tied, at the end of the last full tile and in
    # the row's last element
    r = torch.randn(V, generator=g)
    r[V - 1] = 6.0
    r[min(V // vec // tile * tile * vec, V) - 1] = 6.0
    rows.append(r)
    return torch.stack(rows).to(dtype)


@pytest.mark.parametrize("shift", [0, 1])
@pytest.mark.parametrize("dtype,V", [(torch.bfloat16, 151936), (torch.float32, 65549)])
def test_persistent_candidate_paths(ctx, dtype, V, shift):
    """The persistent kernel's candidate tiles: a thread's best tile from shared
    memory, its second-best and (for a thread with three tiles above theta1)
    all its other tiles from the row, on both shared buffers (600 rows, more
    than one per CTA); with shift 1 the rows start off the 16-byte grid and
    take the element-load path."""
    _set(ctx, split=1)
    pad = (-V) % 8 + 8  # a row stride of a multiple of 16 bytes
    base, ch = random_rows(600, V + pad, dtype, seed=4242)
    x = base[:, shift:shift + V]
    ch = ch % V
    pat = _tile_pattern_rows(V, dtype, seed=4243)
    for j in range(pat.size(0)):
        for r0 in (0, 470):
            x[r0 + 3 * j] = pat[j].cuda()
    feat, top2, rf = B.pr_token_features(ctx, x, ch, topk=20)
    of, oi, ofl = _oracle_rows(x.contiguous(), ch)
    _check_features(feat, top2, rf, of, oi, ofl, "candidate paths V=%d shift=%d" % (V, shift))
    _set(ctx)


def test_rows_past_the_persistent_kernels_tile_limit(ctx):
    """Rows of more than 2^16 tiles (268,443,648 fp32 values, 1.07 GB a row)
    leave the persistent kernel, whose tile indices are 16-bit, even with
    split 1 forced; the largest values sit in the rows' last tiles."""
    _set(ctx, split=1)
    V = (1 << 28) + 2 * 4096
    free, _ = torch.cuda.mem_get_info()
    if free < 8 * V * 4:
        pytest.skip("needs about 9 GB of free device memory")
    g = torch.Generator(device="cuda")
    g.manual_seed(5)
    x = torch.randn(2, V, device="cuda", generator=g)
    x[0, V - 1] = 40.0
    x[0, V - 5000] = 39.0
    x[1, 3] = 41.0
    x[1, V - 2] = 42.0
    ch = torch.tensor([V - 1, 7], dtype=torch.int32, device="cuda")
    feat, top2, rf = B.pr_token_features(ctx, x, ch, topk=20)
    of, oi, ofl = _oracle_rows(x, ch)
    assert oi[0].tolist() == [V - 1, V - 5000] and oi[1].tolist() == [V - 2, 3]
    _check_features(feat, top2, rf, of, oi, ofl, "rows of 65,538 tiles")
    _set(ctx)


def test_features_rho(ctx):
    lengths = [5, 1, 0, 9, 3]
    off = torch.tensor(np.concatenate([[0], np.cumsum(lengths)]), dtype=torch.int64).cuda()
    n = int(sum(lengths))
    x, ch = random_rows(n, 999, torch.float32, seed=5)
    feat, _, _ = B.pr_token_features(ctx, x, ch, topk=20, offsets=off)
    rho = feat[:, 5].cpu().numpy()
    expect = np.concatenate([np.arange(1, T + 1) / T for T in lengths if T > 0])
    assert_close(rho, expect, "rho", rtol=1e-7, atol=0)


# ---- pooling, scoring, the ship rule ---------------------------------------------------------

def _batch(lengths, V, dtype, seed):
    off = np.concatenate([[0], np.cumsum(lengths)]).astype(np.int64)
    x, ch = random_rows(int(off[-1]), V, dtype, seed=seed)
    g = np.random.default_rng(seed)
    w = (g.standard_normal(11) * 0.1).astype(np.float32)
    b = float(np.float32(g.standard_normal() * 0.1))
    return x, ch, off, w, b


def _check_requests(score, ship, rflags, agg, o, tau, what):
    rflags = rflags.cpu().numpy().astype(np.uint32)
    assert np.array_equal(rflags, o["req_flags"]), what
    assert_close(agg.cpu().numpy(), o["agg"], what + " agg")
    assert_close(score.cpu().numpy(), o["score"], what + " score")
    assert_ship(ship.cpu().numpy(), o["ship"], o["score"], tau)


@pytest.mark.parametrize("split", [0, 1])
@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_route_matches_oracle(ctx, dtype, split):
    _set(ctx, split=split)
    lengths = [3, 0, 40, 1, 77, 0, 12, 130, 2]
    x, ch, off, w, b = _batch(lengths, 3001, dtype, seed=21)
    o = oracle.route(as_oracle(x), ch.cpu().numpy(), off, w.astype(np.float64), b, 0.5)
    dw = torch.from_numpy(w).cuda()
    doff = torch.from_numpy(off).cuda()
    score, ship, rf, agg = B.pr_route(ctx, x, ch, doff, dw, b, 0.5)
    _check_requests(score, ship, rf, agg, o, 0.5, "route")
    # and the same through the two separate calls
    feat, top2, rfl = B.pr_token_features(ctx, x, ch, topk=20, offsets=doff)
    agg2, score2, ship2, rf2 = B.pr_aggregate_score(ctx, feat, doff, dw, b, 0.5, row_flags=rfl)
    _check_requests(score2, ship2, rf2, agg2, o, 0.5, "features+aggregate")
    assert torch.equal(agg.nan_to_num(7.0), agg2.nan_to_num(7.0))
    assert torch.equal(ship, ship2)


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_every_launch_shape_of_the_automatic_policy(ctx, dtype):
    """The automatic launch shape changes with the batch: clusters of 8, 4,
    2 CTAs per row for small batches, one CTA per row (no cluster) from one
    row per SM up to one wave of resident CTAs, the persistent kernel above.
    Batches on both sides of each switch, against the oracle; features and
    routing alike."""
    _set(ctx)
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    # resident CTAs of the split kernel: 3 or 4 per SM on this GPU
    sizes = sorted({1, 7, 37, 38, 39, 75, 76, 77, sms - 1, sms, sms + 1, 3 * sms, 4 * sms,
                    4 * sms + 1, 5 * sms})
    for i, n in enumerate(sizes):
        lengths = [n // 2, n - n // 2] if n > 1 else [1]
        x, ch, off, w, b = _batch(lengths, 2053, dtype, seed=300 + i)
        o = oracle.route(as_oracle(x), ch.cpu().numpy(), off, w.astype(np.float64), b, 0.5)
        dw, doff = torch.from_numpy(w).cuda(), torch.from_numpy(off).cuda()
        score, ship, rf, agg = B.pr_route(ctx, x, ch, doff, dw, b, 0.5)
        feat, top2, rfl = B.pr_token_features(ctx, x, ch, topk=20)
        torch.cuda.synchronize()
        _check_requests(score, ship, rf, agg, o, 0.5, "route n=%d" % n)
        assert np.array_equal(top2.cpu().numpy(), o["idx"]), "top2 n=%d" % n
        assert_close(feat.cpu().numpy()[:, [0, 1, 2, 3, 4, 6, 7]],
                     o["feat"][:, [0, 1, 2, 3, 4, 6, 7]], "features n=%d" % n)


def test_route_threshold_and_flags(ctx):
    """Zero weights give score 1/2, which ships at tau = 1/2 (ship iff p >= tau)."""
    lengths = [4, 6]
    x, ch, off, _, _ = _batch(lengths, 500, torch.float32, seed=2)
    ch[2] = 10_000  # a bad token id escalates request 0
    w = torch.zeros(11, device="cuda")
    doff = torch.from_numpy(off).cuda()
    score, ship, rf, agg = B.pr_route(ctx, x, ch, doff, w, 0.0, 0.5)
    assert ship.tolist() == [0, 1]
    assert rf.tolist() == [B.PR_FLAG_BAD_CHOSEN, 0]
    assert torch.isnan(score[0]) and score[1].item() == 0.5
    score, ship, rf, agg = B.pr_route(ctx, x, ch, doff, w, 0.0, 0.5000001)
    assert ship.tolist() == [0, 0]


def test_route_bad_offsets(ctx):
    x, ch, off, w, b = _batch([3, 3], 300, torch.float32, seed=3)
    B.pr_ctx_flags(ctx, clear=True)
    doff = torch.tensor([0, 4, 2], dtype=torch.int64, device="cuda")
    score, ship, rf, agg = B.pr_route(ctx, x[:6], ch[:6], doff, torch.from_numpy(w).cuda(), b, 0.5)
    torch.cuda.synchronize()
    assert rf[1].item() == B.PR_FLAG_BAD_OFFSETS and ship[1].item() == 0
    assert B.pr_ctx_flags(ctx, clear=True) & B.PR_FLAG_BAD_OFFSETS
    B.pr_ctx_reset(ctx)


@pytest.mark.parametrize("chunk", [1, 7, 64, 1000])
def test_chunked_route_equals_whole(ctx, chunk):
    """Requests straddling chunks are finished by whichever chunk ends them;
    chunk order does not matter and the results are bit-identical."""
    lengths = [5, 0, 33, 1, 64, 17, 0, 120, 9]
    x, ch, off, w, b = _batch(lengths, 2048, torch.bfloat16, seed=31)
    _set(ctx, split=2)  # the automatic split depends on the rows per call
    dw, doff = torch.from_numpy(w).cuda(), torch.from_numpy(off).cuda()
    ref = B.pr_route(ctx, x, ch, doff, dw, b, 0.5)
    n = x.size(0)
    starts = list(range(0, n, chunk))
    np.random.default_rng(chunk).shuffle(starts)
    nr = len(lengths)
    score = torch.full((nr,), -5.0, device="cuda")
    ship = torch.full((nr,), 9, dtype=torch.uint8, device="cuda")
    rf = torch.full((nr,), -1, dtype=torch.int32, device="cuda")
    agg = torch.zeros(nr, 11, device="cuda")
    for s in starts:
        e = min(n, s + chunk)
        B.pr_route(ctx, x[s:e], ch[s:e], doff, dw, b, 0.5, row_base=s, score=score, ship=ship,
                   req_flags=rf, agg=agg)
    assert torch.equal(score.nan_to_num(3.0), ref[0].nan_to_num(3.0))
    assert torch.equal(ship, ref[1]) and torch.equal(rf, ref[2])
    assert torch.equal(agg.nan_to_num(3.0), ref[3].nan_to_num(3.0))
    _set(ctx)


def test_route_is_one_launch(ctx):
    x, ch, off, w, b = _batch([10, 20], 1000, torch.bfloat16, seed=4)
    dw, doff = torch.from_numpy(w).cuda(), torch.from_numpy(off).cuda()
    n0 = B.launch_count()
    B.pr_route(ctx, x, ch, doff, dw, b, 0.5)
    assert B.launch_count() - n0 == 1


@pytest.mark.parametrize("chunk_rows", [37, 1 << 40])
def test_route_host_matches_route(ctx, chunk_rows):
    # 37: several chunks through both staging buffers; 2^40: one chunk, the
    # staging area sized by the batch, not by the requested chunk
    lengths = [50, 3, 0, 200, 11]
    x, ch, off, w, b = _batch(lengths, 4096, torch.bfloat16, seed=41)
    _set(ctx, split=1)  # the automatic split depends on the rows per call
    dw, doff = torch.from_numpy(w).cuda(), torch.from_numpy(off).cuda()
    ref = B.pr_route(ctx, x, ch, doff, dw, b, 0.5)
    hx = x.cpu().pin_memory()
    hc = ch.cpu().pin_memory()
    hoff = torch.from_numpy(off)
    hw = torch.from_numpy(w)
    agg = torch.empty(len(lengths), 11)
    score, ship, rf, _ = B.pr_route_host(ctx, hx, hc, hoff, hw, b, 0.5, chunk_rows=chunk_rows,
                                         agg=agg)
    assert torch.equal(score.nan_to_num(3.0), ref[0].cpu().nan_to_num(3.0))
    assert torch.equal(ship, ref[1].cpu()) and torch.equal(rf, ref[2].cpu())
    assert torch.equal(agg.nan_to_num(3.0), ref[3].cpu().nan_to_num(3.0))
    _set(ctx)


def test_output_guards(ctx):
    """Nothing is written outside the output slices."""
    lengths = [7, 0, 19]
    x, ch, off, w, b = _batch(lengths, 1500, torch.float32, seed=8)
    dw, doff = torch.from_numpy(w).cuda(), torch.from_numpy(off).cuda()
    n, nr, G = x.size(0), len(lengths), 64
    sent = 123456.0
    feat = torch.full((n + 2 * G // 8, 8), sent, device="cuda")
    top2 = torch.full((n + 2 * G, 2), 77, dtype=torch.int32, device="cuda")
    rfl = torch.full((n + 2 * G,), 55, dtype=torch.int32, device="cuda")
    g8 = G // 8
    B.pr_token_features(ctx, x, ch, topk=20, feat=feat[g8:g8 + n], top2=top2[G:G + n],
                        row_flags=rfl[G:G + n])
    score = torch.full((nr + 2 * G,), sent, device="cuda")
    ship = torch.full((nr + 2 * G,), 200, dtype=torch.uint8, device="cuda")
    rf = torch.full((nr + 2 * G,), 99, dtype=torch.int32, device="cuda")
    agg = torch.full((nr + 2 * G, 11), sent, device="cuda")
    B.pr_route(ctx, x, ch, doff, dw, b, 0.5, score=score[G:G + nr], ship=ship[G:G + nr],
               req_flags=rf[G:G + nr], agg=agg[G:G + nr])
    torch.cuda.synchronize()
    for t, v, lo, hi in ((feat, sent, g8, g8 + n), (top2, 77, G, G + n), (rfl, 55, G, G + n),
                         (score, sent, G, G + nr), (ship, 200, G, G + nr), (rf, 99, G, G + nr),
                         (agg, sent, G, G + nr)):
        assert (t[:lo] == v).all() and (t[hi:] == v).all()


def test_invalid_arguments(ctx):
    x, ch, off, w, b = _batch([3], 100, torch.float32, seed=1)
    dw, doff = torch.from_numpy(w).cuda(), torch.from_numpy(off).cuda()
    with pytest.raises(B.PRError) as e:
        B.pr_token_features(ctx, x, ch, topk=0)
    assert e.value.status == B.PR_ERR_INVALID_ARG
    with pytest.raises(B.PRError):
        B.pr_token_features(ctx, x, ch, topk=33)
    with pytest.raises(B.PRError):
        B.pr_route(ctx, x, ch, doff, dw, b, 0.5, row_base=(1 << 16))
    with pytest.raises(TypeError):
        B.pr_token_features(ctx, x.half(), ch)  # fp16 is not a verifier dtype
    with pytest.raises(B.PRError):
        B.pr_ctx_set_option(ctx, B.PR_OPT_SPLIT, 3)


# ---- incremental decode steps ------------------------------------------------------------------

def _decode_run(ctx, trace_rows, n_slots, steps, eos, w, b, stop=None, state=None):
    """Run steps [0, stop) (or all) and return per-slot outputs at every EOS."""
    V = trace_rows[0][0].size(1)
    score = torch.full((n_slots,), -1.0, device="cuda")
    ship = torch.zeros(n_slots, dtype=torch.uint8, device="cuda")
    fl = torch.zeros(n_slots, dtype=torch.int32, device="cuda")
    agg = torch.zeros(n_slots, 11, device="cuda")
    slot = torch.arange(n_slots, dtype=torch.int32, device="cuda")
    dw = torch.from_numpy(w).cuda()
    ends = {}
    for s in range(steps if stop is None else stop):
        x, ch = trace_rows[s]
        e = torch.from_numpy(eos[s]).cuda()
        B.pr_decode_step(ctx, x, slot, ch, e, dw, b, 0.5, score, ship, fl, agg_out=agg)
        for sl in np.nonzero(eos[s])[0]:
            ends[(int(sl), s)] = (score[sl].item(), ship[sl].item(), fl[sl].item(),
                                  agg[sl].cpu().numpy().copy())
    return ends


def _small_trace(n_slots=6, steps=80, V=1500, seed=9):
    g = np.random.default_rng(seed)
    eos = np.zeros((steps, n_slots), np.uint8)
    reqs = []
    for s in range(n_slots):
        t = 0
        while t < steps:
            L = int(g.integers(1, 30))
            reqs.append((s, t, L))
            if t + L - 1 < steps:
                eos[t + L - 1, s] = 1
            t += L
    rows = [random_rows(n_slots, V, torch.bfloat16, seed=1000 + k) for k in range(steps)]
    w = (g.standard_normal(11) * 0.1).astype(np.float32)
    b = float(np.float32(g.standard_normal() * 0.1))
    return rows, eos, reqs, w, b


def test_decode_matches_oracle(ctx):
    _set(ctx)
    n_slots, steps = 6, 80
    rows, eos, reqs, w, b = _small_trace(n_slots, steps)
    B.pr_ctx_reset(ctx)
    ends = _decode_run(ctx, rows, n_slots, steps, eos, w, b)
    xs = [as_oracle(r[0]) for r in rows]
    cs = [r[1].cpu().numpy() for r in rows]
    checked = 0
    for (sl, t0, L) in reqs:
        if t0 + L > steps:
            continue
        X = np.stack([xs[t][sl] for t in range(t0, t0 + L)])
        C = np.array([cs[t][sl] for t in range(t0, t0 + L)], np.int32)
        o = oracle.route(X, C, np.array([0, L]), w.astype(np.float64), b, 0.5)
        sc, sh, fl, ag = ends[(sl, t0 + L - 1)]
        assert fl == o["req_flags"][0]
        assert_close(ag, o["agg"][0], "decode agg")
        assert_close(sc, o["score"][0], "decode score")
        assert_ship([sh], o["ship"], o["score"], 0.5)
        checked += 1
    assert checked >= 15
    B.pr_ctx_reset(ctx)


def test_decode_checkpoint_resume(ctx):
    n_slots, steps = 6, 80
    rows, eos, reqs, w, b = _small_trace(n_slots, steps, seed=12)
    B.pr_ctx_reset(ctx)
    full = _decode_run(ctx, rows, n_slots, steps, eos, w, b)
    B.pr_ctx_reset(ctx)
    first = _decode_run(ctx, rows, n_slots, steps, eos, w, b, stop=37)
    state = B.pr_state_export(ctx)
    other = B.pr_ctx_create(0, max_rows=16, max_requests=1024)
    try:
        B.pr_state_import(other, state)
        score = torch.full((n_slots,), -1.0, device="cuda")
        ship = torch.zeros(n_slots, dtype=torch.uint8, device="cuda")
        fl = torch.zeros(n_slots, dtype=torch.int32, device="cuda")
        agg = torch.zeros(n_slots, 11, device="cuda")
        slot = torch.arange(n_slots, dtype=torch.int32, device="cuda")
        dw = torch.from_numpy(w).cuda()
        for s in range(37, steps):
            x, ch = rows[s]
            B.pr_decode_step(other, x, slot, ch, torch.from_numpy(eos[s]).cuda(), dw, b, 0.5, score,
                             ship, fl, agg_out=agg)
            for sl in np.nonzero(eos[s])[0]:
                ref = full[(int(sl), s)]
                assert score[sl].item() == ref[0] or (np.isnan(ref[0]) and np.isnan(score[sl].item()))
                assert ship[sl].item() == ref[1] and fl[sl].item() == ref[2]
                assert np.array_equal(agg[sl].cpu().numpy(), ref[3])
        for k, v in first.items():
            assert v[1] == full[k][1]
    finally:
        B.pr_ctx_destroy(other)
    with pytest.raises(B.PRError):
        B.pr_state_import(ctx, state[:-4])
    B.pr_ctx_reset(ctx)


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_decode_and_route_agree_on_the_same_requests(ctx, dtype):
    """The incremental mode and the full-response mode on the same requests.
    Route pools a request's records with a fixed-order lane-strided sum;
    a decode slot keeps a compensated running sum in step order.  So the
    minima and the mean position fraction are bit-identical between the
    modes, and the five means agree within the parity tolerance, with each
    other and with the oracle; the decisions are equal outside the band
    around tau.  Both modes run the same launch shape (8 CTAs per row), so
    each row's features are computed identically."""
    _set(ctx, split=8)
    lengths = [1, 2, 7, 33, 64, 129, 300, 1000]
    x, ch, off, w, b = _batch(lengths, 4097, dtype, seed=77)
    dw, doff = torch.from_numpy(w).cuda(), torch.from_numpy(off).cuda()
    n = len(lengths)
    r_score, r_ship, r_flags, r_agg = B.pr_route(ctx, x, ch, doff, dw, b, 0.5)
    # decode: request r in slot r, one row per step while it is live
    B.pr_ctx_reset(ctx)
    d_score = torch.zeros(1024, device="cuda")
    d_ship = torch.zeros(1024, dtype=torch.uint8, device="cuda")
    d_flags = torch.zeros(1024, dtype=torch.int32, device="cuda")
    d_agg = torch.zeros(1024, 11, device="cuda")
    for t in range(max(lengths)):
        live = [r for r in range(n) if lengths[r] > t]
        rows = torch.tensor([int(off[r]) + t for r in live], dtype=torch.int64, device="cuda")
        slot = torch.tensor(live, dtype=torch.int32, device="cuda")
        eos = torch.tensor([1 if lengths[r] == t + 1 else 0 for r in live], dtype=torch.uint8,
                           device="cuda")
        B.pr_decode_step(ctx, x.index_select(0, rows), slot, ch.index_select(0, rows).contiguous(),
                         eos, dw, b, 0.5, d_score, d_ship, d_flags, agg_out=d_agg)
    torch.cuda.synchronize()
    ra, da = r_agg.cpu().numpy(), d_agg[:n].cpu().numpy()
    mins_and_rho = [1, 3, 5, 7, 9, 10]
    assert np.array_equal(ra[:, mins_and_rho], da[:, mins_and_rho])
    assert_close(da, ra, "decode vs route agg")
    assert_close(d_score[:n].cpu().numpy(), r_score.cpu().numpy(), "decode vs route score")
    assert np.array_equal(d_flags[:n].cpu().numpy(), r_flags.cpu().numpy())
    o = oracle.route(as_oracle(x), ch.cpu().numpy(), off, w.astype(np.float64), b, 0.5)
    _check_requests(d_score[:n], d_ship[:n], d_flags[:n], d_agg[:n], o, 0.5, "decode")
    _check_requests(r_score, r_ship, r_flags, r_agg, o, 0.5, "route")
    B.pr_ctx_reset(ctx)
    _set(ctx)


def test_decode_bad_slot_flagged(ctx):
    B.pr_ctx_reset(ctx)
    x, ch = random_rows(2, 300, torch.float32, seed=1)
    slot = torch.tensor([0, 5000], dtype=torch.int32, device="cuda")
    eos = torch.ones(2, dtype=torch.uint8, device="cuda")
    out = torch.zeros(1024, device="cuda")
    ship = torch.zeros(1024, dtype=torch.uint8, device="cuda")
    fl = torch.zeros(1024, dtype=torch.int32, device="cuda")
    B.pr_decode_step(ctx, x, slot, ch, eos, torch.zeros(11, device="cuda"), 0.0, 0.5, out, ship, fl)
    assert B.pr_ctx_flags(ctx, clear=True) & B.PR_FLAG_BAD_SLOT
    assert ship[0].item() == 1 and out[0].item() == 0.5
    B.pr_ctx_reset(ctx)


def test_last_error_reads_the_flag_word_after_the_device_finishes(ctx):
    """pr_last_error waits for all work on the context's device, not one
    stream: a flagged decode step queued on a side stream (never synchronised
    by the test) shows up in its answer.  The word is left as it is, so a
    second read gives the same bits, until pr_ctx_flags clears it."""
    B.pr_ctx_reset(ctx)
    B.pr_ctx_flags(ctx, clear=True)
    assert B.pr_last_error(ctx) == 0
    side = torch.cuda.Stream()
    x, ch = random_rows(3, 5000, torch.bfloat16, seed=4)
    slot = torch.tensor([0, 4096, 1], dtype=torch.int32, device="cuda")
    eos = torch.zeros(3, dtype=torch.uint8, device="cuda")
    out = torch.zeros(1024, device="cuda")
    ship = torch.zeros(1024, dtype=torch.uint8, device="cuda")
    fl = torch.zeros(1024, dtype=torch.int32, device="cuda")
    torch.cuda.synchronize()
    with torch.cuda.stream(side):
        # a long chain of work first, so the flagged step is still queued when
        # the host asks
        big = torch.randn(4096, 4096, device="cuda")
        for _ in range(8):
            big = big @ big
            big /= big.norm()
        B.pr_decode_step(ctx, x, slot, ch, eos, torch.zeros(11, device="cuda"), 0.0, 0.5, out,
                         ship, fl, stream=side)
    word = B.pr_last_error(ctx)
    assert word == B.PR_FLAG_BAD_SLOT, word
    assert B.pr_last_error(ctx) == word  # read only
    assert B.pr_ctx_flags(ctx, clear=True) == word
    assert B.pr_last_error(ctx) == 0
    # a route call whose request reaches past the context's rows raises
    # PR_FLAG_BAD_OFFSETS in the same word
    off = torch.tensor([0, 2, (1 << 16) + 5], dtype=torch.int64, device="cuda")
    x2, ch2 = random_rows(2, 300, torch.float32, seed=5)
    score, sh, rf, _ = B.pr_route(ctx, x2, ch2, off, torch.zeros(11, device="cuda"), 0.0, 0.5)
    assert B.pr_last_error(ctx) == B.PR_FLAG_BAD_OFFSETS
    assert rf[1].item() == B.PR_FLAG_BAD_OFFSETS and np.isnan(score[1].item())
    assert rf[0].item() == 0 and score[0].item() == 0.5
    B.pr_ctx_flags(ctx, clear=True)
    B.pr_ctx_reset(ctx)


def test_overlap_option_changes_nothing_but_timing(ctx):
    """With PR_OPT_OVERLAP a call may start while the previous one finishes;
    back-to-back route calls and decode steps give bit-identical results."""
    lengths = [40, 0, 75, 3, 150]
    x, ch, off, w, b = _batch(lengths, 5000, torch.bfloat16, seed=91)
    dw, doff = torch.from_numpy(w).cuda(), torch.from_numpy(off).cuda()
    results = {}
    for overlap in (0, 1):
        B.pr_ctx_set_option(ctx, B.PR_OPT_OVERLAP, overlap)
        outs = []
        for split in (1, 2):  # the persistent kernel and the cluster kernel
            _set(ctx, split=split)
            for rep in range(4):
                outs.append(B.pr_route(ctx, x, ch, doff, dw, b, 0.5))
        torch.cuda.synchronize()
        results[overlap] = outs
    for (a0, a1) in zip(results[0], results[1]):
        for t0, t1 in zip(a0, a1):
            assert torch.equal(t0.nan_to_num(5.0), t1.nan_to_num(5.0))
    # decode: the same trace with and without overlap
    n_slots, steps = 6, 60
    rows, eos, reqs, w2, b2 = _small_trace(n_slots, steps, seed=5)
    ends = {}
    for overlap in (0, 1):
        B.pr_ctx_set_option(ctx, B.PR_OPT_OVERLAP, overlap)
        B.pr_ctx_reset(ctx)
        ends[overlap] = _decode_run(ctx, rows, n_slots, steps, eos, w2, b2)
    for k, v in ends[0].items():
        v1 = ends[1][k]
        assert v[1:3] == v1[1:3] and np.array_equal(v[3], v1[3], equal_nan=True)
        assert v[0] == v1[0] or (np.isnan(v[0]) and np.isnan(v1[0]))
    B.pr_ctx_set_option(ctx, B.PR_OPT_OVERLAP, 0)
    _set(ctx)
    B.pr_ctx_reset(ctx)
