"""GPU parity at the five workloads' full sizes (through the C ABI), against
the float64 oracle on sampled whole requests.

  tiny    every row and request
  full    the whole batch in one pr_route launch (the benchmark's launch), plus
          per-row features on the sampled requests' rows
  ragged  1,024 requests streamed in 8,192-row chunks; every request that
          crosses a chunk boundary is checked
  wide    147,828 rows of V = 262,144 fp32 (155 GB) streamed in chunks; sampled
          requests include rows with an exact top-1 tie
  decode  256 slots x 1,000 steps of pr_decode_step; every finished request of
          the sampled slots is checked
"""
import os

import numpy as np
import pytest
import torch

import oracle
from _util import assert_close, assert_ship

pytestmark = pytest.mark.gpu

THREADS = os.cpu_count() or 1
B = None
W = None


@pytest.fixture(scope="module")
def ctx():
    global B, W
    assert torch.cuda.is_available(), "the GPU tests need a CUDA device"
    from paper_2608_28726_gb300 import build
    build.build()
    from paper_2608_28726_gb300 import binding, workloads
    B, W = binding, workloads
    h = B.pr_ctx_create(0, max_rows=200_000, max_requests=1024)
    yield h
    B.pr_ctx_destroy(h)


def _oracle_requests(wl, reqs, device="cuda"):
    """Oracle results for whole requests `reqs` (rows regenerated on the GPU)."""
    off = wl.offsets
    out = {}
    for r in reqs:
        lo, hi = int(off[r]), int(off[r + 1])
        x, ch = W.rows(wl, lo, hi, device=device)
        o = oracle.route(W.to_oracle_array(x), ch.cpu().numpy(), np.array([0, hi - lo]),
                         wl.w.astype(np.float64), wl.b, wl.tau, n_threads=THREADS)
        out[r] = o
    return out


def _check_sampled(o_by_req, score, ship, flags, agg, tau, what):
    score, ship, flags, agg = (t.cpu().numpy() for t in (score, ship, flags, agg))
    for r, o in o_by_req.items():
        assert flags[r] == o["req_flags"][0], "%s request %d flags" % (what, r)
        assert_close(agg[r], o["agg"][0], "%s request %d agg" % (what, r))
        assert_close(score[r], o["score"][0], "%s request %d score" % (what, r))
        assert_ship([ship[r]], o["ship"], o["score"], tau)


def _outputs(n, device="cuda"):
    return (torch.full((n,), -9.0, device=device), torch.full((n,), 7, dtype=torch.uint8, device=device),
            torch.full((n,), -1, dtype=torch.int32, device=device), torch.zeros(n, 11, device=device))


def test_tiny_every_row_and_request(ctx):
    wl = W.make("tiny")
    x, ch = W.rows(wl, 0, wl.n_rows, device="cuda")
    off, w = torch.from_numpy(wl.offsets).cuda(), torch.from_numpy(wl.w).cuda()
    score, ship, flags, agg = B.pr_route(ctx, x, ch, off, w, wl.b, wl.tau)
    feat, top2, rfl = B.pr_token_features(ctx, x, ch, topk=20, offsets=off)
    o = oracle.route(W.to_oracle_array(x), ch.cpu().numpy(), wl.offsets, wl.w.astype(np.float64),
                     wl.b, wl.tau, n_threads=THREADS)
    assert np.array_equal(top2.cpu().numpy(), o["idx"])
    assert np.array_equal(rfl.cpu().numpy().astype(np.uint32), o["row_flags"])
    assert_close(feat.cpu().numpy(), o["feat"], "tiny features")
    assert np.array_equal(flags.cpu().numpy().astype(np.uint32), o["req_flags"])
    assert_close(agg.cpu().numpy(), o["agg"], "tiny agg")
    assert_close(score.cpu().numpy(), o["score"], "tiny score")
    assert_ship(ship.cpu().numpy(), o["ship"], o["score"], wl.tau)


def test_full_response_batch(ctx):
    """The benchmark's launch: all 8,847 rows of V = 151,936 bf16 in one pr_route."""
    wl = W.make("full")
    x, ch = W.rows(wl, 0, wl.n_rows, device="cuda")
    off, w = torch.from_numpy(wl.offsets).cuda(), torch.from_numpy(wl.w).cuda()
    score, ship, flags, agg = B.pr_route(ctx, x, ch, off, w, wl.b, wl.tau)
    reqs = [0, 1, 17, 40, 63]
    o = _oracle_requests(wl, reqs)
    _check_sampled(o, score, ship, flags, agg, wl.tau, "full")
    # per-row features of the sampled requests, in the same kernel family
    for r in reqs[:2]:
        lo, hi = int(wl.offsets[r]), int(wl.offsets[r + 1])
        sub_off = torch.tensor([0, hi - lo], dtype=torch.int64, device="cuda")
        feat, top2, rfl = B.pr_token_features(ctx, x[lo:hi], ch[lo:hi], topk=20, offsets=sub_off)
        assert np.array_equal(top2.cpu().numpy(), o[r]["idx"])
        assert_close(feat.cpu().numpy(), o[r]["feat"], "full features")
    # every request got an answer and no request was flagged
    assert (flags.cpu().numpy() == 0).all()
    assert set(np.unique(ship.cpu().numpy())) <= {0, 1}


def test_ragged_chunked(ctx):
    """1,024 requests in 8,192-row chunks on one stream; requests cross chunks."""
    wl = W.make("ragged")
    off_np = wl.offsets
    off, w = torch.from_numpy(off_np).cuda(), torch.from_numpy(wl.w).cuda()
    score, ship, flags, agg = _outputs(wl.n_req)
    for lo in range(0, wl.n_rows, wl.chunk_rows):
        hi = min(wl.n_rows, lo + wl.chunk_rows)
        x, ch = W.rows(wl, lo, hi, device="cuda")
        B.pr_route(ctx, x, ch, off, w, wl.b, wl.tau, row_base=lo, score=score, ship=ship,
                   req_flags=flags, agg=agg)
        del x, ch
    torch.cuda.synchronize()
    bounds = np.arange(wl.chunk_rows, wl.n_rows, wl.chunk_rows)
    crossing = [int(r) for r in range(wl.n_req)
                if np.any((off_np[r] < bounds) & (bounds < off_np[r + 1]))]
    assert len(crossing) >= 10
    sample = crossing + [0, 511, 1023]
    o = _oracle_requests(wl, sample)
    _check_sampled(o, score, ship, flags, agg, wl.tau, "ragged")
    assert (flags.cpu().numpy() == 0).all()


def test_wide_vocab_chunked(ctx):
    """147,828 rows of V = 262,144 fp32 (155 GB) in 4,096-row chunks."""
    wl = W.make("wide")
    off, w = torch.from_numpy(wl.offsets).cuda(), torch.from_numpy(wl.w).cuda()
    score, ship, flags, agg = _outputs(wl.n_req)
    chunk = 4096
    for lo in range(0, wl.n_rows, chunk):
        hi = min(wl.n_rows, lo + chunk)
        x, ch = W.rows(wl, lo, hi, device="cuda")
        B.pr_route(ctx, x, ch, off, w, wl.b, wl.tau, row_base=lo, score=score, ship=ship,
                   req_flags=flags, agg=agg)
        del x, ch
    torch.cuda.synchronize()
    reqs = [0, 200, 511]
    o = _oracle_requests(wl, reqs)
    _check_sampled(o, score, ship, flags, agg, wl.tau, "wide")
    # the sampled rows include exact top-1 ties: indices must match, lower first
    r = reqs[0]
    lo, hi = int(wl.offsets[r]), int(wl.offsets[r + 1])
    x, ch = W.rows(wl, lo, hi, device="cuda")
    feat, top2, _ = B.pr_token_features(ctx, x, ch, topk=20)
    top2 = top2.cpu().numpy()
    assert np.array_equal(top2, o[r]["idx"])
    tied = (o[r]["feat"][:, oracle.MARGIN] == 0.0)
    assert tied.sum() >= 3 and (top2[tied, 0] < top2[tied, 1]).all()
    assert_close(feat.cpu().numpy()[:, :5], o[r]["feat"][:, :5], "wide features")


def test_decode_steps(ctx):
    """256 live slots x 1,000 steps; each step's row is folded into its slot."""
    tr = W.decode_trace()
    wl = tr.as_workload()
    S, steps = tr.n_slots, tr.n_steps
    B.pr_ctx_reset(ctx)
    slot = torch.arange(S, dtype=torch.int32, device="cuda")
    w = torch.from_numpy(tr.w).cuda()
    score, ship, flags, agg = _outputs(1024)
    sampled = [0, 1, 2]
    kept = {s: [] for s in sampled}
    ends = {}
    eos_dev = torch.from_numpy(tr.eos).cuda()
    for t in range(steps):
        x, ch = W.rows(wl, t * S, (t + 1) * S, device="cuda")
        B.pr_decode_step(ctx, x, slot, ch, eos_dev[t], w, tr.b, tr.tau, score, ship, flags,
                         agg_out=agg)
        for s in sampled:
            kept[s].append((W.to_oracle_array(x[s:s + 1])[0], int(ch[s].item())))
            if tr.eos[t, s]:
                ends[(s, t)] = (score[s].item(), ship[s].item(), flags[s].item(),
                                agg[s].cpu().numpy().copy())
    checked = 0
    for (s, t0, L) in tr.requests:
        if s not in sampled or t0 + L > steps:
            continue
        X = np.stack([kept[s][t][0] for t in range(t0, t0 + L)])
        C = np.array([kept[s][t][1] for t in range(t0, t0 + L)], np.int32)
        o = oracle.route(X, C, np.array([0, L]), tr.w.astype(np.float64), tr.b, tr.tau,
                         n_threads=THREADS)
        sc, sh, fl, ag = ends[(s, t0 + L - 1)]
        assert fl == o["req_flags"][0]
        assert_close(ag, o["agg"][0], "decode agg")
        assert_close(sc, o["score"][0], "decode score")
        assert_ship([sh], o["ship"], o["score"], tr.tau)
        checked += 1
    assert checked >= 3
    B.pr_ctx_reset(ctx)
