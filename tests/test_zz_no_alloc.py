"""pr_route_noalloc, the verification call for hosts that cannot let a
library allocate device memory (an engine that owns a pre-reserved memory
pool, or a serving loop that cannot afford the synchronisation cudaMalloc may
bring).  It must give the same answers as pr_route and the float64 oracle,
call after call, although all its calls share one fixed scratch array inside
the library.  The cases cover both of its launch shapes: a cluster of CTAs per
row for small batches, and one CTA per row once the batch fills two waves of
resident CTAs (up to its largest accepted batch).

This file is collected last on purpose, and it builds everything it needs, so
it passes both alone in a fresh process and after the other tests."""
import os

import numpy as np
import pytest
import torch

import oracle
from _util import as_oracle, assert_close, assert_ship, random_rows

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def B():
    assert torch.cuda.is_available(), "needs a CUDA device"
    from paper_2608_28726_gb300 import build
    build.build()
    from paper_2608_28726_gb300 import binding
    torch.cuda.set_device(0)
    return binding


def _batch(name, n_req, max_len, device):
    from paper_2608_28726_gb300 import workloads as W
    wl = W.make(name, n_req=n_req, max_len=max_len)
    x, ch = W.rows(wl, 0, wl.n_rows, device=device)
    off = torch.from_numpy(wl.offsets).to(device)
    w = torch.from_numpy(wl.w).to(device)
    return wl, x, ch, off, w


def _outputs(n, dev="cuda"):
    return (torch.full((n,), -7.0, device=dev), torch.full((n,), 9, dtype=torch.uint8, device=dev),
            torch.full((n,), -1, dtype=torch.int32, device=dev), torch.zeros(n, 11, device=dev))


def _same_as_route(B, ctx, x, ch, off, w, b, tau, got):
    score, ship, flags, agg = got
    ref = B.pr_route(ctx, x, ch, off, w, b, tau)
    torch.cuda.synchronize()
    assert_close(score.cpu().numpy(), ref[0].cpu().numpy(), "noalloc score vs pr_route")
    assert_close(agg.cpu().numpy(), ref[3].cpu().numpy(), "noalloc agg vs pr_route")
    assert np.array_equal(ship.cpu().numpy(), ref[1].cpu().numpy())
    assert np.array_equal(flags.cpu().numpy(), ref[2].cpu().numpy())


def _same_as_oracle(x, ch, off, w, b, tau, got, n_req=None):
    score, ship, flags, agg = got
    o = oracle.route(as_oracle(x), ch.cpu().numpy(), off.cpu().numpy(),
                     w.cpu().numpy().astype(np.float64), b, tau, n_threads=os.cpu_count() or 1)
    k = len(o["score"]) if n_req is None else n_req
    assert_close(agg.cpu().numpy()[:k], o["agg"][:k], "noalloc agg vs oracle")
    assert_close(score.cpu().numpy()[:k], o["score"][:k], "noalloc score vs oracle")
    assert_ship(ship.cpu().numpy()[:k], o["ship"][:k], o["score"][:k], tau)
    assert np.array_equal(flags.cpu().numpy()[:k].astype(np.uint32), o["req_flags"][:k])


def test_noalloc_matches_route_on_two_calls_in_a_row(B):
    dev = torch.device("cuda", 0)
    # two different batches back to back: bf16 at the small model's vocabulary,
    # then fp32 at another width, so a stale scratch would show
    batches = [_batch("full", 6, 90, dev), _batch("tiny", 5, 40, dev)]
    ctx = B.pr_ctx_create(0, max_rows=max(b[0].n_rows for b in batches), max_requests=16)
    try:
        outs = []
        for wl, x, ch, off, w in batches:
            got = _outputs(wl.n_req)
            B.pr_route_noalloc(x, ch, off, w, wl.b, wl.tau, *got[:3], agg=got[3])
            outs.append(got)
        torch.cuda.synchronize()
        for (wl, x, ch, off, w), got in zip(batches, outs):
            _same_as_route(B, ctx, x, ch, off, w, wl.b, wl.tau, got)
            _same_as_oracle(x, ch, off, w, wl.b, wl.tau, got)
    finally:
        B.pr_ctx_destroy(ctx)


def test_noalloc_one_cta_per_row_at_full_vocabulary(B):
    """About 4,000 rows of V = 151,936 bf16 (the full-response workload's
    first requests): more rows than two waves of resident CTAs, so each row
    takes one CTA.  Checked against the float64 oracle on every request, and
    against pr_route."""
    dev = torch.device("cuda", 0)
    wl, x, ch, off, w = _batch("full", 26, None, dev)
    assert 3500 <= wl.n_rows <= B.PR_NOALLOC_MAX_ROWS
    ctx = B.pr_ctx_create(0, max_rows=wl.n_rows, max_requests=wl.n_req)
    try:
        for _ in range(2):
            got = _outputs(wl.n_req)
            B.pr_route_noalloc(x, ch, off, w, wl.b, wl.tau, *got[:3], agg=got[3])
            torch.cuda.synchronize()
            _same_as_oracle(x, ch, off, w, wl.b, wl.tau, got)
            _same_as_route(B, ctx, x, ch, off, w, wl.b, wl.tau, got)
    finally:
        B.pr_ctx_destroy(ctx)


def _ragged(n_rows, n_req, V, seed, dtype=torch.float32):
    rng = np.random.Generator(np.random.PCG64(seed))
    cuts = np.sort(rng.choice(np.arange(1, n_rows), size=n_req - 1, replace=False))
    off = np.concatenate([[0], cuts, [n_rows]]).astype(np.int64)
    x, ch = random_rows(n_rows, V, dtype, seed=seed)
    w = (rng.normal(0.0, 0.1, 11)).astype(np.float32)
    return x, ch, torch.from_numpy(off).cuda(), torch.from_numpy(w).cuda(), float(rng.normal(0, .1))


def test_noalloc_largest_batch(B):
    """PR_NOALLOC_MAX_ROWS rows in PR_NOALLOC_MAX_REQUESTS requests (small
    vocabulary): the largest batch the call accepts, one CTA per row."""
    n, R = B.PR_NOALLOC_MAX_ROWS, B.PR_NOALLOC_MAX_REQUESTS
    x, ch, off, w, b = _ragged(n, R, 700, seed=11)
    ctx = B.pr_ctx_create(0, max_rows=n, max_requests=R)
    try:
        got = _outputs(R)
        B.pr_route_noalloc(x, ch, off, w, b, 0.5, *got[:3], agg=got[3])
        torch.cuda.synchronize()
        _same_as_route(B, ctx, x, ch, off, w, b, 0.5, got)
        _same_as_oracle(x, ch, off, w, b, 0.5, got)
    finally:
        B.pr_ctx_destroy(ctx)


def test_noalloc_on_both_sides_of_each_split_switch(B):
    """The split halves as the batch grows (8, 4, 2, then one CTA per row at
    two waves of resident CTAs).  The switch points depend on the kernel's
    residency, so batch sizes straddle every two-wave size a residency of 1
    to 8 CTAs per SM would give."""
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    sizes = sorted({n for bps in range(1, 9) for k in (1, 2) for n in
                    (k * sms * bps - 1, k * sms * bps, k * sms * bps + 1)})
    ctx = B.pr_ctx_create(0, max_rows=max(sizes), max_requests=64)
    try:
        for i, n in enumerate(sizes):
            x, ch, off, w, b = _ragged(n, 17, 333, seed=100 + i)
            got = _outputs(17)
            B.pr_route_noalloc(x, ch, off, w, b, 0.5, *got[:3], agg=got[3])
            torch.cuda.synchronize()
            _same_as_route(B, ctx, x, ch, off, w, b, 0.5, got)
            _same_as_oracle(x, ch, off, w, b, 0.5, got)
    finally:
        B.pr_ctx_destroy(ctx)


def test_noalloc_reports_rows_outside_every_request(B):
    """offsets[n_req] < n_rows: the rows after the last request belong to no
    request.  The call has no flag word the caller could read, so the last
    request carries PR_FLAG_BAD_OFFSETS (score NaN, not shipped); the other
    requests are verified as usual."""
    x, ch, off, w, b = _ragged(300, 5, 500, seed=21)
    short = off.clone()
    short[-1] = 290
    got = _outputs(5)
    B.pr_route_noalloc(x, ch, short, w, b, 0.5, *got[:3], agg=got[3])
    torch.cuda.synchronize()
    score, ship, flags, agg = got
    assert flags[4].item() == B.PR_FLAG_BAD_OFFSETS
    assert np.isnan(score[4].item()) and ship[4].item() == 0
    assert np.isnan(agg[4].cpu().numpy()).all()
    _same_as_oracle(x, ch, short, w, b, 0.5, got, n_req=4)
    # the same call with consistent offsets right after: nothing carried over
    got = _outputs(5)
    B.pr_route_noalloc(x, ch, off, w, b, 0.5, *got[:3], agg=got[3])
    torch.cuda.synchronize()
    _same_as_oracle(x, ch, off, w, b, 0.5, got)


def test_noalloc_rejects_batches_above_its_limit(B):
    dev = torch.device("cuda", 0)
    n = B.PR_NOALLOC_MAX_ROWS + 1
    x = torch.zeros(n, 8, device=dev)
    ch = torch.zeros(n, dtype=torch.int32, device=dev)
    off = torch.tensor([0, n], dtype=torch.int64, device=dev)
    w = torch.zeros(11, device=dev)
    out = (torch.empty(1, device=dev), torch.empty(1, dtype=torch.uint8, device=dev),
           torch.empty(1, dtype=torch.int32, device=dev))
    with pytest.raises(B.PRError) as e:
        B.pr_route_noalloc(x, ch, off, w, 0.0, 0.5, *out)
    assert e.value.status == B.PR_ERR_INVALID_ARG
    # host tensors never reach the library
    with pytest.raises(B.PRError) as e:
        B.pr_route_noalloc(x[:4].cpu(), ch[:4].cpu(), off.cpu(), w.cpu(), 0.0, 0.5,
                           *(t.cpu() for t in out))
    assert e.value.status == B.PR_ERR_INVALID_ARG
