"""pr_route_noalloc, the verification call for hosts that cannot let a
library allocate device memory (an engine that owns a pre-reserved memory
pool, or a serving loop that cannot afford the synchronisation cudaMalloc may
bring).  It must give the same answers as pr_route, call after call, although
all its calls share one fixed scratch array inside the library.

This file is collected last on purpose, and it builds everything it needs, so
it passes both alone in a fresh process and after the other tests."""
import numpy as np
import pytest
import torch

from _util import assert_close

pytestmark = pytest.mark.gpu


def _batch(name, n_req, max_len, device):
    from paper_2608_28726_gb300 import workloads as W
    wl = W.make(name, n_req=n_req, max_len=max_len)
    x, ch = W.rows(wl, 0, wl.n_rows, device=device)
    off = torch.from_numpy(wl.offsets).to(device)
    w = torch.from_numpy(wl.w).to(device)
    return wl, x, ch, off, w


def test_noalloc_matches_route_on_two_calls_in_a_row():
    assert torch.cuda.is_available(), "needs a CUDA device"
    from paper_2608_28726_gb300 import build
    build.build()
    from paper_2608_28726_gb300 import binding as B

    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    # two different batches back to back: bf16 at the small model's vocabulary,
    # then fp32 at another width, so a stale scratch would show
    batches = [_batch("full", 6, 90, dev), _batch("tiny", 5, 40, dev)]
    ctx = B.pr_ctx_create(0, max_rows=max(b[0].n_rows for b in batches), max_requests=16)
    try:
        outs = []
        for wl, x, ch, off, w in batches:
            n = wl.n_req
            score = torch.full((n,), -7.0, device=dev)
            ship = torch.full((n,), 9, dtype=torch.uint8, device=dev)
            flags = torch.full((n,), -1, dtype=torch.int32, device=dev)
            agg = torch.zeros(n, 11, device=dev)
            B.pr_route_noalloc(x, ch, off, w, wl.b, wl.tau, score, ship, flags, agg=agg)
            outs.append((score, ship, flags, agg))
        torch.cuda.synchronize()
        for (wl, x, ch, off, w), (score, ship, flags, agg) in zip(batches, outs):
            ref = B.pr_route(ctx, x, ch, off, w, wl.b, wl.tau)
            torch.cuda.synchronize()
            assert_close(score.cpu().numpy(), ref[0].cpu().numpy(), "noalloc score")
            assert_close(agg.cpu().numpy(), ref[3].cpu().numpy(), "noalloc agg")
            assert np.array_equal(ship.cpu().numpy(), ref[1].cpu().numpy())
            assert np.array_equal(flags.cpu().numpy(), ref[2].cpu().numpy())
    finally:
        B.pr_ctx_destroy(ctx)


def test_noalloc_rejects_batches_above_its_limit():
    from paper_2608_28726_gb300 import build
    build.build()
    from paper_2608_28726_gb300 import binding as B
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
