"""The verifier calls captured in CUDA graphs: a graph of several pr_route
calls and a graph of a whole decode trace (context reset + every step)
replay to bit-identical outputs of the same calls issued on a stream, and the
decode state they leave is byte-identical.  This is how launch-bound loops
(small batches, one decode step per generated token) are meant to run."""
import numpy as np
import pytest
import torch

from _util import random_rows

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def B():
    from paper_2608_28726_gb300 import build
    build.build()
    from paper_2608_28726_gb300 import binding
    return binding


def _capture(fn):
    """Capture fn() (which issues its work on the current stream) in a graph."""
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, capture_error_mode="thread_local"):
        fn()
    return g


@pytest.mark.parametrize("overlap", [0, 1])
def test_route_calls_replay_in_a_graph(B, overlap):
    ctx = B.pr_ctx_create(0, max_rows=4096, max_requests=64)
    try:
        B.pr_ctx_set_option(ctx, B.PR_OPT_OVERLAP, overlap)
        batches = []
        for k, (n, V, dt) in enumerate([(300, 5000, torch.bfloat16), (257, 32000, torch.float32),
                                       (64, 151936, torch.bfloat16)]):
            x, ch = random_rows(n, V, dt, seed=50 + k)
            cuts = np.sort(np.random.default_rng(k).choice(np.arange(1, n), 5, replace=False))
            off = torch.from_numpy(np.concatenate([[0], cuts, [n]]).astype(np.int64)).cuda()
            w = torch.linspace(-0.2, 0.2, 11, device="cuda")
            outs = (torch.empty(6, device="cuda"), torch.empty(6, dtype=torch.uint8, device="cuda"),
                    torch.empty(6, dtype=torch.int32, device="cuda"), torch.empty(6, 11, device="cuda"))
            batches.append((x, ch, off, w, outs))

        def run():
            for x, ch, off, w, outs in batches:
                B.pr_route(ctx, x, ch, off, w, 0.05, 0.5, score=outs[0], ship=outs[1],
                           req_flags=outs[2], agg=outs[3])

        run()  # eager on the current stream (also the first-call set-up)
        torch.cuda.synchronize()
        ref = [[t.clone() for t in b[4]] for b in batches]
        for b in batches:
            for t in b[4]:
                t.fill_(0)
        g = _capture(run)
        for _ in range(2):
            g.replay()
        torch.cuda.synchronize()
        for r, b in zip(ref, batches):
            for t0, t1 in zip(r, b[4]):
                assert torch.equal(t0.view(torch.uint8), t1.view(torch.uint8))
        assert B.pr_ctx_flags(ctx) == 0
    finally:
        B.pr_ctx_destroy(ctx)


@pytest.mark.parametrize("n_slots,overlap", [(8, 0), (8, 1), (256, 0), (256, 1)])
def test_decode_trace_replays_in_a_graph(B, n_slots, overlap):
    """A decode trace captured in a CUDA graph gives the bits of the same
    trace run call by call without overlap: with 8 slots (clusters of CTAs
    per row) and with 256 (one CTA per row, two launches resident at once
    when the overlap option lets the next step start early)."""
    steps, V = 60, 3000
    g0 = np.random.default_rng(3)
    eos = (g0.random((steps, n_slots)) < 0.08).astype(np.uint8)
    rows = [random_rows(n_slots, V, torch.bfloat16, seed=700 + t) for t in range(steps)]
    eos_d = [torch.from_numpy(eos[t]).cuda() for t in range(steps)]
    slot = torch.arange(n_slots, dtype=torch.int32, device="cuda")
    w = torch.linspace(-0.1, 0.3, 11, device="cuda")
    score = torch.zeros(steps, n_slots, device="cuda")
    ship = torch.zeros(steps, n_slots, dtype=torch.uint8, device="cuda")
    fl = torch.zeros(steps, n_slots, dtype=torch.int32, device="cuda")
    ctx = B.pr_ctx_create(0, max_rows=n_slots, max_requests=n_slots)
    try:
        def trace():
            B.pr_ctx_reset(ctx, stream=torch.cuda.current_stream())
            for t in range(steps):
                x, ch = rows[t]
                B.pr_decode_step(ctx, x, slot, ch, eos_d[t], w, -0.1, 0.5, score[t], ship[t],
                                 fl[t])

        B.pr_ctx_set_option(ctx, B.PR_OPT_OVERLAP, 0)
        trace()
        torch.cuda.synchronize()
        ref = (score.clone(), ship.clone(), fl.clone())
        ref_state = B.pr_state_export(ctx)
        for t in (score, ship, fl):
            t.fill_(0)
        B.pr_ctx_set_option(ctx, B.PR_OPT_OVERLAP, overlap)
        g = _capture(trace)
        g.replay()
        torch.cuda.synchronize()
        assert torch.equal(ref[0].view(torch.int32), score.view(torch.int32))
        assert torch.equal(ref[1], ship) and torch.equal(ref[2], fl)
        assert B.pr_state_export(ctx) == ref_state
        assert int(eos.sum()) > 10
    finally:
        B.pr_ctx_destroy(ctx)
