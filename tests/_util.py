"""Shared helpers of the GPU parity tests (comparison rules, random rows)."""
import numpy as np
import torch

RTOL = 1e-4  # float features, aggregates and scores: |gpu - oracle| <= ATOL + RTOL |oracle|
ATOL = 1e-5
SHIP_BAND = 1e-6  # requests whose oracle score is this close to tau are exempt from ship parity


def close_mask(g, o, rtol=RTOL, atol=ATOL):
    g = np.asarray(g, np.float64)
    o = np.asarray(o, np.float64)
    both_nan = np.isnan(g) & np.isnan(o)
    same_inf = np.isinf(g) & np.isinf(o) & (np.sign(g) == np.sign(o))
    with np.errstate(invalid="ignore"):
        ok = np.abs(g - o) <= atol + rtol * np.abs(o)
    return ok | both_nan | same_inf


def assert_close(g, o, what="", rtol=RTOL, atol=ATOL):
    ok = close_mask(g, o, rtol, atol)
    if not ok.all():
        g = np.asarray(g, np.float64)
        o = np.asarray(o, np.float64)
        bad = np.argwhere(~ok)[:8]
        msg = ["%s: %d of %d differ" % (what, (~ok).sum(), ok.size)]
        for i in bad:
            i = tuple(i)
            msg.append("  at %s gpu=%r oracle=%r" % (i, g[i], o[i]))
        raise AssertionError("\n".join(msg))


def assert_ship(ship_g, ship_o, score_o, tau):
    ship_g = np.asarray(ship_g)
    ship_o = np.asarray(ship_o)
    exempt = np.abs(np.asarray(score_o, np.float64) - tau) < SHIP_BAND
    bad = (ship_g != ship_o) & ~exempt
    assert not bad.any(), "ship differs at %s" % np.argwhere(bad)[:8].ravel()


def as_oracle(t: torch.Tensor) -> np.ndarray:
    t = t.detach().cpu().contiguous()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy().view(np.uint16)
    return t.numpy()


def random_rows(n, V, dtype, seed, device="cuda", spike=True, ties=True):
    """Rows with a per-row scale, optional spike and optional exact top ties."""
    g = torch.Generator(device="cpu")
    g.manual_seed(seed)
    s = 0.5 + 3.5 * torch.rand(n, 1, generator=g)
    x = torch.randn(n, V, generator=g) * s
    if spike and V > 1:
        pos = torch.randint(0, V, (n,), generator=g)
        amp = torch.rand(n, generator=g) * 12
        on = torch.rand(n, generator=g) < 0.6
        x[torch.arange(n), pos] += torch.where(on, amp, torch.zeros_like(amp))
    if ties and V > 2:
        for r in range(0, n, 3):
            top = int(torch.argmax(x[r]))
            other = int(torch.randint(0, V, (1,), generator=g))
            x[r, other] = x[r, top]
    x = x.to(dtype)
    chosen = torch.randint(0, V, (n,), generator=g, dtype=torch.int32)
    return x.to(device), chosen.to(device)
