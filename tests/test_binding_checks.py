"""The Python binding refuses, before anything reaches the library, tensors
that the C ABI would take as device pointers but that are not CUDA tensors on
the call's device (a host tensor handed to a kernel would be an illegal
address on the GPU), as well as wrong dtypes and short output buffers.  Runs
on the CPU: every call below must raise PRError without launching anything."""
import numpy as np
import pytest
import torch

from paper_2608_28726_gb300 import build as prbuild

prbuild.build()
from paper_2608_28726_gb300 import binding as B  # noqa: E402


def _host_batch(n=4, V=64, n_req=2):
    x = torch.zeros(n, V, dtype=torch.bfloat16)
    ch = torch.zeros(n, dtype=torch.int32)
    off = torch.tensor([0, 2, n], dtype=torch.int64)
    w = torch.zeros(11, dtype=torch.float32)
    return x, ch, off, w


def _raises_invalid(fn, *a, **k):
    n0 = B.launch_count()
    with pytest.raises(B.PRError) as e:
        fn(*a, **k)
    assert e.value.status in (B.PR_ERR_INVALID_ARG, B.PR_ERR_UNSUPPORTED)
    assert B.launch_count() == n0
    return str(e.value)


def test_host_tensors_are_refused_by_device_calls():
    x, ch, off, w = _host_batch()
    msg = _raises_invalid(B.pr_route, None, x, ch, off, w, 0.0, 0.5)
    assert "CUDA tensor" in msg
    _raises_invalid(B.pr_token_features, None, x, ch)
    feat = torch.zeros(4, 8)
    _raises_invalid(B.pr_aggregate_score, None, feat, off, w, 0.0, 0.5)
    _raises_invalid(B.pr_decode_step, None, x, ch, ch, torch.zeros(4, dtype=torch.uint8), w, 0.0,
                    0.5, torch.zeros(4), torch.zeros(4, dtype=torch.uint8),
                    torch.zeros(4, dtype=torch.int32))
    _raises_invalid(B.pr_head_score, None, feat, off, torch.zeros(B.pr_head_param_count(2)), 2,
                    0.5)
    _raises_invalid(B.pr_quantile_score, None, feat, off, torch.zeros(B.PR_QMLP_PARAMS), 0.5)
    _raises_invalid(B.pr_selective_metrics, None, torch.zeros(10), 0.5)
    h = torch.zeros(2, 64, dtype=torch.bfloat16)
    _raises_invalid(B.pr_lmhead_features, None, h, torch.zeros(256, 64, dtype=torch.bfloat16),
                    torch.zeros(2, dtype=torch.int32))
    _raises_invalid(B.pr_route_noalloc, x, ch, off, w, 0.0, 0.5, torch.zeros(2),
                    torch.zeros(2, dtype=torch.uint8), torch.zeros(2, dtype=torch.int32))


def test_numpy_arrays_are_refused_by_device_calls():
    x, ch, off, w = _host_batch()
    _raises_invalid(B.pr_selective_metrics, None, np.zeros(10, np.float32), 0.5)


def test_checks_name_the_offending_argument(monkeypatch):
    """With the device check passed (faked here: no GPU on this machine), the
    dtype, contiguity and size checks still stop the call."""
    call = "pr_route"
    t = torch.zeros(3, dtype=torch.int64)
    # the check helper on its own, with a fake device tensor
    fake = torch.zeros(3, dtype=torch.int64)
    monkeypatch.setattr(torch.Tensor, "is_cuda", property(lambda self: True))
    monkeypatch.setattr(torch.Tensor, "device", property(lambda self: torch.device("cuda", 0)))
    with pytest.raises(B.PRError, match="chosen has dtype"):
        B._dev(call, 0, "chosen", fake, B._I32_T, 3)
    with pytest.raises(B.PRError, match="holds 3 elements, the call needs 4"):
        B._dev(call, 0, "offsets", t, B._I64_T, 4)
    with pytest.raises(B.PRError, match="must be contiguous"):
        B._dev(call, 0, "agg", torch.zeros(4, 11).t(), B._F32_T)
    with pytest.raises(B.PRError, match="on cuda:1"):
        B._dev(call, 1, "score", torch.zeros(4), B._F32_T)
    B._dev(call, 0, "score", torch.zeros(4), B._F32_T, 4)  # passes
    B._dev(call, 0, "agg", None, B._F32_T, 44, optional=True)  # optional and absent
    with pytest.raises(B.PRError, match="is required"):
        B._dev(call, 0, "w", None, B._F32_T)


def test_host_call_refuses_device_tensors(monkeypatch):
    x, ch, off, w = _host_batch()
    monkeypatch.setattr(torch.Tensor, "is_cuda", property(lambda self: True))
    _raises_invalid(B.pr_route_host, None, x, ch, off, w, 0.0, 0.5)
