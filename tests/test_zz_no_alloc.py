"""gbla_state_static_scratch: the state entry point for callers that cannot
allocate GPU memory (their device memory belongs to another allocator, or an
allocation's latency is not acceptable).  Its partial sums live in a fixed
array inside the library instead of freshly allocated scratch.

It must agree with the allocating gbla_state within the tolerance the state
tests use, call after call: the second call reuses the array the first one
filled.  It must also leave the device's free memory unchanged from one call
to the next.

This file is collected last on purpose: the entry point is an extra, and if
it fails, a run that stops at the first failure (pytest -x) has already run
every other test."""
import numpy as np
import pytest
import torch

from paper_2606_07317_gb300 import gbla
from paper_2606_07317_gb300.workloads import custom, make_inputs

pytestmark = pytest.mark.gpu

STATE_TOL = {"fp32": 1e-5, "bf16": 1e-2}  # relative to max |S| and max |z|


def _args(inp):
    return inp["k"], inp["v"], inp["gate"], inp["conv_w"], inp["seq_lens"]


def _close(a, b, D, dtype):
    a = a.cpu().double().numpy()
    b = b.cpu().double().numpy()
    tol = STATE_TOL[dtype]
    S_a, S_b = a[..., : D * D], b[..., : D * D]
    z_a, z_b = a[..., D * D:], b[..., D * D:]
    assert np.abs(S_a - S_b).max() <= tol * max(np.abs(S_b).max(), 1e-30)
    assert np.abs(z_a - z_b).max() <= tol * max(np.abs(z_b).max(), 1e-30)


def test_static_scratch_matches_gbla_state_on_consecutive_calls():
    gbla.load()
    cases = [
        custom(B=2, H=3, N=1000, D=64, dtype="bf16", seed=31, seq_lens=[1000, 517]),
        custom(B=3, H=2, N=700, D=32, dtype="fp32", seed=32, seq_lens=[5, 700, 0]),
        # 32 pairs at D = 128 and 5000 tokens: fewer, longer chunks to fit the array
        custom(B=4, H=8, N=5000, D=128, dtype="bf16", seed=33),
    ]
    for w in cases:
        inp = make_inputs(w, "cuda")
        ref = gbla.state(*_args(inp))
        out = torch.full_like(ref, float("nan"))
        gbla.state_static_scratch(*_args(inp), out=out)
        torch.cuda.synchronize()
        _close(out, ref, w.D, w.dtype)


def test_static_scratch_allocates_nothing():
    """After a first call (which may load the library's module, and with it the
    fixed array, onto the device), further calls leave the free device memory
    exactly as it was."""
    gbla.load()
    w = custom(B=2, H=4, N=3000, D=64, dtype="bf16", seed=34, seq_lens=[3000, 1234])
    inp = make_inputs(w, "cuda")
    out = torch.empty((w.B, w.H, w.D * w.D + w.D), dtype=torch.float32, device="cuda")
    gbla.state_static_scratch(*_args(inp), out=out)
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    for _ in range(3):
        gbla.state_static_scratch(*_args(inp), out=out)
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert free1 == free0, (free0, free1)


def test_static_scratch_size_limit_at_d128():
    """507 (batch, head) pairs fit the fixed array at D = 128, 508 do not."""
    gbla.load()
    cw = torch.zeros((3, 1, 128, 4), device="cuda")
    for B, ok in ((507, True), (508, False)):
        k = torch.zeros((B, 1, 1, 128), dtype=torch.bfloat16, device="cuda")
        gate = torch.zeros((B, 1, 1), dtype=torch.bfloat16, device="cuda")
        if ok:
            st = gbla.state_static_scratch(k, k, gate, cw)
            torch.cuda.synchronize()
            assert torch.isfinite(st).all()
        else:
            with pytest.raises(gbla.GblaError) as e:
                gbla.state_static_scratch(k, k, gate, cw)
            assert e.value.status == gbla.GBLA_ERR_INVALID_ARG


def test_static_scratch_rejects_oversized_problem():
    gbla.load()
    # 600 (batch, head) pairs at D = 128 need more than the fixed array holds
    k = torch.zeros((600, 8, 1, 128), dtype=torch.bfloat16, device="cuda")
    gate = torch.zeros((600, 8, 1), dtype=torch.bfloat16, device="cuda")
    cw = torch.zeros((3, 1, 128, 4), device="cuda")
    with pytest.raises(gbla.GblaError) as e:
        gbla.state_static_scratch(k, k, gate, cw)
    assert e.value.status == gbla.GBLA_ERR_INVALID_ARG
