"""GPU parity of gbla_backward against the oracle's fp64 backward (the chain
rule through the layer core, pinned in test_oracle_backward.py) on the same
seeded inputs.

Comparison rule (per gradient tensor, normwise-max): max |g - g_ref| <=
tol * max |g_ref| + 1e-6, tol = 1e-4 for fp32 storage (fp32 arithmetic
throughout) and 2e-2 for bf16 storage (bf16 outputs carry 2^-9 relative
rounding, and the recomputed forward state has the bf16-operand contraction's
error, as the forward's own tolerance allows)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_07317_gb300 import gbla
from paper_2606_07317_gb300.workloads import custom, make_inputs

pytestmark = pytest.mark.gpu

NAMES = ("dq", "dk", "dv", "dgate", "dout_gate", "dconv_w", "dnorm_w")


def _to64(t):
    return t.detach().to("cpu", torch.float64).numpy()


def _dy(inp, seed):
    g = torch.Generator(device="cuda")
    g.manual_seed(seed)
    return torch.randn(inp["q"].shape, generator=g, device="cuda").to(inp["q"].dtype)


def _oracle(inp, dy):
    sl = inp["seq_lens"].cpu().numpy() if inp["seq_lens"] is not None else None
    return oracle.gbla_backward(
        _to64(inp["q"]), _to64(inp["k"]), _to64(inp["v"]), _to64(inp["gate"]),
        _to64(inp["out_gate"]), _to64(inp["conv_w"]), _to64(inp["norm_w"]), _to64(dy),
        seq_lens=sl)


def _run(inp, dy):
    return gbla.backward(inp["q"], inp["k"], inp["v"], inp["gate"], inp["out_gate"],
                         inp["conv_w"], inp["norm_w"], inp["seq_lens"], dy)


def _check(got, ref, dtype):
    tol = 1e-4 if dtype == "fp32" else 2e-2
    bad = []
    for n in NAMES:
        g, r = _to64(got[n]), ref[n]
        assert g.shape == r.shape, n
        err = float(np.abs(g - r).max())
        scale = float(np.abs(r).max())
        if not (np.all(np.isfinite(g)) and err <= tol * scale + 1e-6):
            bad.append(f"{n}: max err {err:.3e} vs max |ref| {scale:.3e}")
    assert not bad, "; ".join(bad)


@pytest.mark.parametrize("dtype,D", [("fp32", 32), ("fp32", 64), ("bf16", 64), ("bf16", 128),
                                     ("fp32", 128)])
def test_backward_matches_oracle(dtype, D):
    # two 256-token chunks and a ragged tail; one shorter sequence
    w = custom(B=2, H=2, N=300, D=D, dtype=dtype, seed=21, seq_lens=[300, 77])
    inp = make_inputs(w, "cuda")
    dy = _dy(inp, 22)
    got = _run(inp, dy)
    _check(got, _oracle(inp, dy), dtype)


def test_backward_full_length_bf16():
    w = custom(B=1, H=4, N=1000, D=64, dtype="bf16", seed=23)
    inp = make_inputs(w, "cuda")
    dy = _dy(inp, 24)
    _check(_run(inp, dy), _oracle(inp, dy), "bf16")


def test_backward_padding_rows_zero_and_deterministic():
    w = custom(B=3, H=2, N=260, D=64, dtype="bf16", seed=25, seq_lens=[260, 5, 0])
    inp = make_inputs(w, "cuda")
    dy = _dy(inp, 26)
    a = _run(inp, dy)
    b = _run(inp, dy)
    for n in NAMES:
        assert torch.equal(a[n], b[n]), n
    for n in ("dq", "dk", "dv", "dout_gate"):
        assert torch.all(a[n][1, 5:] == 0) and torch.all(a[n][2] == 0), n
    assert torch.all(a["dgate"][1, 5:] == 0) and torch.all(a["dgate"][2] == 0)
    _check(a, _oracle(inp, dy), "bf16")


def test_backward_ragged_chunks_bf16():
    """Sequences spanning several 1024-token chunks of the tensor-core query pass,
    lengths that are not multiples of the 128-token tile, an empty sequence and
    a chunk lying wholly in the padding; padded rows zero."""
    w = custom(B=3, H=2, N=2500, D=64, dtype="bf16", seed=29, seq_lens=[2500, 1100, 0])
    inp = make_inputs(w, "cuda")
    dy = _dy(inp, 30)
    got = _run(inp, dy)
    for n in ("dq", "dk", "dv", "dout_gate"):
        assert torch.all(got[n][1, 1100:] == 0) and torch.all(got[n][2] == 0), n
    assert torch.all(got["dgate"][1, 1100:] == 0) and torch.all(got["dgate"][2] == 0)
    _check(got, _oracle(inp, dy), "bf16")


def test_backward_rejects_aliasing():
    w = custom(B=1, H=2, N=64, D=64, dtype="bf16", seed=27)
    inp = make_inputs(w, "cuda")
    dy = _dy(inp, 28)
    lib = gbla.load()
    p = gbla._ptr
    B, N, H, D = inp["q"].shape
    dq = torch.empty_like(inp["q"])
    others = [torch.empty_like(inp["q"]) for _ in range(3)]
    dgate = torch.empty_like(inp["gate"])
    dcw = torch.empty((3, H, D, 4), device="cuda")
    dnw = torch.empty((H, D), device="cuda")
    # dq aliasing the input q
    st = lib.gbla_backward(p(inp["q"]), p(inp["k"]), p(inp["v"]), p(inp["gate"]),
                           p(inp["out_gate"]), p(inp["conv_w"]), p(inp["norm_w"]), None, p(dy),
                           p(inp["q"]), p(others[0]), p(others[1]), p(dgate), p(others[2]),
                           p(dcw), p(dnw), B, H, N, D, 1, None)
    assert st == 1  # GBLA_ERR_INVALID_ARG
    # dk aliasing dq
    st = lib.gbla_backward(p(inp["q"]), p(inp["k"]), p(inp["v"]), p(inp["gate"]),
                           p(inp["out_gate"]), p(inp["conv_w"]), p(inp["norm_w"]), None, p(dy),
                           p(dq), p(dq), p(others[1]), p(dgate), p(others[2]), p(dcw), p(dnw),
                           B, H, N, D, 1, None)
    assert st == 1
