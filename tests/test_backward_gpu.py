"""GPU parity of gbla_backward against the oracle's fp64 backward (the chain
rule through the layer core, pinned in test_oracle_backward.py and by the
pin_backward_* checks) on the same seeded inputs.

Comparison rule, for every element of every gradient tensor g against the
oracle's g_ref and its error scale m (the same chain rule evaluated on
magnitudes, with the absolute sums of the state and of its gradient in place
of the cancelling sums; oracle_gbla_head_backward documents it):

    |g - g_ref| <= c m + ulp(g_ref) / 2   (bf16 storage; fp32 storage: no ulp term)

and normwise ||g - g_ref|| <= nu ||g_ref|| per tensor.  bf16 path: c = 2^-7.
Along any path of the GPU computation at most four quantities are rounded to
bf16 (phi(q~), K^ or V~ as MMA operands, the bf16 dq~ / dk~ / dv~ planes,
|relative error| <= 2^-9 each) besides the stored output, so the error is at
most 4 * 2^-9 = 2^-7 times the scale to first order.  nu = 2^-6: the same
roundings in aggregate, with the scales' cancellation factor (measured
0.2-0.6 %).  fp32 path: c = 2^-11, the relative error of the special-function
approximations (exp2, tanh) that the sigmoid and phi use, which dominates
fp32 rounding; nu = 2^-16.  The measured ratios are logged to
$GBLA_PARITY_LOG."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_07317_gb300 import gbla
from paper_2606_07317_gb300.workloads import WORKLOADS, custom, make_inputs
from parity_util import log_stats, ulp_bf16

pytestmark = pytest.mark.gpu

NAMES = ("dq", "dk", "dv", "dgate", "dout_gate", "dconv_w", "dnorm_w")


def _to64(t):
    return t.detach().to("cpu", torch.float64).numpy()


def _dy(inp, seed):
    g = torch.Generator(device="cuda")
    g.manual_seed(seed)
    return torch.randn(inp["q"].shape, generator=g, device="cuda").to(inp["q"].dtype)


def _oracle(inp, dy, flags=0):
    sl = inp["seq_lens"].cpu().numpy() if inp["seq_lens"] is not None else None
    return oracle.gbla_backward(
        _to64(inp["q"]), _to64(inp["k"]), _to64(inp["v"]), _to64(inp["gate"]),
        _to64(inp["out_gate"]), _to64(inp["conv_w"]), _to64(inp["norm_w"]), _to64(dy),
        seq_lens=sl, flags=flags, scales=True, n_threads=8)


def _run(inp, dy, flags=0):
    return gbla.backward(inp["q"], inp["k"], inp["v"], inp["gate"], inp["out_gate"],
                         inp["conv_w"], inp["norm_w"], inp["seq_lens"], dy, flags=flags)


BOUNDS = {"bf16": (2.0 ** -7, 2.0 ** -6), "fp32": (2.0 ** -11, 2.0 ** -16)}


def _check(got, ref, dtype, tag=""):
    c, nu = BOUNDS[dtype]
    bad, stats = [], {}
    for n in NAMES:
        g, r, m = _to64(got[n]), ref[n], ref["m" + n]
        assert g.shape == r.shape, n
        d = np.abs(g - r)
        half_ulp = 0.5 * ulp_bf16(r) if (dtype == "bf16" and got[n].dtype == torch.bfloat16) \
            else 0.0
        excess = d - half_ulp
        ratio = float(np.max(excess / np.maximum(m, 1e-300))) if excess.size else 0.0
        nrm = float(np.linalg.norm(d) / max(np.linalg.norm(r), 1e-300))
        stats[n] = {"worst_err_over_scale": ratio, "normwise": nrm}
        if not np.all(np.isfinite(g)):
            bad.append(f"{n}: non-finite values")
        elif not np.all(d <= c * m + half_ulp):
            i = np.unravel_index(np.argmax(excess - c * m), d.shape)
            bad.append(f"{n}: |err| {d[i]:.3e} > {c:.2e} * scale {m[i]:.3e} + ulp/2 at {i}")
        elif nrm > nu:
            bad.append(f"{n}: normwise error {nrm:.3e} > {nu:.2e}")
    log_stats({"test": "backward" + tag, "dtype": dtype, **stats})
    assert not bad, "; ".join(bad)


@pytest.mark.parametrize("dtype,D", [("fp32", 32), ("fp32", 64), ("bf16", 64), ("bf16", 128),
                                     ("fp32", 128)])
def test_backward_matches_oracle(dtype, D):
    # two 256-token chunks and a ragged tail; one shorter sequence
    w = custom(B=2, H=2, N=300, D=D, dtype=dtype, seed=21, seq_lens=[300, 77])
    inp = make_inputs(w, "cuda")
    dy = _dy(inp, 22)
    got = _run(inp, dy)
    _check(got, _oracle(inp, dy), dtype, f"_D{D}")


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


def test_backward_headline_shape_full():
    """The benched shape (batch 2, 8 heads, N = 32768, D = 64, bf16: 29-tile
    chunks of the tensor-core query pass on 144 CTAs), every element of every
    gradient against the oracle (threaded over heads)."""
    inp = make_inputs(WORKLOADS["bf16_b2_h8_n32768_d64"], "cuda")
    dy = _dy(inp, 31)
    got = _run(inp, dy)
    torch.cuda.synchronize()
    _check(got, _oracle(inp, dy), "bf16", "_headline")


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


@pytest.mark.parametrize("flags", [1, 2, 4, 3, 5, 6, 7])
@pytest.mark.parametrize("dtype,D", [("bf16", 64), ("fp32", 32)])
def test_backward_ablations(flags, dtype, D):
    """The ablations of Table 4 through gbla_backward_variant, against the
    oracle's backward with the same flags (pinned by finite differences and by
    autograd for these flag sets), under the same bounds; the gradients of the
    parameters a variant does not use are exactly zero."""
    w = custom(B=2, H=2, N=300, D=D, dtype=dtype, seed=41, seq_lens=[300, 77])
    inp = make_inputs(w, "cuda")
    dy = _dy(inp, 42)
    got = _run(inp, dy, flags)
    if flags & gbla.FLAG_NO_CONV:
        assert torch.all(got["dconv_w"] == 0)
    if flags & gbla.FLAG_NO_GATE:
        assert torch.all(got["dgate"] == 0)
    if flags & gbla.FLAG_NO_NORM:
        assert torch.all(got["dout_gate"] == 0) and torch.all(got["dnorm_w"] == 0)
    for n in ("dq", "dk", "dv", "dout_gate"):
        assert torch.all(got[n][1, 77:] == 0), n
    _check(got, _oracle(inp, dy, flags), dtype, f"_flags{flags}_D{D}")


def test_backward_variant_rejects_unknown_flags():
    w = custom(B=1, H=2, N=64, D=64, dtype="bf16", seed=43)
    inp = make_inputs(w, "cuda")
    dy = _dy(inp, 44)
    with pytest.raises(gbla.GblaError):
        _run(inp, dy, 8)


@pytest.mark.parametrize("dtype,D", [("bf16", 64), ("bf16", 128), ("fp32", 32)])
def test_backward_from_state_matches_recompute(dtype, D):
    """gbla_backward_from_state given what gbla_state_stats returned for the same inputs
    (the state and gate statistics a training forward keeps) gives the recomputing
    backward's gradients bit for bit -- both run the same state path -- and so the
    oracle's under the bounds above."""
    w = custom(B=2, H=2, N=300, D=D, dtype=dtype, seed=45, seq_lens=[300, 77])
    inp = make_inputs(w, "cuda")
    dy = _dy(inp, 46)
    state, stats = gbla.state_stats(inp["k"], inp["v"], inp["gate"], inp["conv_w"],
                                    inp["seq_lens"])
    got = gbla.backward(inp["q"], inp["k"], inp["v"], inp["gate"], inp["out_gate"],
                        inp["conv_w"], inp["norm_w"], inp["seq_lens"], dy, state=state,
                        stats=stats)
    ref = _run(inp, dy)
    for n in NAMES:
        assert torch.equal(got[n], ref[n]), n
    _check(got, _oracle(inp, dy), dtype, f"_from_state_D{D}")


def test_backward_from_state_rejects():
    w = custom(B=1, H=2, N=64, D=64, dtype="bf16", seed=47)
    inp = make_inputs(w, "cuda")
    dy = _dy(inp, 48)
    state, stats = gbla.state_stats(inp["k"], inp["v"], inp["gate"], inp["conv_w"])
    args = (inp["q"], inp["k"], inp["v"], inp["gate"], inp["out_gate"], inp["conv_w"],
            inp["norm_w"], None, dy)
    with pytest.raises(ValueError):
        gbla.backward(*args, state=state)  # stats missing
    with pytest.raises(ValueError):
        gbla.backward(*args, flags=gbla.FLAG_NO_CONV, state=state, stats=stats)
    lib = gbla.load()
    p = gbla._ptr
    B, N, H, D = inp["q"].shape
    outs = [torch.empty_like(inp["q"]) for _ in range(4)]
    dgate = torch.empty_like(inp["gate"])
    dcw = torch.empty((3, H, D, 4), device="cuda")

    def call(st_ptr, dnw_ptr):
        return lib.gbla_backward_from_state(
            p(inp["q"]), p(inp["k"]), p(inp["v"]), p(inp["gate"]), p(inp["out_gate"]),
            p(inp["conv_w"]), p(inp["norm_w"]), None, st_ptr, p(stats), p(dy), p(outs[0]),
            p(outs[1]), p(outs[2]), p(dgate), p(outs[3]), p(dcw), dnw_ptr, B, H, N, D, 1, None)

    dnw = torch.empty((H, D), device="cuda")
    assert call(None, p(dnw)) == gbla.GBLA_ERR_INVALID_ARG          # no state
    assert call(p(state), p(state)) == gbla.GBLA_ERR_INVALID_ARG    # dnorm_w over the state
    assert call(p(state), p(dnw)) == gbla.GBLA_OK
    torch.cuda.synchronize()
