"""GPU parity of the layer front end (gbla_project: X-space Conv1D and the
stacked Q, K, V, R, w_g projections of Sec. 2.1) and of the whole layer
(gbla_layer_forward) against the oracle, through the C ABI.

Comparison rule for gbla_project (bf16 in and out), per output element y with
the oracle's fp64 value y_ref and magnitude sum A = sum_c |x~_c w_c|:

    |y - y_ref| <= E + ulp_bf16(|y_ref| + E) / 2 + 1e-4,
    E = A (2^-8 + d 2^-23)

The kernel rounds X~ once to bf16 (relative error <= 2^-8 per term), sums d
products in fp32 (<= d 2^-23 A with room for the tensor core's summation
order) and rounds the result once to bf16 (half an ulp); 1e-4 covers the fp32
Conv1D itself.  A second, statistical check bounds the normwise error of each
output tensor of 256 or more elements by 2^-7 (rounding noise is about 2^-8
of the norm)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_07317_gb300 import gbla
from paper_2606_07317_gb300.workloads import make_layer_inputs
from parity_util import ulp_bf16

pytestmark = pytest.mark.gpu

STREAMS = ("q", "k", "v", "out_gate", "gate")


def _to64(t):
    return t.detach().to("cpu", torch.float64).numpy()


def _oracle_project(inp, H, D):
    sl = inp["seq_lens"].cpu().numpy() if inp["seq_lens"] is not None else None
    return oracle.gbla_project(_to64(inp["x"]), _to64(inp["conv_x"]), _to64(inp["w_proj"]),
                               H, D, seq_lens=sl, absdot=True)


def _absdot_of(ref, H, D):
    """Split the oracle's [B, N, F] magnitude sums like the outputs."""
    A = ref["absdot"]
    B, N, _ = A.shape
    HD = H * D
    parts = {n: A[..., s * HD:(s + 1) * HD].reshape(B, N, H, D)
             for s, n in enumerate(("q", "k", "v", "out_gate"))}
    parts["gate"] = A[..., 4 * HD:]
    return parts


def _check_project(out, ref, d, H, D, lens):
    A = _absdot_of(ref, H, D)
    bad = []
    for n in STREAMS:
        g = _to64(out[n])
        r = ref[n]
        for b, L in enumerate(lens):
            gv, rv, av = g[b, :L], r[b, :L], A[n][b, :L]
            E = av * (2.0 ** -8 + d * 2.0 ** -23)
            bound = E + 0.5 * ulp_bf16(np.abs(rv) + E) + 1e-4
            err = np.abs(gv - rv)
            if not np.all(np.isfinite(gv)) or np.any(err > bound):
                i = np.unravel_index(np.argmax(err - bound), err.shape)
                bad.append(f"{n}[b={b}] at {i}: |d|={err[i]:.3e} > {bound[i]:.3e}")
            nw = np.linalg.norm(gv - rv) / max(np.linalg.norm(rv), 1e-30)
            if gv.size >= 256 and nw > 2.0 ** -7:  # a statistical bound: many elements
                bad.append(f"{n}[b={b}] normwise error {nw:.3e}")
    assert not bad, "; ".join(bad[:6])


def _inputs(B, N, d, H, D, seed, seq_lens=None):
    return make_layer_inputs(B, N, d, H, D, seed=seed, seq_lens=seq_lens, device="cuda")


def _sentinel_out(B, N, H, D):
    out = {n: torch.full((B, N, H, D), 7.0, device="cuda", dtype=torch.bfloat16)
           for n in ("q", "k", "v", "out_gate")}
    out["gate"] = torch.full((B, N, H), 7.0, device="cuda", dtype=torch.bfloat16)
    return out


# (B, N, d, H, D, seq_lens): several 128-token tiles with a ragged tail, every
# d block count, head layouts whose 256-column chunks span two streams
# (H D = 192), D = 32, 64, 128, and tiles wholly inside the padding.
CASES = [
    (2, 300, 512, 8, 64, [300, 77]),
    (1, 260, 64, 2, 32, None),
    (2, 200, 192, 3, 64, [200, 1]),
    (1, 384, 256, 4, 128, None),
    (3, 129, 320, 1, 64, [129, 128, 0]),
]


@pytest.mark.parametrize("B,N,d,H,D,sl", CASES,
                         ids=[f"b{c[0]}_n{c[1]}_d{c[2]}_h{c[3]}_D{c[4]}" for c in CASES])
def test_project_matches_oracle(B, N, d, H, D, sl):
    inp = _inputs(B, N, d, H, D, seed=11 + d + H, seq_lens=sl)
    out = _sentinel_out(B, N, H, D)
    gbla.project(inp["x"], inp["conv_x"], inp["w_proj"], H, D, seq_lens=inp["seq_lens"],
                 out=out)
    torch.cuda.synchronize()
    assert gbla.device_error() == 0
    lens = sl if sl is not None else [N] * B
    ref = _oracle_project(inp, H, D)
    _check_project(out, ref, d, H, D, lens)
    # rows past seq_lens[b] are not written
    for n in STREAMS:
        g = out[n].float().cpu()
        for b, L in enumerate(lens):
            assert torch.all(g[b, L:] == 7.0), n


def test_project_deterministic():
    B, N, d, H, D = 2, 640, 512, 8, 64
    inp = _inputs(B, N, d, H, D, seed=5)
    a = gbla.project(inp["x"], inp["conv_x"], inp["w_proj"], H, D)
    b = gbla.project(inp["x"], inp["conv_x"], inp["w_proj"], H, D)
    torch.cuda.synchronize()
    for n in STREAMS:
        assert torch.equal(a[n], b[n]), n


def test_project_full_size_sampled():
    """The headline shape (B = 2, N = 32768, d = 512, 8 heads of 64) in the
    launch configuration the benchmark times; rows checked against the oracle
    one by one: every tile's first and last rows plus random rows."""
    B, N, d, H, D = 2, 32768, 512, 8, 64
    inp = _inputs(B, N, d, H, D, seed=3)
    out = gbla.project(inp["x"], inp["conv_x"], inp["w_proj"], H, D)
    torch.cuda.synchronize()
    assert gbla.device_error() == 0
    rng = np.random.default_rng(0)
    rows = sorted(set([0, 1, 2, 3, 127, 128, 129, N - 1] + list(range(255, N, 4096)) +
                      list(range(4096, N, 4096)) + list(rng.integers(0, N, 24))))
    x64 = _to64(inp["x"])
    cx, w = _to64(inp["conv_x"]), _to64(inp["w_proj"])
    for b in range(B):
        for t in rows:
            lo = max(0, t - 3)
            # a causal window: the slice's last row sees exactly rows t-3..t
            r = oracle.gbla_project(x64[b:b + 1, lo:t + 1], cx, w, H, D, absdot=True)
            one = {n: r[n][:, -1:] for n in STREAMS}
            one["absdot"] = r["absdot"][:, -1:]
            got = {n: out[n][b:b + 1, t:t + 1] for n in STREAMS}
            _check_project(got, one, d, H, D, [1])


def test_project_rejects():
    B, N, d, H, D = 1, 128, 128, 2, 32
    inp = _inputs(B, N, d, H, D, seed=1)
    lib = gbla.load()
    out = _sentinel_out(B, N, H, D)
    s = gbla._stream(None)
    P = gbla._ptr

    def call(x, cx, w, q, k, v, og, g, dd=d, HH=H, DD=D, dt=gbla.GBLA_BF16):
        return lib.gbla_project(P(x), P(cx), P(w), None, P(q), P(k), P(v), P(og), P(g),
                                B, N, dd, HH, DD, dt, s)

    args = (inp["x"], inp["conv_x"], inp["w_proj"], out["q"], out["k"], out["v"],
            out["out_gate"], out["gate"])
    assert call(*args) == gbla.GBLA_OK
    assert call(*args, dt=gbla.GBLA_FP32) == gbla.GBLA_ERR_UNSUPPORTED
    assert call(*args, dd=96) == gbla.GBLA_ERR_UNSUPPORTED      # d not a multiple of 64
    assert call(*args, dd=1024) == gbla.GBLA_ERR_UNSUPPORTED    # d above the resident tile
    assert call(*args, HH=1) == gbla.GBLA_ERR_UNSUPPORTED       # H D = 32
    alias = list(args)
    alias[4] = out["q"]                                         # k output = q output
    assert call(*alias) == gbla.GBLA_ERR_INVALID_ARG
    alias = list(args)
    alias[3] = inp["x"]                                         # q output over x
    assert call(*alias) == gbla.GBLA_ERR_INVALID_ARG
    torch.cuda.synchronize()


def test_layer_is_project_then_core():
    """gbla_layer_forward equals gbla_project followed by the core with its
    Conv1D off, bit for bit."""
    B, N, d, H, D = 2, 700, 512, 8, 64
    sl = [700, 300]
    inp = _inputs(B, N, d, H, D, seed=9, seq_lens=sl)
    y = gbla.layer_forward(inp["x"], inp["conv_x"], inp["w_proj"], inp["norm_w"], H, D,
                           seq_lens=inp["seq_lens"])
    pr = gbla.project(inp["x"], inp["conv_x"], inp["w_proj"], H, D, seq_lens=inp["seq_lens"])
    unused_taps = torch.zeros((3, H, D, 4), device="cuda")
    y2 = gbla.forward(pr["q"], pr["k"], pr["v"], pr["gate"], pr["out_gate"], unused_taps,
                      inp["norm_w"], seq_lens=inp["seq_lens"], flags=gbla.FLAG_NO_CONV)
    torch.cuda.synchronize()
    for b, L in enumerate(sl):
        assert torch.equal(y[b, :L], y2[b, :L])


@pytest.mark.parametrize("N,sl", [(1024, None), (2048, [2048, 555])])
def test_layer_matches_oracle(N, sl):
    """The whole layer against the oracle's layer, which stores the front end's
    outputs in bf16 between the two halves as the library does (round to
    nearest).

    Tolerance, derived from the oracle alone: the library's intermediates are
    the bf16 rounding of fp32 values that carry X~'s bf16 rounding, so they
    differ from the oracle's by one bf16 ulp at a fraction of the elements
    (about 40 % here), whereas storing in bf16 at all moves every element by
    up to half an ulp (an RMS of 0.29 ulp).  The first perturbation is at most
    sqrt(0.5) / 0.29 < 2.5 times the second in norm, so o may differ from the
    oracle's by 3 times the effect the oracle measures for the bf16 storage
    (its layer with and without the rounding), normwise and elementwise, plus
    half a bf16 ulp of the stored o."""
    B, d, H, D = 2 if sl else 1, 512, 8, 64
    inp = _inputs(B, N, d, H, D, seed=21, seq_lens=sl)
    y = gbla.layer_forward(inp["x"], inp["conv_x"], inp["w_proj"], inp["norm_w"], H, D,
                           seq_lens=inp["seq_lens"])
    torch.cuda.synchronize()

    def to_bf16(a):
        return torch.from_numpy(np.ascontiguousarray(a)).to(torch.bfloat16).to(
            torch.float64).numpy()

    args = (_to64(inp["x"]), _to64(inp["conv_x"]), _to64(inp["w_proj"]), _to64(inp["norm_w"]),
            H, D)
    ref = oracle.gbla_layer(*args, seq_lens=sl, store=to_bf16)
    exact = oracle.gbla_layer(*args, seq_lens=sl)
    lens = sl if sl is not None else [N] * B
    g = _to64(y)
    for b, L in enumerate(lens):
        gv, rv, ev = g[b, :L], ref[b, :L], exact[b, :L]
        s_max = float(np.abs(rv - ev).max())
        s_norm = float(np.linalg.norm(rv - ev) / np.linalg.norm(ev))
        err = np.abs(gv - rv)
        nw = float(np.linalg.norm(gv - rv) / np.linalg.norm(rv))
        assert np.all(np.isfinite(gv))
        assert nw <= 3 * s_norm, (nw, s_norm)
        excess = err - (3 * s_max + 0.5 * ulp_bf16(rv))
        assert float(excess.max()) <= 0.0, (float(err.max()), s_max)
