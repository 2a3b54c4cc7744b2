"""GPU path vs the fp64 oracle on the same seeded inputs, through the C ABI.

Tolerances (see parity_util): fp32 max |d| / max(|y|, 1) <= 1e-4; bf16
|d| <= 2e-2 + half a bf16 ulp of the true value.  Rows past a sequence's end
must keep the sentinel the output was filled with.
"""
import numpy as np
import pytest
import torch

from paper_2606_07317_gb300 import gbla
from paper_2606_07317_gb300.workloads import WORKLOADS, custom, make_inputs
from parity_util import (compare, compare_prenorm, log_stats, oracle_full, oracle_head,
                         oracle_rows, to64, valid_mask)

pytestmark = pytest.mark.gpu

SENTINEL = -777.0
ALGOS = {"auto": gbla.ALGO_AUTO, "simt": gbla.ALGO_SIMT}
# The benchmark spec's bound on the bf16 path's computation error after the gated
# RMSNorm, applied literally to the fp32 output of gbla_forward_f32out.
LITERAL_ABS_TOL = 2e-2

_INPUTS, _REFS = {}, {}


def _named(name):
    """Seeded inputs (on the GPU) and the oracle per batch row, computed once per
    workload for the whole module."""
    if name not in _INPUTS:
        inp = make_inputs(WORKLOADS[name], "cuda")
        _INPUTS[name] = inp
        _REFS[name] = oracle_rows(inp)
    return _INPUTS[name], _REFS[name]


def _rows_vs_ref(y_t, refs, lens):
    """(gpu valid rows, oracle valid rows) as flat float64 arrays, plus a check that
    every padded row still holds the sentinel."""
    yc = y_t.cpu()
    ys, rs = [], []
    for b, L in enumerate(lens):
        ys.append(to64(yc[b, :L]).ravel())
        rs.append(refs[b].ravel())
        if L < yc.shape[1]:
            assert torch.all(yc[b, L:] == torch.tensor(SENTINEL, dtype=yc.dtype)), \
                f"rows past the end of sequence {b} were written"
    return np.concatenate(ys), np.concatenate(rs)


@pytest.fixture(scope="module", autouse=True)
def _lib():
    gbla.load()
    torch.cuda.init()


def _run(inp, algo=gbla.ALGO_AUTO):
    out = torch.full_like(inp["q"], SENTINEL)
    gbla.forward(inp["q"], inp["k"], inp["v"], inp["gate"], inp["out_gate"],
                 inp["conv_w"], inp["norm_w"], inp["seq_lens"], out=out, algo=algo)
    torch.cuda.synchronize()
    return out


def _check_against(y_gpu_t, y_ref, inp, dtype):
    B, N = inp["q"].shape[:2]
    sl = inp["seq_lens"]
    mask = valid_mask(B, N, None if sl is None else sl.cpu().numpy())
    y_gpu = to64(y_gpu_t)
    st = compare(y_gpu[mask], y_ref[mask], dtype)
    assert st["ok"], st
    pad = y_gpu[~mask]
    assert np.all(pad == np.float64(torch.tensor(SENTINEL, dtype=y_gpu_t.dtype).item())), \
        "rows past the sequence end were written"
    return st


@pytest.mark.parametrize("algo", list(ALGOS), ids=list(ALGOS))
@pytest.mark.parametrize("name", ["tiny_fp32_b1_h2_n256_d32", "bf16_b8_h8_n2048_d64",
                                  "bf16_b4_h8_n8192_d64"])
def test_parity_workload(name, algo):
    w = WORKLOADS[name]
    inp, refs = _named(name)
    y = _run(inp, ALGOS[algo])
    st = compare(*_rows_vs_ref(y, refs, w.lengths()), w.dtype)
    log_stats({"test": "parity", "workload": name, "algo": algo, **st})
    assert st["ok"], st


def test_parity_headline_n32768():
    name = "bf16_b2_h8_n32768_d64"
    w = WORKLOADS[name]
    inp, refs = _named(name)
    y = _run(inp)
    st = compare(*_rows_vs_ref(y, refs, w.lengths()), w.dtype)
    log_stats({"test": "parity", "workload": name, "algo": "auto", **st})
    assert st["ok"], st


def test_parity_ragged_d128():
    """Full-size ragged workload (32 rows, log-normal lengths up to 32768, D = 128):
    every one of the 32 x 8 (batch, head) sequences against the oracle, element by
    element, and every padded row left untouched."""
    name = "bf16_ragged_b32_h8_d128"
    w = WORKLOADS[name]
    inp, refs = _named(name)
    y = _run(inp)
    st = compare(*_rows_vs_ref(y, refs, w.lengths()), "bf16")
    log_stats({"test": "parity", "workload": name, "algo": "auto", **st})
    assert st["ok"], st


@pytest.mark.parametrize("algo", list(ALGOS), ids=list(ALGOS))
@pytest.mark.parametrize("name", ["bf16_b8_h8_n2048_d64", "bf16_b4_h8_n8192_d64",
                                  "bf16_b2_h8_n32768_d64", "bf16_ragged_b32_h8_d128"])
def test_literal_budget_before_output_rounding(name, algo):
    """The bf16 path's own arithmetic error, apart from the rounding of its stored
    output: gbla_forward_f32out runs the same kernels and stores y in fp32.  Its
    max |y - y_ref| must be <= 2e-2 literally (Sec. 2.1 item 3 output), and rounding
    it to bf16 must give gbla_forward's output bit for bit (same arithmetic)."""
    w = WORKLOADS[name]
    inp, refs = _named(name)
    y16 = _run(inp, ALGOS[algo])
    y32 = torch.full(inp["q"].shape, SENTINEL, dtype=torch.float32, device="cuda")
    gbla.forward_f32out(inp["q"], inp["k"], inp["v"], inp["gate"], inp["out_gate"],
                        inp["conv_w"], inp["norm_w"], inp["seq_lens"], out=y32,
                        algo=ALGOS[algo])
    torch.cuda.synchronize()
    g32, r = _rows_vs_ref(y32, refs, w.lengths())
    g16, _ = _rows_vs_ref(y16, refs, w.lengths())
    assert torch.equal(y32.to(torch.bfloat16), y16), "f32 output rounds to a different o"
    d32, d16 = np.abs(g32 - r), np.abs(g16 - r)
    rec = {"test": "literal", "workload": name, "algo": algo,
           "max_abs_before_rounding": float(d32.max()),
           "max_abs_after_rounding": float(d16.max()),
           "rms_err_before_rounding": float(np.sqrt(np.mean(d32 ** 2))),
           "max_abs_ref": float(np.abs(r).max()), "elements": int(r.size)}
    log_stats(rec)
    assert np.all(np.isfinite(g32)), rec
    assert rec["max_abs_before_rounding"] <= LITERAL_ABS_TOL, rec


@pytest.mark.parametrize("algo", list(ALGOS), ids=list(ALGOS))
@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
@pytest.mark.parametrize("D", [32, 64, 128])
def test_edge_lengths_and_garbage_padding(D, dtype, algo):
    """Lengths 0..3 (shorter than the conv), a ragged tail, a full row; the
    padding holds NaN and huge logits, which must not leak into valid rows."""
    lens = [0, 1, 2, 3, 129, 333]
    w = custom(B=len(lens), H=2, N=333, D=D, dtype=dtype, seed=7, seq_lens=lens)
    inp = make_inputs(w, "cuda")
    for b, L in enumerate(lens):
        for name in ("q", "k", "v", "out_gate"):
            inp[name][b, L:] = float("nan")
        inp["gate"][b, L:] = 1e30 if dtype == "fp32" else 1e30
    y = _run(inp, ALGOS[algo])
    _check_against(y, oracle_full(inp), inp, dtype)


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
def test_state_matches_oracle(dtype):
    """gbla_state writes S = K^T V~ and z = K^T 1 with the true softmax gate."""
    w = custom(B=2, H=3, N=1000, D=64, dtype=dtype, seed=11, seq_lens=[1000, 517])
    inp = make_inputs(w, "cuda")
    st = gbla.state(inp["k"], inp["v"], inp["gate"], inp["conv_w"], inp["seq_lens"])
    torch.cuda.synchronize()
    st = st.cpu().double().numpy()
    tol = 1e-5 if dtype == "fp32" else 1e-2
    for b in range(2):
        for h in range(3):
            _, inter = oracle_head(inp, b, h, intermediates=True)
            S = st[b, h, :64 * 64].reshape(64, 64)
            z = st[b, h, 64 * 64:]
            assert np.abs(S - inter["S"]).max() <= tol * np.abs(inter["S"]).max()
            assert np.abs(z - inter["z"]).max() <= tol * np.abs(inter["z"]).max()


def test_readout_scale_invariant():
    """A positive common scale of S and z cancels in the readout."""
    w = custom(B=1, H=2, N=700, D=64, dtype="bf16", seed=12)
    inp = make_inputs(w, "cuda")
    st = gbla.state(inp["k"], inp["v"], inp["gate"], inp["conv_w"])
    o1 = gbla.readout(inp["q"], inp["out_gate"], inp["conv_w"], inp["norm_w"], st)
    o2 = gbla.readout(inp["q"], inp["out_gate"], inp["conv_w"], inp["norm_w"], st * 4.0)
    torch.cuda.synchronize()
    assert torch.equal(o1, o2)


@pytest.mark.parametrize("name", ["bf16_b8_h8_n2048_d64", "tiny_fp32_b1_h2_n256_d32"])
def test_deterministic(name):
    inp = make_inputs(WORKLOADS[name], "cuda")
    assert torch.equal(_run(inp), _run(inp))


def test_large_gate_logits():
    """Logits near the fp32 exp overflow limit: the max-rescaled gate is stable."""
    w = custom(B=2, H=2, N=600, D=64, dtype="bf16", seed=13)
    inp = make_inputs(w, "cuda")
    inp["gate"].mul_(30.0).add_(500.0)
    y = _run(inp)
    _check_against(y, oracle_full(inp), inp, "bf16")


def test_host_entry_matches_device():
    w = custom(B=3, H=2, N=500, D=64, dtype="bf16", seed=14, seq_lens=[500, 77, 0])
    inp = make_inputs(w, "cuda")
    y_dev = _run(inp)
    host = {k_: (v_.cpu().pin_memory() if v_ is not None else None) for k_, v_ in inp.items()}
    out = torch.full_like(host["q"], SENTINEL).pin_memory()
    gbla.forward_host(host["q"], host["k"], host["v"], host["gate"], host["out_gate"],
                      host["conv_w"], host["norm_w"], host["seq_lens"], out=out)
    assert torch.equal(out, y_dev.cpu())


@pytest.mark.parametrize("dtype,D", [("bf16", 64), ("bf16", 128), ("fp32", 32)])
def test_host_entry_chunks_match_device(dtype, D):
    """gbla_forward_host reads out in chunks of 4096 tokens, each seeing the 3 rows
    before it as conv history: lengths at, just past and just short of chunk edges
    give gbla_forward's o bit for bit, and padded rows keep their sentinel."""
    w = custom(B=4, H=2, N=9000, D=D, dtype=dtype, seed=16,
               seq_lens=[9000, 4096, 4099, 8191])
    inp = make_inputs(w, "cuda")
    y_dev = _run(inp)
    host = {k_: (v_.cpu().pin_memory() if v_ is not None else None) for k_, v_ in inp.items()}
    out = torch.full_like(host["q"], SENTINEL).pin_memory()
    gbla.forward_host(host["q"], host["k"], host["v"], host["gate"], host["out_gate"],
                      host["conv_w"], host["norm_w"], host["seq_lens"], out=out)
    assert torch.equal(out, y_dev.cpu())
    for b, L in enumerate([9000, 4096, 4099, 8191]):
        assert torch.equal(out[b, L:], torch.full_like(out[b, L:], SENTINEL))


def test_empty_inputs_are_noops():
    for shape in [(0, 5, 2, 64), (2, 0, 2, 64), (2, 5, 0, 64)]:
        q = torch.empty(shape, dtype=torch.bfloat16, device="cuda")
        g = torch.empty(shape[:3], dtype=torch.bfloat16, device="cuda")
        cw = torch.empty((3, shape[2], 64, 4), device="cuda")
        nw = torch.empty((shape[2], 64), device="cuda")
        gbla.forward(q, q, q, g, q, cw, nw, None, out=torch.empty_like(q))
    torch.cuda.synchronize()


def test_invalid_arguments_rejected():
    w = custom(B=1, H=2, N=64, D=64, dtype="bf16", seed=15)
    inp = make_inputs(w, "cuda")
    args = [inp[n] for n in ("q", "k", "v", "gate", "out_gate", "conv_w", "norm_w")]
    with pytest.raises(gbla.GblaError) as e:   # output aliases q
        gbla.forward(*args, None, out=inp["q"])
    assert e.value.status == gbla.GBLA_ERR_INVALID_ARG
    flat = torch.empty(inp["q"].numel() + 8, dtype=torch.bfloat16, device="cuda")
    mis = flat[1:1 + inp["q"].numel()].view_as(inp["q"])   # 2-byte offset
    with pytest.raises(gbla.GblaError) as e:
        gbla.forward(mis, *args[1:], None)
    assert e.value.status == gbla.GBLA_ERR_INVALID_ARG
    q48 = torch.zeros((1, 64, 2, 48), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(gbla.GblaError) as e:
        gbla.forward(q48, q48, q48, inp["gate"], q48, inp["conv_w"], inp["norm_w"], None)
    assert e.value.status == gbla.GBLA_ERR_UNSUPPORTED


@pytest.mark.parametrize("D", [64, 128])
def test_tensor_core_path_matches_simt_and_oracle(D):
    """The tcgen05 family against the CUDA-core family and the oracle on a
    ragged batch spanning several chunks and tiles; no bounded wait ran out."""
    lens = [1500, 129, 1, 700]
    w = custom(B=4, H=4, N=1500, D=D, dtype="bf16", seed=21, seq_lens=lens)
    inp = make_inputs(w, "cuda")
    gbla.device_error(reset=True)
    y_tc = _run(inp, gbla.ALGO_TC)
    y_simt = _run(inp, gbla.ALGO_SIMT)
    assert gbla.device_error() == 0
    ref = oracle_full(inp)
    _check_against(y_tc, ref, inp, "bf16")
    _check_against(y_simt, ref, inp, "bf16")


def test_tensor_core_state_matches_oracle():
    w = custom(B=2, H=3, N=3000, D=64, dtype="bf16", seed=22, seq_lens=[3000, 1111])
    inp = make_inputs(w, "cuda")
    st = gbla.state(inp["k"], inp["v"], inp["gate"], inp["conv_w"], inp["seq_lens"],
                    algo=gbla.ALGO_TC)
    torch.cuda.synchronize()
    assert gbla.device_error() == 0
    st = st.cpu().double().numpy()
    for b in range(2):
        for h in range(3):
            _, inter = oracle_head(inp, b, h, intermediates=True)
            S = st[b, h, :64 * 64].reshape(64, 64)
            z = st[b, h, 64 * 64:]
            assert np.abs(S - inter["S"]).max() <= 1e-2 * np.abs(inter["S"]).max()
            assert np.abs(z - inter["z"]).max() <= 1e-2 * np.abs(inter["z"]).max()


def test_many_tiles_per_cta_with_empty_sequences():
    """Enough 128-token tiles that every persistent CTA walks several of them
    across head and batch boundaries, with empty sequences in between."""
    lens = [4096, 0, 1000, 0, 0, 2500, 129]
    w = custom(B=len(lens), H=8, N=4096, D=64, dtype="bf16", seed=23, seq_lens=lens)
    inp = make_inputs(w, "cuda")
    gbla.device_error(reset=True)
    y = _run(inp, gbla.ALGO_TC)
    assert gbla.device_error() == 0
    _check_against(y, oracle_full(inp), inp, "bf16")


@pytest.mark.parametrize("flags", [1, 2, 4, 3, 5, 6, 7], ids=lambda f: f"flags{f}")
@pytest.mark.parametrize("algo,dtype", [("tc", "bf16"), ("simt", "fp32"), ("simt", "bf16")])
def test_ablation_variants(flags, algo, dtype):
    """The ablations of Table 4 (identity Conv1D, uniform key gate, no gated
    RMSNorm) and Eq. bla (all three) against the oracle with the same flags."""
    lens = [1500, 777]
    w = custom(B=2, H=4, N=1500, D=64, dtype=dtype, seed=40 + flags, seq_lens=lens)
    inp = make_inputs(w, "cuda")
    out = torch.full_like(inp["q"], SENTINEL)
    gbla.device_error(reset=True)
    gbla.forward(inp["q"], inp["k"], inp["v"], inp["gate"], inp["out_gate"], inp["conv_w"],
                 inp["norm_w"], inp["seq_lens"], out=out,
                 algo=gbla.ALGO_TC if algo == "tc" else gbla.ALGO_SIMT, flags=flags)
    torch.cuda.synchronize()
    assert gbla.device_error() == 0
    ref = oracle_full(inp, flags=flags)
    mask = valid_mask(2, 1500, np.array(lens))
    y = to64(out)
    st = (compare_prenorm if flags & gbla.FLAG_NO_NORM else compare)(y[mask], ref[mask], dtype)
    assert st["ok"], st
    assert np.all(y[~mask] == np.float64(torch.tensor(SENTINEL, dtype=out.dtype).item()))


def test_ablation_flags_rejected():
    w = custom(B=1, H=2, N=64, D=64, dtype="bf16", seed=15)
    inp = make_inputs(w, "cuda")
    with pytest.raises(gbla.GblaError) as e:
        gbla.forward(inp["q"], inp["k"], inp["v"], inp["gate"], inp["out_gate"], inp["conv_w"],
                     inp["norm_w"], None, flags=8)
    assert e.value.status == gbla.GBLA_ERR_INVALID_ARG
