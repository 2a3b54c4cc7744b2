"""Sequence split (paper_2606_07317_gb300.sequence_split) on one GPU: the
sequences cut into P contiguous segments, each segment's state and softmax
statistics from its own rows (3 conv-history rows in front, gate -inf there),
the partials combined by gbla_combine_states, each segment read out on its
own; the stitched output against the oracle on the whole sequences under the
forward's parity rule, and the combined state against the oracle's S and z.

Lengths are chosen so that segment boundaries fall inside sequences, a
sequence ends inside the next segment's history rows (no token of its own
there), and a short sequence leaves later segments empty (weight 0)."""
import numpy as np
import pytest
import torch

from paper_2606_07317_gb300 import gbla, sequence_split as ss
from paper_2606_07317_gb300.workloads import custom, make_inputs
from parity_util import compare, oracle_full, oracle_head, to64, valid_mask

pytestmark = pytest.mark.gpu


def _split_forward(inp, P):
    B, N = inp["q"].shape[:2]
    sl = inp["seq_lens"]
    parts, views = [], []
    for r in range(P):
        t0, t1 = ss.segment_bounds(N, P, r)
        loc = {n: ss.local_rows(inp[n], t0, t1)[0] for n in ("q", "k", "v", "gate", "out_gate")}
        h0 = min(ss.HALO, t0)
        ll = ss.local_lengths(sl, B, N, t0, t1, h0, inp["q"].device)
        parts.append(ss.partial_state(loc["k"], loc["v"], loc["gate"], inp["conv_w"], ll, h0))
        views.append((t0, t1, h0, loc, ll))
    states = torch.stack([p[0] for p in parts])
    stats = torch.stack([p[1] for p in parts])
    state, out_stats = ss.combine_partials(states, stats)
    o = torch.full_like(inp["q"], 7.0)
    for t0, t1, h0, loc, ll in views:
        o[:, t0:t1] = ss.local_readout(loc["q"], loc["out_gate"], inp["conv_w"], inp["norm_w"],
                                       ll, state, h0)
    torch.cuda.synchronize()
    return o, state, stats, out_stats


@pytest.mark.parametrize("dtype,D,P", [("bf16", 64, 3), ("fp32", 32, 2), ("bf16", 128, 4)])
def test_sequence_split_matches_oracle(dtype, D, P):
    N = 1500
    lens = [1500, 502, 499, 40] if P == 3 else [1500, 751, 748, 40]
    w = custom(B=len(lens), H=2, N=N, D=D, dtype=dtype, seed=51, seq_lens=lens)
    inp = make_inputs(w, "cuda")
    o, state, stats, out_stats = _split_forward(inp, P)
    mask = valid_mask(len(lens), N, np.array(lens))
    st = compare(to64(o)[mask], oracle_full(inp)[mask], dtype)
    assert st["ok"], st
    # the combined state is the whole sequences' state (the oracle's S and z)
    tol = 1e-5 if dtype == "fp32" else 1e-2
    stn = state.cpu().double().numpy()
    for b in range(len(lens)):
        for h in range(2):
            _, inter = oracle_head(inp, b, h, intermediates=True)
            S, z = stn[b, h, :D * D].reshape(D, D), stn[b, h, D * D:]
            assert np.abs(S - inter["S"]).max() <= tol * np.abs(inter["S"]).max(), (b, h)
            assert np.abs(z - inter["z"]).max() <= tol * np.abs(inter["z"]).max(), (b, h)
    # statistics: the whole sequence's max logit, and the sum of exp(logit - max)
    g = to64(inp["gate"])
    so = out_stats.cpu().double().numpy()
    for b, L in enumerate(lens):
        for h in range(2):
            a = g[b, :L, h]
            assert so[b, h, 0] == pytest.approx(a.max(), abs=0)
            assert so[b, h, 1] == pytest.approx(np.exp(a - a.max()).sum(), rel=1e-4)
    # a sequence with no token in a segment contributes weight 0 there
    t0_last = ss.segment_bounds(N, P, P - 1)[0]
    assert float(stats[P - 1, 3, 0, 1]) == 0.0 and lens[3] <= t0_last


def test_combine_states_single_part_is_identity():
    """One segment: the combination returns its state and statistics unchanged."""
    w = custom(B=2, H=2, N=300, D=64, dtype="bf16", seed=52, seq_lens=[300, 0])
    inp = make_inputs(w, "cuda")
    st, sts = gbla.state_stats(inp["k"], inp["v"], inp["gate"], inp["conv_w"], inp["seq_lens"])
    whole = gbla.state(inp["k"], inp["v"], inp["gate"], inp["conv_w"], inp["seq_lens"])
    state, out_stats = gbla.combine_states(st[None], sts[None])
    torch.cuda.synchronize()
    assert torch.equal(st, whole)
    assert torch.allclose(state, st, rtol=1e-6, atol=0)
    assert torch.equal(out_stats[:, :, 0], sts[:, :, 0])
    assert torch.all(state[1] == 0) and float(out_stats[1, 0, 1]) == 0.0


def test_combine_states_rejects_bad_arguments():
    s = torch.zeros((2, 1, 1, 64 * 64 + 64), device="cuda")
    t = torch.zeros((2, 1, 1, 2), device="cuda")
    out = torch.zeros((1, 1, 64 * 64 + 64), device="cuda")
    outs = torch.zeros((1, 1, 2), device="cuda")
    lib = gbla.load()
    assert lib.gbla_combine_states(s.data_ptr(), t.data_ptr(), 0, out.data_ptr(),
                                   outs.data_ptr(), 1, 1, 64, None) == gbla.GBLA_ERR_INVALID_ARG
    assert lib.gbla_combine_states(s.data_ptr(), t.data_ptr(), 2, out.data_ptr(),
                                   outs.data_ptr(), 1, 1, 48, None) == gbla.GBLA_ERR_UNSUPPORTED
    assert lib.gbla_combine_states(s.data_ptr(), t.data_ptr(), 2, s.data_ptr(),
                                   outs.data_ptr(), 1, 1, 64, None) == gbla.GBLA_ERR_INVALID_ARG
