"""Sequence split of the GBLA core across devices (context parallelism).

The state of Sec. 2.1 item 2 is a softmax-weighted sum over a whole sequence,
so a sequence cut into contiguous token segments, one per rank, needs one
exchange: every rank computes the normalised state of its own segment together
with that segment's softmax statistics (gbla_state_stats), the ranks gather
all of them, and each combines them into the sequence's state
(gbla_combine_states: the same max-rescaled combination the state reduction
applies to its partial records, in rank order, so every rank gets the same
result).  Each rank then reads out its own tokens (gbla_readout).

The Conv1D is causal with width 4, so a segment starting at t0 > 0 also needs
the 3 rows before t0 as conv history: the local tensors carry h0 = min(3, t0)
history rows in front.  Those rows are conv input only; their gate logits are
replaced by -inf on a copy, which gives them weight 0 in the state, and their
readout rows are dropped.

This module does argument plumbing only: the slicing of a rank's rows, the
local lengths and the gather; every step of the method runs in the library's
kernels.  The headline path runs on one GPU and never calls it.
"""
from __future__ import annotations

import torch
import torch.distributed as dist

from . import gbla

HALO = gbla.CONV_WIDTH - 1  # conv history rows a segment needs in front


def segment_bounds(N: int, world: int, rank: int) -> tuple[int, int]:
    """Token range [t0, t1) of `rank`'s segment of an N-token padded sequence."""
    return N * rank // world, N * (rank + 1) // world


def local_rows(x: torch.Tensor, t0: int, t1: int) -> tuple[torch.Tensor, int]:
    """Rows [t0 - h0, t1) of a token-major [B, N, ...] tensor (h0 = min(3, t0) rows
    of conv history in front), as a contiguous copy; returns (rows, h0)."""
    h0 = min(HALO, t0)
    return x[:, t0 - h0:t1].contiguous(), h0


def local_lengths(seq_lens, B: int, N: int, t0: int, t1: int, h0: int,
                  device) -> torch.Tensor:
    """Valid local rows of each batch row's segment: its history rows and tokens up
    to min(L_b, t1); 0 when the sequence ends at or before t0 (no token of its own)."""
    if seq_lens is None:
        L = torch.full((B,), N, dtype=torch.int64, device=device)
    else:
        L = seq_lens.to(device=device, dtype=torch.int64)
    local = torch.where(L > t0, torch.clamp(L, max=t1) - (t0 - h0), torch.zeros_like(L))
    return local.to(torch.int32)


def partial_state(k_loc, v_loc, gate_loc, conv_w, local_lens, h0: int):
    """State and softmax statistics of one segment from its local rows (h0 history
    rows in front, whose gate logits are set to -inf on a copy)."""
    if h0:
        gate_loc = gate_loc.clone()
        gate_loc[:, :h0] = float("-inf")
    return gbla.state_stats(k_loc, v_loc, gate_loc, conv_w, local_lens)


def gather_partials(state: torch.Tensor, stats: torch.Tensor, group=None):
    """Every rank's (state, stats), stacked in rank order on every rank."""
    world = dist.get_world_size(group)
    states = [torch.empty_like(state) for _ in range(world)]
    statss = [torch.empty_like(stats) for _ in range(world)]
    dist.all_gather(states, state.contiguous(), group=group)
    dist.all_gather(statss, stats.contiguous(), group=group)
    return torch.stack(states), torch.stack(statss)


def combine_partials(states: torch.Tensor, stats: torch.Tensor):
    """(state, stats) of the whole sequences from the stacked segment partials."""
    return gbla.combine_states(states, stats)


def local_readout(q_loc, og_loc, conv_w, norm_w, local_lens, state, h0: int):
    """o of the segment's own tokens (the history rows' outputs are dropped); rows
    past the local lengths are left as allocated."""
    o = gbla.readout(q_loc, og_loc, conv_w, norm_w, state, local_lens)
    return o[:, h0:]


def forward(q, k, v, gate, out_gate, conv_w, norm_w, seq_lens, t0: int, t1: int, N: int,
            group=None):
    """One rank's part of the sequence-split forward.  q, k, v, gate, out_gate are the
    rank's local rows (rows [t0 - h0, t1) of the padded sequences, h0 = min(3, t0));
    seq_lens the global lengths.  Returns o of tokens [t0, t1)."""
    B = q.shape[0]
    h0 = min(HALO, t0)
    ll = local_lengths(seq_lens, B, N, t0, t1, h0, q.device)
    st, ss = partial_state(k, v, gate, conv_w, ll, h0)
    state, _ = combine_partials(*gather_partials(st, ss, group))
    return local_readout(q, out_gate, conv_w, norm_w, ll, state, h0)
