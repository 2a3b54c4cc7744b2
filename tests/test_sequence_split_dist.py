"""The exchange of the sequence split on CPU: world size 2 over gloo.

Each rank holds one contiguous token segment of the sequences (3 conv-history
rows in front, their gate logits -inf).  Its partial state (S, z of the
segment, from the oracle) and softmax statistics (max logit, sum of exp) go
through sequence_split.gather_partials; every rank must receive all of them
in rank order, and combining them (the max-rescaled sum, written out here in
numpy) must give the oracle's state of the whole sequences.  The combination
itself runs on the GPU in the product (gbla_combine_states) and is tested in
test_sequence_split_gpu.py."""
import os
import socket

import numpy as np
import torch
import torch.multiprocessing as mp

WS = 2
B, H, N, D, W = 2, 2, 40, 4, 4
LENS = [40, 23]


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _inputs():
    rng = np.random.default_rng(3)
    x = {n: rng.standard_normal((B, N, H, D)) for n in ("q", "k", "v", "og")}
    x["a"] = rng.standard_normal((B, N, H))
    x["w"] = 0.5 * rng.standard_normal((3, H, D, W))
    x["nw"] = 1.0 + 0.02 * rng.standard_normal((H, D))
    return x


def _head(x, b, h, lo, hi, h0):
    """Oracle S, z and statistics of rows [lo, hi) of (b, h); the first h0 rows are
    conv history only (logit -inf)."""
    import oracle
    a = x["a"][b, lo:hi, h].copy()
    a[:h0] = -np.inf
    _, inter = oracle.gbla_head(x["q"][b, lo:hi, h], x["k"][b, lo:hi, h], x["v"][b, lo:hi, h],
                                a, x["og"][b, lo:hi, h], x["w"][0, h], x["w"][1, h],
                                x["w"][2, h], x["nw"][h], intermediates=True)
    m = a.max()
    return np.concatenate([inter["S"].ravel(), inter["z"]]), (m, np.exp(a - m).sum())


def _worker(rank, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(WS))
    import torch.distributed as dist
    from paper_2606_07317_gb300 import sequence_split as ss
    dist.init_process_group("gloo", rank=rank, world_size=WS)
    x = _inputs()
    t0, t1 = ss.segment_bounds(N, WS, rank)
    h0 = min(ss.HALO, t0)
    F = D * D + D
    state = torch.zeros((B, H, F), dtype=torch.float64)
    stats = torch.zeros((B, H, 2), dtype=torch.float64)
    stats[:, :, 0] = -np.inf
    for b in range(B):
        hi = min(LENS[b], t1)
        if LENS[b] <= t0:
            continue  # no token of this sequence in the segment: weight 0
        for h in range(H):
            s, (m, l) = _head(x, b, h, t0 - h0, hi, h0)
            state[b, h] = torch.from_numpy(s)
            stats[b, h, 0], stats[b, h, 1] = m, l
    states, statss = ss.gather_partials(state, stats)
    dist.destroy_process_group()
    np.savez(os.path.join(out, f"r{rank}.npz"), states=states.numpy(), stats=statss.numpy(),
             own=state.numpy())


def test_gather_partials_and_combination(tmp_path):
    import oracle
    oracle.load()  # build the C oracle once, before the ranks start
    mp.start_processes(_worker, args=(_free_port(), str(tmp_path)), nprocs=WS,
                       start_method="spawn")
    res = [np.load(tmp_path / f"r{r}.npz") for r in range(WS)]
    # every rank holds every rank's partial, in rank order
    for r in range(WS):
        assert np.array_equal(res[r]["states"], res[0]["states"])
        assert np.array_equal(res[r]["stats"], res[0]["stats"])
        assert np.array_equal(res[0]["states"][r], res[r]["own"])
    states, stats = res[0]["states"], res[0]["stats"]
    m, l = stats[..., 0], stats[..., 1]
    M = np.max(np.where(l > 0, m, -np.inf), axis=0)
    wgt = np.where(l > 0, l * np.exp(m - M), 0.0)
    comb = (wgt[..., None] * states).sum(0) / wgt.sum(0)[..., None]
    x = _inputs()
    for b in range(B):
        for h in range(H):
            s_ref, _ = _head(x, b, h, 0, LENS[b], 0)
            assert np.allclose(comb[b, h], s_ref, rtol=1e-12, atol=1e-14), (b, h)
