"""The sequence split's host-side arithmetic on CPU: the segments partition the
padded length, each segment carries min(3, t0) rows of Conv1D history in front,
and the local lengths count the history rows and the segment's own valid tokens
(0 when the sequence ends at or before the segment's start)."""
import torch

from paper_2606_07317_gb300 import sequence_split as ss


def test_segments_partition_the_length():
    for N in (1, 3, 7, 64, 1000, 32768):
        for world in (1, 2, 3, 4, 8):
            bounds = [ss.segment_bounds(N, world, r) for r in range(world)]
            assert bounds[0][0] == 0 and bounds[-1][1] == N
            for (a0, a1), (b0, b1) in zip(bounds, bounds[1:]):
                assert a1 == b0 and a0 <= a1
            sizes = [t1 - t0 for t0, t1 in bounds]
            assert max(sizes) - min(sizes) <= 1


def test_local_rows_carry_the_conv_history():
    x = torch.arange(2 * 20).reshape(2, 20)
    for t0, t1 in [(0, 5), (2, 9), (3, 10), (11, 20)]:
        rows, h0 = ss.local_rows(x, t0, t1)
        assert h0 == min(ss.HALO, t0)
        assert torch.equal(rows, x[:, t0 - h0:t1]) and rows.is_contiguous()


def test_local_lengths():
    N, t0, t1 = 100, 40, 70
    h0 = min(ss.HALO, t0)
    lens = torch.tensor([10, 40, 41, 55, 70, 99, 100], dtype=torch.int32)
    got = ss.local_lengths(lens, len(lens), N, t0, t1, h0, "cpu").tolist()
    # ends before or at t0: nothing; inside: history + own tokens; past t1: the whole segment
    assert got == [0, 0, 1 + h0, 15 + h0, 30 + h0, 30 + h0, 30 + h0]
    assert ss.local_lengths(None, 3, N, t0, t1, h0, "cpu").tolist() == [30 + h0] * 3
    # the first segment has no history
    assert ss.local_lengths(lens, len(lens), N, 0, 40, 0, "cpu").tolist() == [10, 40, 40, 40,
                                                                               40, 40, 40]
