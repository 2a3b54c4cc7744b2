"""Bidirectional softmax attention (Sec. 2), the SA layer of the hybrid encoder,
on tensor cores through the C ABI, against the fp64 oracle on the same seeded
inputs.

Tolerance.  The kernel multiplies bf16 inputs exactly, accumulates in fp32
and rounds the probabilities p_j to bf16 (relative error at most 2^-9 each)
before the second product, so |o - o_ref| <= 2^-9 sum_j p_j |v_j| / sum_j p_j
plus fp32 accumulation and the rounding of the stored bf16 output (half an
ulp of o_ref).  The test allows twice the probability term:
    |o - o_ref| <= 2^-8 A + ulp_bf16(o_ref) / 2 + 1e-6,   A = sum_j p_j |v_j| / sum_j p_j
(A from the oracle), and a normwise error of at most 2^-7.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_07317_gb300 import gbla
from parity_util import log_stats, to64, ulp_bf16

pytestmark = pytest.mark.gpu

SENTINEL = -777.0
SENTINEL_BF16 = float(torch.tensor(SENTINEL, dtype=torch.bfloat16).item())  # -776


def _inputs(B, N, H, D=64, seed=0, lens=None, device="cuda"):
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    q, k, v = (torch.randn((B, N, H, D), generator=g, device=device).to(torch.bfloat16)
               for _ in range(3))
    sl = torch.tensor(lens, dtype=torch.int32, device=device) if lens is not None else None
    return q, k, v, sl


def _check(y, ref, a, mask=None):
    d = np.abs(y - ref)
    bound = 2.0 ** -8 * a + 0.5 * ulp_bf16(ref) + 1e-6
    st = {"max_abs": float(d.max()), "worst_excess": float((d - bound).max()),
          "normwise": float(np.linalg.norm(d) / max(np.linalg.norm(ref), 1e-300)),
          "max_ref": float(np.abs(ref).max())}
    assert np.all(np.isfinite(y)), st
    assert st["worst_excess"] <= 0.0, st
    assert st["normwise"] <= 2.0 ** -7, st
    return st


def _run(q, k, v, sl):
    out = torch.full_like(q, SENTINEL)
    gbla.device_error(reset=True)
    gbla.attention(q, k, v, sl, out=out)
    torch.cuda.synchronize()
    assert gbla.device_error() == 0
    return out


@pytest.fixture(scope="module", autouse=True)
def _lib():
    gbla.load()


@pytest.mark.parametrize("B,N,H,lens,seed", [
    (2, 333, 3, [333, 200], 1),        # several query tiles and key blocks, ragged tails
    (1, 1000, 2, None, 2),
    (3, 300, 2, [1, 127, 129], 3),     # lengths around one block
    (1, 256, 1, [128], 4),             # exactly one block
])
def test_attention_matches_oracle(B, N, H, lens, seed):
    q, k, v, sl = _inputs(B, N, H, seed=seed, lens=lens)
    if lens is not None:  # the padding holds NaN, which must not reach valid rows
        for b, L in enumerate(lens):
            for t_ in (q, k, v):
                t_[b, L:] = float("nan")
    y = _run(q, k, v, sl)
    ref, a = oracle.softmax_attention(to64(q), to64(k), to64(v),
                                      None if sl is None else sl.cpu().numpy(), absout=True,
                                      n_threads=8)
    yy = to64(y)
    Ls = lens if lens is not None else [N] * B
    for b, L in enumerate(Ls):
        st = _check(yy[b, :L], ref[b, :L], a[b, :L])
        assert np.all(yy[b, L:] == SENTINEL_BF16), "rows past the sequence end were written"
    log_stats({"test": "attention", "shape": [B, N, H], **st})


def test_attention_empty_sequence_and_sizes():
    q, k, v, sl = _inputs(2, 200, 2, seed=5, lens=[0, 200])
    y = _run(q, k, v, sl)
    assert torch.all(y[0] == SENTINEL_BF16)
    for shape in [(0, 5, 2, 64), (2, 0, 2, 64), (2, 5, 0, 64)]:
        z = torch.empty(shape, dtype=torch.bfloat16, device="cuda")
        gbla.attention(z, z, z, None, out=torch.empty_like(z))


def test_attention_table5_shape_sampled_rows():
    """Table 5's batch and head count (batch 8, 16 heads of 64) at L = 2048: every
    (batch, head), 24 query rows each spread over all query tiles, against the
    oracle row by row."""
    B, N, H = 8, 2048, 16
    q, k, v, _ = _inputs(B, N, H, seed=6)
    y = _run(q, k, v, None)
    rows = np.linspace(0, N - 1, 24).astype(int)
    qc, kc, vc, yc = (to64(t) for t in (q, k, v, y))
    worst = None
    for b in range(B):
        for h in range(H):
            ref, a = oracle.softmax_attention_rows(qc[b, rows, h], kc[b, :, h], vc[b, :, h])
            st = _check(yc[b, rows, h], ref, a)
            if worst is None or st["worst_excess"] > worst["worst_excess"]:
                worst = st
    log_stats({"test": "attention_sampled", "shape": [B, N, H], **worst})


def test_attention_table5_longest_sampled_rows():
    """Table 5's longest length (batch 8, 16 heads of 64, L = 32768: 256 query
    tiles and 256 key blocks per (b, h)), 6 query rows per (batch, head) spread
    over the sequence, against the oracle row by row over all 32768 keys."""
    B, N, H = 8, 32768, 16
    q, k, v, _ = _inputs(B, N, H, seed=9)
    y = _run(q, k, v, None)
    rows = np.array([0, 127, 128, 16383, 30001, N - 1])
    worst = None
    for b in range(B):
        kc, vc = to64(k[b]), to64(v[b])
        qc, yc = to64(q[b, rows]), to64(y[b, rows])
        for h in range(H):
            ref, a = oracle.softmax_attention_rows(qc[:, h], kc[:, h], vc[:, h])
            st = _check(yc[:, h], ref, a)
            if worst is None or st["worst_excess"] > worst["worst_excess"]:
                worst = st
    log_stats({"test": "attention_sampled_32768", "shape": [B, N, H], **worst})


def test_attention_dominant_scores_are_stable():
    """Scores far above the rest (row maxima growing block after block) are
    handled by the running maximum: the output is the dominant key's value."""
    B, N, H = 1, 640, 1
    q, k, v, _ = _inputs(B, N, H, seed=7)
    kk = k.clone()
    # key 513 (fifth block) dominates query rows 0..3 by a wide margin
    kk[0, 513, 0] = (q[0, 0, 0].float() * 3.0).to(torch.bfloat16)
    y = _run(q, kk, v, None)
    ref, a = oracle.softmax_attention(to64(q), to64(kk), to64(v), absout=True, n_threads=8)
    _check(to64(y)[0], ref[0], a[0])


def test_attention_deterministic_and_rejects():
    q, k, v, sl = _inputs(2, 300, 2, seed=8, lens=[300, 150])
    assert torch.equal(_run(q, k, v, sl), _run(q, k, v, sl))
    with pytest.raises(gbla.GblaError) as e:  # output aliases q
        gbla.attention(q, k, v, sl, out=q)
    assert e.value.status == gbla.GBLA_ERR_INVALID_ARG
    q128 = torch.zeros((1, 64, 2, 128), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(gbla.GblaError) as e:  # D = 128 is not covered
        gbla.attention(q128, q128, q128)
    assert e.value.status == gbla.GBLA_ERR_UNSUPPORTED
