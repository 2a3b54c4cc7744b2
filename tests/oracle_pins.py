"""Checks that pin the fp64 oracle to something other than itself.

Each check takes the loaded oracle library (so the same checks can be run
against deliberately broken copies of the oracle) and raises AssertionError
when the oracle disagrees with the paper or the mathematics.  The sources of
truth are library routines (scipy, torch), closed forms, the quadratic form of
Sec. 2.1 item 2 and invariants the equations imply.
"""
from __future__ import annotations

import math

import numpy as np
import scipy.signal
import scipy.special
import torch

import oracle

W = oracle.CONV_W


def _rng(seed):
    return np.random.default_rng(seed)


def _head_inputs(rng, L, D, Wd=W):
    q, k, v, og = (rng.standard_normal((L, D)) for _ in range(4))
    a = rng.standard_normal(L)
    wq, wk, wv = (0.5 * rng.standard_normal((D, Wd)) for _ in range(3))
    nw = 1.0 + 0.02 * rng.standard_normal(D)
    return q, k, v, a, og, wq, wk, wv, nw


# --- element functions -------------------------------------------------------

def pin_phi_closed_form(lib):
    """phi = elu + 1 (Sec. 2): x+1 for x>0, e^x for x<=0; continuous, positive."""
    for x, want in [(0.0, 1.0), (1.0, 2.0), (2.5, 3.5), (-1.0, math.exp(-1.0)),
                    (-3.0, math.exp(-3.0)), (1e-9, 1.0 + 1e-9), (-40.0, math.exp(-40.0))]:
        got = oracle.phi(x, lib)
        assert abs(got - want) <= 1e-15 * max(1.0, abs(want)), (x, got, want)
    xs = np.linspace(-30, 30, 601)
    ys = np.array([oracle.phi(x, lib) for x in xs])
    assert np.all(ys > 0)
    # elu+1 by torch's library elu; elu(x)+1 cancels for very negative x, so the
    # comparison is absolute there
    ref = torch.nn.functional.elu(torch.tensor(xs, dtype=torch.float64)).numpy() + 1.0
    np.testing.assert_allclose(ys, ref, rtol=1e-14, atol=1e-15)


def pin_silu_library(lib):
    """SiLU(x) = x * sigmoid(x) (gated RMSNorm, Sec. 2.1 item 3) vs torch and scipy."""
    xs = np.linspace(-20, 20, 401)
    got = np.array([oracle.silu(x, lib) for x in xs])
    ref_t = torch.nn.functional.silu(torch.tensor(xs, dtype=torch.float64)).numpy()
    ref_s = xs * scipy.special.expit(xs)
    np.testing.assert_allclose(got, ref_t, rtol=1e-13, atol=1e-300)
    np.testing.assert_allclose(got, ref_s, rtol=1e-13, atol=1e-300)


def pin_conv1d_library(lib):
    """Causal depthwise Conv1D (Sec. 2.1 item 1) equals a causal FIR filter
    (scipy lfilter with reversed taps) and torch's conv1d with W-1 left zeros."""
    rng = _rng(11)
    L, C = 37, 6
    x = rng.standard_normal((L, C))
    w = rng.standard_normal((C, W))
    y = oracle.conv1d(x, w, lib)
    for c in range(C):
        ref = scipy.signal.lfilter(w[c, ::-1], [1.0], x[:, c])
        np.testing.assert_allclose(y[:, c], ref, rtol=1e-12, atol=1e-12)
    xt = torch.tensor(x.T[None], dtype=torch.float64)          # [1, C, L]
    xt = torch.nn.functional.pad(xt, (W - 1, 0))
    ref = torch.nn.functional.conv1d(xt, torch.tensor(w[:, None, :]), groups=C)[0].T.numpy()
    np.testing.assert_allclose(y, ref, rtol=1e-12, atol=1e-12)


def pin_conv1d_impulse(lib):
    """An impulse at position s reaches only s..s+W-1 (causal), tap W-1 first."""
    L, C, s = 12, 3, 5
    rng = _rng(12)
    w = rng.standard_normal((C, W))
    x = np.zeros((L, C)); x[s, :] = 1.0
    y = oracle.conv1d(x, w, lib)
    for t in range(L):
        for c in range(C):
            want = w[c, W - 1 - (t - s)] if 0 <= t - s < W else 0.0
            assert y[t, c] == want, (t, c, y[t, c], want)


def pin_softmax_library(lib):
    """Key gate g = softmax over the sequence (Sec. 2.1 item 2) vs scipy; stable
    for logits near the exp overflow limit."""
    rng = _rng(13)
    for L in (1, 2, 7, 100):
        a = 3.0 * rng.standard_normal(L)
        np.testing.assert_allclose(oracle.softmax(a, lib), scipy.special.softmax(a),
                                   rtol=1e-13, atol=1e-300)
    a = np.array([1000.0, 999.0, 1001.0, -5.0])
    g = oracle.softmax(a, lib)
    assert np.all(np.isfinite(g))
    np.testing.assert_allclose(g, scipy.special.softmax(a), rtol=1e-13, atol=1e-300)
    assert abs(g.sum() - 1.0) < 1e-15


def pin_rmsnorm_library(lib):
    """Gated RMSNorm (Sec. 2.1 item 3) equals torch's rms_norm times SiLU(og)."""
    rng = _rng(14)
    for D in (1, 5, 64):
        O = rng.standard_normal(D) * 0.01
        og = rng.standard_normal(D)
        w = 1.0 + 0.1 * rng.standard_normal(D)
        y = oracle.gated_rmsnorm_row(O, og, w, 1e-6, lib)
        Ot = torch.tensor(O[None])
        ref = (torch.nn.functional.rms_norm(Ot, (D,), torch.tensor(w), eps=1e-6)[0]
               * torch.nn.functional.silu(torch.tensor(og))).numpy()
        np.testing.assert_allclose(y, ref, rtol=1e-12, atol=1e-15)


def pin_rmsnorm_closed_form(lib):
    """rms(y / (w * SiLU(og))) = sqrt(ms / (ms + eps)) with ms = mean O^2."""
    rng = _rng(15)
    D, eps = 16, 1e-3
    O = 0.05 * rng.standard_normal(D)
    og = np.abs(rng.standard_normal(D)) + 0.1
    w = 1.0 + 0.1 * rng.standard_normal(D)
    y = oracle.gated_rmsnorm_row(O, og, w, eps, lib)
    u = y / (w * og * scipy.special.expit(og))
    ms = np.mean(O ** 2)
    assert abs(np.sqrt(np.mean(u ** 2)) - np.sqrt(ms / (ms + eps))) < 1e-13
    np.testing.assert_allclose(u / O, 1.0 / np.sqrt(ms + eps) * np.ones(D), rtol=1e-12)


# --- the layer ---------------------------------------------------------------

def pin_linear_equals_quadratic(lib):
    """The linear-time matrix form equals the explicit L x L form (Sec. 2.1
    item 2: both displayed equations), for every ablation setting."""
    for seed, L, D in [(21, 13, 5), (22, 1, 3), (23, 40, 8)]:
        args = _head_inputs(_rng(seed), L, D)
        for f in range(8):
            y1 = oracle.gbla_head(*args, flags=f, lib=lib)
            y2, _ = oracle.gbla_head_quadratic(*args, flags=f, lib=lib)
            np.testing.assert_allclose(y1, y2, rtol=1e-11, atol=1e-13)


def pin_bla_textbook(lib):
    """With conv, gate and norm switched off GBLA is Eq. bla; O is also a
    convex combination of the v rows (weights phi(q)^T phi(k_j), normalised)."""
    rng = _rng(31)
    L, D = 9, 4
    q, k, v, a, og, wq, wk, wv, nw = _head_inputs(rng, L, D)
    y = oracle.gbla_head(q, k, v, a, og, wq, wk, wv, nw, flags=oracle.BLA, lib=lib)
    pq = np.where(q > 0, q + 1, np.exp(np.minimum(q, 0)))
    pk = np.where(k > 0, k + 1, np.exp(np.minimum(k, 0)))
    sim = pq @ pk.T                        # L x L similarities
    P = sim / sim.sum(axis=1, keepdims=True)
    np.testing.assert_allclose(y, P @ v, rtol=1e-12, atol=1e-14)
    # "W/o key gating" is the uniform gate softmax(0) = 1/L; z is then the mean
    # of phi(k_j) over the sequence
    _, inter = oracle.gbla_head(q, k, v, a, og, wq, wk, wv, nw, flags=oracle.BLA,
                                intermediates=True, lib=lib)
    np.testing.assert_allclose(inter["g"], np.full(L, 1.0 / L), rtol=1e-15)
    np.testing.assert_allclose(inter["z"], pk.mean(axis=0), rtol=1e-13)


def pin_hand_worked_d1(lib):
    """D=1, L=2, no conv: q cancels and O = sum g phi(k) v / sum g phi(k).
    a = (0, ln 3) gives g = (1/4, 3/4); k = (0, 1) gives phi = (1, 2);
    v = (2, -1) gives O = (1/2 - 3/2) / (1/4 + 3/2) = -4/7 for both rows."""
    one = np.ones((1, W))
    q = np.array([[0.3], [-2.0]]); k = np.array([[0.0], [1.0]])
    v = np.array([[2.0], [-1.0]]); og = np.array([[1.0], [-0.5]])
    a = np.array([0.0, math.log(3.0)])
    nw = np.array([1.5])
    _, inter = oracle.gbla_head(q, k, v, a, og, one, one, one, nw,
                                flags=oracle.NO_CONV | oracle.NO_NORM,
                                intermediates=True, lib=lib)
    np.testing.assert_allclose(inter["g"], [0.25, 0.75], rtol=1e-15)
    np.testing.assert_allclose(inter["z"], [0.25 + 1.5], rtol=1e-15)
    np.testing.assert_allclose(inter["S"], [[0.5 - 1.5]], rtol=1e-15)
    np.testing.assert_allclose(inter["O"][:, 0], [-4 / 7, -4 / 7], rtol=1e-14)
    # Gated RMSNorm with D=1: y = O / sqrt(O^2 + eps) * w * silu(og)
    eps = 1e-6
    y = oracle.gbla_head(q, k, v, a, og, one, one, one, nw, eps=eps,
                         flags=oracle.NO_CONV, lib=lib)
    O = -4 / 7
    for i, g_in in enumerate([1.0, -0.5]):
        want = O / math.sqrt(O * O + eps) * 1.5 * g_in / (1 + math.exp(-g_in))
        assert abs(y[i, 0] - want) < 1e-14, (y[i, 0], want)


def pin_constant_values(lib):
    """If every v~ row is the same vector c, every O row equals c (O is a
    weighted mean of the v~ rows).  Identity taps on v keep v~ = v."""
    rng = _rng(41)
    L, D = 50, 6
    q, k, v, a, og, wq, wk, wv, nw = _head_inputs(rng, L, D)
    c = rng.standard_normal(D)
    v = np.tile(c, (L, 1))
    wv = np.zeros((D, W)); wv[:, W - 1] = 1.0
    _, inter = oracle.gbla_head(q, k, v, a, og, wq, wk, wv, nw, intermediates=True, lib=lib)
    np.testing.assert_allclose(inter["O"], np.tile(c, (L, 1)), rtol=1e-12, atol=1e-14)


def pin_state_ones(lib):
    """With v~ = 1 the state rows equal the normaliser: S[d, e] = z[d] (both are
    K^T applied to V and to 1)."""
    rng = _rng(42)
    L, D = 30, 5
    q, k, v, a, og, wq, wk, wv, nw = _head_inputs(rng, L, D)
    v = np.ones((L, D))
    wv = np.zeros((D, W)); wv[:, W - 1] = 1.0
    _, inter = oracle.gbla_head(q, k, v, a, og, wq, wk, wv, nw, intermediates=True, lib=lib)
    np.testing.assert_allclose(inter["S"], np.tile(inter["z"][:, None], (1, D)), rtol=1e-13)
    assert np.all(inter["z"] > 0)
    assert abs(inter["g"].sum() - 1.0) < 1e-14


def pin_single_token(lib):
    """L = 1: the softmax gate is 1, O = v~_0 = w_v[:, W-1] * v_0 (only the last
    tap sees a real token), and the key side cancels."""
    rng = _rng(43)
    D = 7
    q, k, v, a, og, wq, wk, wv, nw = _head_inputs(rng, 1, D)
    _, inter = oracle.gbla_head(q, k, v, a, og, wq, wk, wv, nw, intermediates=True, lib=lib)
    np.testing.assert_allclose(inter["O"][0], wv[:, W - 1] * v[0], rtol=1e-13)
    np.testing.assert_allclose(inter["g"], [1.0], rtol=0, atol=0)


def pin_permutation_equivariance(lib):
    """Without the Conv1D the bidirectional core has no notion of order:
    permuting positions permutes the outputs."""
    rng = _rng(51)
    L, D = 23, 4
    q, k, v, a, og, wq, wk, wv, nw = _head_inputs(rng, L, D)
    p = rng.permutation(L)
    y = oracle.gbla_head(q, k, v, a, og, wq, wk, wv, nw, flags=oracle.NO_CONV, lib=lib)
    yp = oracle.gbla_head(q[p], k[p], v[p], a[p], og[p], wq, wk, wv, nw,
                          flags=oracle.NO_CONV, lib=lib)
    np.testing.assert_allclose(yp, y[p], rtol=1e-12, atol=1e-14)


def pin_gate_shift_invariance(lib):
    """softmax(a + c) = softmax(a): a shift of all gate logits changes nothing."""
    rng = _rng(52)
    L, D = 31, 4
    q, k, v, a, og, wq, wk, wv, nw = _head_inputs(rng, L, D)
    y = oracle.gbla_head(q, k, v, a, og, wq, wk, wv, nw, lib=lib)
    y2 = oracle.gbla_head(q, k, v, a + 7.25, og, wq, wk, wv, nw, lib=lib)
    np.testing.assert_allclose(y2, y, rtol=1e-12, atol=1e-14)


def pin_gate_weights_keys(lib):
    """A dominant gate logit makes that key the only one: O_i -> v~_j for all i."""
    rng = _rng(53)
    L, D, j = 17, 4, 6
    q, k, v, a, og, wq, wk, wv, nw = _head_inputs(rng, L, D)
    a = np.zeros(L); a[j] = 60.0
    _, inter = oracle.gbla_head(q, k, v, a, og, wq, wk, wv, nw, intermediates=True, lib=lib)
    np.testing.assert_allclose(inter["O"], np.tile(inter["vt"][j], (L, 1)), rtol=1e-12, atol=1e-12)


def _layer_inputs(rng, B, N, H, D):
    q, k, v, og = (rng.standard_normal((B, N, H, D)) for _ in range(4))
    gate = rng.standard_normal((B, N, H))
    conv_w = 0.5 * rng.standard_normal((3, H, D, W))
    norm_w = 1.0 + 0.02 * rng.standard_normal((H, D))
    return q, k, v, gate, og, conv_w, norm_w


def pin_layer_indexing(lib):
    """The multi-head driver equals the single-head routine applied to each
    (batch, head) slice with that head's own taps and norm weight (Sec. 2.1,
    multi-head paragraph); threads do not change a bit."""
    rng = _rng(61)
    B, N, H, D = 2, 19, 3, 4
    q, k, v, gate, og, conv_w, norm_w = _layer_inputs(rng, B, N, H, D)
    sl = np.array([19, 11], np.int32)
    y1 = oracle.gbla_forward(q, k, v, gate, og, conv_w, norm_w, sl, n_threads=1, lib=lib)
    y4 = oracle.gbla_forward(q, k, v, gate, og, conv_w, norm_w, sl, n_threads=4, lib=lib)
    assert np.array_equal(np.isnan(y1), np.isnan(y4))
    assert np.array_equal(y1[~np.isnan(y1)], y4[~np.isnan(y4)])
    for b in range(B):
        Lb = sl[b]
        assert np.all(np.isnan(y1[b, Lb:]))
        for h in range(H):
            ref = oracle.gbla_head(q[b, :Lb, h], k[b, :Lb, h], v[b, :Lb, h], gate[b, :Lb, h],
                                   og[b, :Lb, h], conv_w[0, h], conv_w[1, h], conv_w[2, h],
                                   norm_w[h], lib=lib)
            np.testing.assert_array_equal(y1[b, :Lb, h], ref)


def pin_padding_ignored(lib):
    """Rows at t >= L_b (right padding) contribute nothing, whatever they hold:
    a padded run equals the unpadded run on the valid rows."""
    rng = _rng(62)
    B, N, H, D = 2, 24, 2, 4
    q, k, v, gate, og, conv_w, norm_w = _layer_inputs(rng, B, N, H, D)
    sl = np.array([24, 9], np.int32)
    y = oracle.gbla_forward(q, k, v, gate, og, conv_w, norm_w, sl, lib=lib)
    for t in (q, k, v, og):
        t[1, 9:] = np.nan
    gate[1, 9:] = 1e30
    y2 = oracle.gbla_forward(q, k, v, gate, og, conv_w, norm_w, sl, lib=lib)
    np.testing.assert_array_equal(y2[1, :9], y[1, :9])
    cut = [x[1:2, :9] for x in (q, k, v, gate, og)]
    y3 = oracle.gbla_forward(*cut, conv_w, norm_w, None, lib=lib)
    np.testing.assert_array_equal(y3[0], y[1, :9])


def pin_heads_independent(lib):
    """Permuting heads together with their taps and norm weights permutes the
    outputs (heads share nothing)."""
    rng = _rng(63)
    B, N, H, D = 1, 15, 4, 3
    q, k, v, gate, og, conv_w, norm_w = _layer_inputs(rng, B, N, H, D)
    p = np.array([2, 0, 3, 1])
    y = oracle.gbla_forward(q, k, v, gate, og, conv_w, norm_w, lib=lib)
    yp = oracle.gbla_forward(q[:, :, p], k[:, :, p], v[:, :, p], gate[:, :, p], og[:, :, p],
                             conv_w[:, p], norm_w[p], lib=lib)
    np.testing.assert_array_equal(yp, y[:, :, p])


def pin_denominator_positive(lib):
    """phi > 0 and g > 0, so z > 0 and every readout denominator is positive."""
    rng = _rng(64)
    L, D = 40, 6
    q, k, v, a, og, wq, wk, wv, nw = _head_inputs(rng, L, D)
    q *= 30; k *= 30
    _, inter = oracle.gbla_head(q, k, v, a, og, wq, wk, wv, nw, intermediates=True, lib=lib)
    assert np.all(inter["z"] > 0)
    assert np.all(np.isfinite(inter["O"]))


# --- layer front end: X-space Conv1D and stacked projections (Sec. 2.1) ----

def _project_inputs(rng, B, N, d, H, D):
    x = rng.standard_normal((B, N, d))
    conv_x = 0.5 * rng.standard_normal((d, W))
    w = rng.standard_normal((4 * H * D + H, d)) / np.sqrt(d)
    return x, conv_x, w


def _np_conv_x(x, conv_x):
    """Causal depthwise Conv1D of every channel through numpy's convolution:
    y[t] = sum_i w[i] x[t - (W-1) + i] is the full convolution with the
    reversed taps, cut to the first N outputs."""
    B, N, d = x.shape
    y = np.empty_like(x)
    for b in range(B):
        for c in range(d):
            y[b, :, c] = np.convolve(x[b, :, c], conv_x[c, ::-1])[:N]
    return y


def _split(y, H, D):
    B, N, _ = y.shape
    HD = H * D
    parts = [y[..., s * HD:(s + 1) * HD].reshape(B, N, H, D) for s in range(4)]
    return dict(q=parts[0], k=parts[1], v=parts[2], out_gate=parts[3], gate=y[..., 4 * HD:])


def pin_project_library(lib):
    """Front end = numpy convolution of each X channel, then one matrix product
    with the stacked weights, split into Q, K, V, R (per head) and w_g."""
    rng = _rng(70)
    for (B, N, d, H, D) in [(2, 13, 8, 2, 3), (1, 5, 16, 3, 4), (3, 2, 4, 1, 2)]:
        x, conv_x, w = _project_inputs(rng, B, N, d, H, D)
        got = oracle.gbla_project(x, conv_x, w, H, D, lib=lib)
        want = _split(_np_conv_x(x, conv_x) @ w.T, H, D)
        for n in want:
            np.testing.assert_allclose(got[n], want[n], rtol=0, atol=1e-12, err_msg=n)


def pin_project_identity_taps(lib):
    """Conv1D taps (0, ..., 0, 1) are the identity, leaving plain projections."""
    rng = _rng(71)
    B, N, d, H, D = 2, 7, 6, 2, 2
    x, _, w = _project_inputs(rng, B, N, d, H, D)
    taps = np.zeros((d, W)); taps[:, W - 1] = 1.0
    got = oracle.gbla_project(x, taps, w, H, D, lib=lib)
    want = _split(x @ w.T, H, D)
    for n in want:
        np.testing.assert_allclose(got[n], want[n], rtol=0, atol=1e-12, err_msg=n)


def pin_project_causal_window(lib):
    """A change of x at position t0 reaches exactly the outputs at t0 .. t0+W-1
    (causal, width-W receptive field)."""
    rng = _rng(72)
    B, N, d, H, D = 1, 16, 5, 2, 3
    x, conv_x, w = _project_inputs(rng, B, N, d, H, D)
    a = oracle.gbla_project(x, conv_x, w, H, D, lib=lib)
    t0 = 6
    x2 = x.copy(); x2[0, t0] += rng.standard_normal(d)
    b = oracle.gbla_project(x2, conv_x, w, H, D, lib=lib)
    for n in a:
        diff = np.abs(a[n] - b[n]).reshape(N, -1).max(axis=1)
        assert np.all(diff[:t0] == 0) and np.all(diff[t0 + W:] == 0), n
        assert np.all(diff[t0:t0 + W] > 0), n


def pin_project_padding(lib):
    """Rows past seq_lens[b] are not written, and the valid rows equal an
    unpadded run of that length whatever the padding holds."""
    rng = _rng(73)
    B, N, d, H, D = 2, 12, 6, 2, 2
    x, conv_x, w = _project_inputs(rng, B, N, d, H, D)
    sl = np.array([12, 5], np.int32)
    a = oracle.gbla_project(x, conv_x, w, H, D, seq_lens=sl, lib=lib)
    x2 = x.copy(); x2[1, 5:] = 1e30
    b = oracle.gbla_project(x2, conv_x, w, H, D, seq_lens=sl, lib=lib)
    c = oracle.gbla_project(x[1:2, :5], conv_x, w, H, D, lib=lib)
    for n in a:
        assert np.all(np.isnan(a[n][1, 5:])), n
        assert not np.any(np.isnan(a[n][1, :5])) and not np.any(np.isnan(a[n][0])), n
        np.testing.assert_array_equal(b[n][1, :5], a[n][1, :5])
        np.testing.assert_array_equal(c[n][0], a[n][1, :5])


def pin_project_absdot(lib):
    """absdot = |X~| |W|^T (the magnitude sum of every output's terms): equal
    to the output itself when every term is nonnegative, never below |output|."""
    rng = _rng(74)
    B, N, d, H, D = 1, 9, 7, 2, 2
    x, conv_x, w = _project_inputs(rng, B, N, d, H, D)
    r = oracle.gbla_project(x, conv_x, w, H, D, absdot=True, lib=lib)
    xt = _np_conv_x(x, conv_x)
    np.testing.assert_allclose(r["absdot"], np.abs(xt) @ np.abs(w).T, rtol=1e-13, atol=0)
    y = _split(xt @ w.T, H, D)
    full = np.concatenate([y[n].reshape(B, N, -1) for n in ("q", "k", "v", "out_gate", "gate")],
                          axis=-1)
    assert np.all(r["absdot"] >= np.abs(full) - 1e-12)
    xp, cp, wp = np.abs(x), np.abs(conv_x), np.abs(w)
    rp = oracle.gbla_project(xp, cp, wp, H, D, absdot=True, lib=lib)
    yp = np.concatenate([rp[n].reshape(B, N, -1) for n in ("q", "k", "v", "out_gate", "gate")],
                        axis=-1)
    np.testing.assert_allclose(rp["absdot"], yp, rtol=1e-13, atol=0)


def pin_layer_conv_commutes(lib):
    """With one Conv1D kernel shared by all channels, convolving X before the
    projections (Sec. 2.1 item 1, the layer) equals convolving the projected
    q, k, v inside the core: Conv1D(X) W = Conv1D(X W).  Gate and out-gate
    inputs come from X~ in both."""
    rng = _rng(75)
    B, N, d, H, D = 2, 21, 6, 2, 3
    x, _, w = _project_inputs(rng, B, N, d, H, D)
    shared = 0.5 * rng.standard_normal(W)
    conv_x = np.tile(shared, (d, 1))
    norm_w = 1.0 + 0.02 * rng.standard_normal((H, D))
    sl = np.array([21, 14], np.int32)
    y_layer = oracle.gbla_layer(x, conv_x, w, norm_w, H, D, seq_lens=sl, lib=lib)
    plain = _split(x @ w.T, H, D)                      # projections of the raw X
    conved = _split(_np_conv_x(x, conv_x) @ w.T, H, D)  # gate / out-gate from X~
    conv_w = np.tile(shared, (3, H, D, 1))
    y_core = oracle.gbla_forward(plain["q"], plain["k"], plain["v"], conved["gate"],
                                 conved["out_gate"], conv_w, norm_w, seq_lens=sl, lib=lib)
    np.testing.assert_allclose(y_layer, y_core, rtol=0, atol=1e-10)


# --- bidirectional softmax attention (Sec. 2), the SA layer of the hybrid ------

def _sa_inputs(rng, B=2, N=9, H=3, D=5):
    return tuple(rng.standard_normal((B, N, H, D)) for _ in range(3))


def pin_sa_library(lib):
    """Attn(q_i) = softmax_j(q_i . k_j / sqrt(D)) V over the valid keys, by numpy
    matrix products and scipy's softmax, per (batch, head)."""
    rng = _rng(80)
    q, k, v = _sa_inputs(rng)
    sl = np.array([9, 4], np.int32)
    y = oracle.softmax_attention(q, k, v, seq_lens=sl, lib=lib)
    D = q.shape[3]
    for b in range(2):
        L = sl[b]
        for h in range(3):
            s = q[b, :L, h] @ k[b, :L, h].T / math.sqrt(D)
            ref = scipy.special.softmax(s, axis=1) @ v[b, :L, h]
            np.testing.assert_allclose(y[b, :L, h], ref, rtol=1e-12, atol=1e-14)
        assert np.all(np.isnan(y[b, L:])), "rows past the sequence end were written"


def pin_sa_torch(lib):
    """torch's own attention (fp64, keys past the end masked) gives the same rows."""
    rng = _rng(81)
    q, k, v = _sa_inputs(rng, B=2, N=11, H=2, D=8)
    sl = np.array([11, 6], np.int32)
    y = oracle.softmax_attention(q, k, v, seq_lens=sl, lib=lib)
    t = lambda a: torch.tensor(a).permute(0, 2, 1, 3)  # noqa: E731  [B, H, N, D]
    mask = torch.zeros(2, 1, 11, 11, dtype=torch.bool)
    for b in range(2):
        mask[b, :, :, :sl[b]] = True
    ref = torch.nn.functional.scaled_dot_product_attention(t(q), t(k), t(v), attn_mask=mask)
    ref = ref.permute(0, 2, 1, 3).numpy()
    for b in range(2):
        np.testing.assert_allclose(y[b, :sl[b]], ref[b, :sl[b]], rtol=1e-12, atol=1e-14)


def pin_sa_closed_forms(lib):
    """A single key gives its own value; q = 0 gives the mean of the valid values;
    equal value rows give that row back; a dominant score picks its key's value
    without overflow (the row maximum is subtracted)."""
    rng = _rng(82)
    q, k, v = _sa_inputs(rng, B=1, N=7, H=2, D=4)
    y1 = oracle.softmax_attention(q, k, v, seq_lens=np.array([1], np.int32), lib=lib)
    np.testing.assert_allclose(y1[0, 0], v[0, 0], rtol=0, atol=1e-15)
    y0 = oracle.softmax_attention(np.zeros_like(q), k, v, seq_lens=np.array([5], np.int32),
                                  lib=lib)
    np.testing.assert_allclose(y0[0, :5], np.broadcast_to(v[0, :5].mean(axis=0), (5, 2, 4)),
                               rtol=1e-13, atol=1e-15)
    vc = np.broadcast_to(v[:, :1], v.shape).copy()
    yc = oracle.softmax_attention(q, k, vc, lib=lib)
    np.testing.assert_allclose(yc, np.broadcast_to(vc[:, :1], vc.shape), rtol=1e-13, atol=1e-15)
    kb = k.copy()
    # key 3 dominates query 2 with a score of 1000 in both heads (exp would
    # overflow without the row maximum subtracted)
    for h in range(2):
        kb[0, 3, h] = 1000.0 * math.sqrt(4) * q[0, 2, h] / (q[0, 2, h] @ q[0, 2, h])
    yb = oracle.softmax_attention(q * 1.0, kb, v, lib=lib)
    assert np.all(np.isfinite(yb))
    np.testing.assert_allclose(yb[0, 2], v[0, 3], rtol=0, atol=1e-9)


def pin_sa_rows_and_abs_scale(lib):
    """The one-row entry gives the full oracle's rows; the error scale
    sum_j p_j |v_j| / sum_j p_j is at least |o| and equals it for v >= 0."""
    rng = _rng(84)
    q, k, v = _sa_inputs(rng, B=1, N=10, H=2, D=6)
    y, a = oracle.softmax_attention(q, k, v, seq_lens=np.array([8], np.int32), absout=True,
                                    lib=lib)
    for h in range(2):
        yr, ar = oracle.softmax_attention_rows(q[0, [1, 7], h], k[0, :8, h], v[0, :8, h], lib=lib)
        np.testing.assert_allclose(yr, y[0, [1, 7], h], rtol=1e-14, atol=1e-15)
        np.testing.assert_allclose(ar, a[0, [1, 7], h], rtol=1e-14, atol=1e-15)
    assert np.all(a[0, :8] >= np.abs(y[0, :8]) - 1e-15)
    yp, ap = oracle.softmax_attention(q, k, np.abs(v), absout=True, lib=lib)
    np.testing.assert_allclose(ap, yp, rtol=1e-14, atol=0)


def pin_sa_permutations(lib):
    """Permuting the valid keys together with their values changes nothing;
    permuting the queries permutes the rows; heads are independent."""
    rng = _rng(83)
    q, k, v = _sa_inputs(rng, B=1, N=8, H=3, D=4)
    y = oracle.softmax_attention(q, k, v, lib=lib)
    perm = rng.permutation(8)
    yk = oracle.softmax_attention(q, k[:, perm], v[:, perm], lib=lib)
    np.testing.assert_allclose(yk, y, rtol=1e-12, atol=1e-14)
    yq = oracle.softmax_attention(q[:, perm], k, v, lib=lib)
    np.testing.assert_allclose(yq, y[:, perm], rtol=1e-12, atol=1e-14)
    hp = [2, 0, 1]
    yh = oracle.softmax_attention(q[:, :, hp], k[:, :, hp], v[:, :, hp], lib=lib)
    np.testing.assert_allclose(yh, y[:, :, hp], rtol=1e-12, atol=1e-14)


# --- backward (chain rule through Sec. 2.1's steps) and its error scales ------

_BWD = dict(q="dq", k="dk", v="dv", a="da", og="dog", wq="dwq", wk="dwk", wv="dwv",
            norm_w="dnorm_w")
_SCALED = (("dq", "mdq"), ("dk", "mdk"), ("dv", "mdv"), ("da", "mda"), ("dog", "mdog"),
           ("dwq", "mdwq"), ("dwk", "mdwk"), ("dwv", "mdwv"), ("dnorm_w", "mdnorm_w"))


def _bwd_inputs(rng, L, D):
    q, k, v, a, og, wq, wk, wv, nw = _head_inputs(rng, L, D)
    return dict(q=q, k=k, v=v, a=a, og=og, wq=wq, wk=wk, wv=wv, norm_w=nw)


def pin_backward_finite_differences(lib):
    """Every gradient equals the central difference of sum(dy * y) of the
    oracle's forward (full core and Eq. bla's plain form)."""
    rng = _rng(90)
    x = _bwd_inputs(rng, 6, 3)
    dy = rng.standard_normal((6, 3))
    for flags in (0, oracle.BLA):
        g = oracle.gbla_head_backward(**x, dy=dy, eps=1e-3, flags=flags, lib=lib)
        h = 1e-5
        for name, gname in _BWD.items():
            num = np.empty_like(x[name])
            for idx in np.ndindex(x[name].shape):
                xp = {kk: vv.copy() for kk, vv in x.items()}
                xm = {kk: vv.copy() for kk, vv in x.items()}
                xp[name][idx] += h
                xm[name][idx] -= h
                lp = np.sum(dy * oracle.gbla_head(**xp, eps=1e-3, flags=flags, lib=lib))
                lm = np.sum(dy * oracle.gbla_head(**xm, eps=1e-3, flags=flags, lib=lib))
                num[idx] = (lp - lm) / (2 * h)
            np.testing.assert_allclose(g[gname], num, rtol=1e-6, atol=1e-8,
                                       err_msg=f"{gname} flags={flags}")


def pin_backward_threaded_equals_serial(lib):
    """The per-head Python loop (threads over heads) gives exactly the serial
    (batch, head) loop written in C, padding rows zero."""
    rng = _rng(91)
    B, N, H, D = 2, 11, 3, 4
    arrs = dict(q=rng.standard_normal((B, N, H, D)), k=rng.standard_normal((B, N, H, D)),
                v=rng.standard_normal((B, N, H, D)), gate=rng.standard_normal((B, N, H)),
                out_gate=rng.standard_normal((B, N, H, D)),
                conv_w=0.5 * rng.standard_normal((3, H, D, W)),
                norm_w=1.0 + 0.1 * rng.standard_normal((H, D)))
    dy = rng.standard_normal((B, N, H, D))
    a = oracle.gbla_backward(**arrs, dy=dy, seq_lens=[11, 4], n_threads=3, lib=lib)
    b = oracle.gbla_backward_serial(**arrs, dy=dy, seq_lens=[11, 4], lib=lib)
    for n in b:
        assert np.array_equal(a[n], b[n]), n
    assert np.all(a["dq"][1, 4:] == 0) and np.all(a["dgate"][1, 4:] == 0)


def _scaled_case(seed, flags, L=40, D=6):
    rng = _rng(seed)
    x = _bwd_inputs(rng, L, D)
    dy = rng.standard_normal((L, D))
    return x, dy


def pin_backward_scales_dominate(lib):
    """Each error scale is at least the magnitude of its gradient (it is the
    same chain rule on magnitudes, with the absolute state sums)."""
    for flags in (0, oracle.NO_CONV, oracle.NO_GATE, oracle.NO_NORM, oracle.BLA):
        x, dy = _scaled_case(92, flags)
        g = oracle.gbla_head_backward(**x, dy=dy, flags=flags, scales=True, lib=lib)
        for n, m in _SCALED:
            assert np.all(g[m] >= np.abs(g[n]) * (1 - 1e-12)), (n, flags)


def pin_backward_scales_bound_dy_perturbation(lib):
    """The gradients are linear in dy and the scales depend on |dy| only, so a
    perturbation dy -> dy (1 + e r), |r| <= 1, moves every gradient by at most
    e times its scale."""
    x, dy = _scaled_case(93, 0)
    g0 = oracle.gbla_head_backward(**x, dy=dy, scales=True, lib=lib)
    e = 1e-6
    r = _rng(94).uniform(-1, 1, dy.shape)
    g1 = oracle.gbla_head_backward(**x, dy=dy * (1 + e * r), lib=lib)
    for n, m in _SCALED:
        assert np.all(np.abs(g1[n] - g0[n]) <= e * g0[m] * (1 + 1e-6) + 1e-300), n
    g2 = oracle.gbla_head_backward(**x, dy=-3.0 * dy, scales=True, lib=lib)
    for n, m in _SCALED:
        np.testing.assert_allclose(g2[m], 3.0 * g0[m], rtol=1e-12, atol=0, err_msg=m)


def pin_backward_scales_bound_input_perturbation(lib):
    """Relative perturbations e of q, k or v (which reach the rounded
    intermediates phi(q~), K^ and V~ through the Conv1D) move every
    per-token gradient by less than e times its scale."""
    for flags in (0, oracle.NO_CONV):
        x, dy = _scaled_case(95, flags, L=60)
        g0 = oracle.gbla_head_backward(**x, dy=dy, flags=flags, scales=True, lib=lib)
        e = 1e-7
        for name in ("q", "k", "v"):
            r = _rng(96).uniform(-1, 1, x[name].shape)
            x1 = dict(x)
            x1[name] = x[name] * (1 + e * r)
            g1 = oracle.gbla_head_backward(**x1, dy=dy, flags=flags, lib=lib)
            for n, m in _SCALED[:5]:
                assert np.all(np.abs(g1[n] - g0[n]) <= e * g0[m]), (name, n, flags)


def pin_backward_scales_exact_without_cancellation(lib):
    """With nothing that can cancel (Eq. bla's plain form, v >= 0, dy >= 0) the
    value gradient's scale equals the gradient: dv~ = dS^T K^ with dS >= 0."""
    x, dy = _scaled_case(97, oracle.BLA)
    x["v"] = np.abs(x["v"])
    g = oracle.gbla_head_backward(**x, dy=np.abs(dy), flags=oracle.BLA, scales=True, lib=lib)
    np.testing.assert_allclose(g["mdv"], g["dv"], rtol=1e-12, atol=0)


ALL_PINS = [v for k_, v in sorted(globals().items()) if k_.startswith("pin_")]
