"""Pins of the oracle's backward (chain rule through the layer core, Sec. 2.1)
against things other than itself: central finite differences of the oracle's
forward, autograd of an independently written PyTorch fp64 forward, and
invariants of the forward (the softmax's shift invariance; scale invariance of
RMSNorm with eps = 0)."""
import numpy as np
import pytest
import torch

import oracle

FLAG_SETS = [0, oracle.NO_CONV, oracle.NO_GATE, oracle.NO_NORM, oracle.BLA]


def _head(seed, L=7, D=4, W=4):
    rng = np.random.default_rng(seed)
    q, k, v, og, dy = (rng.standard_normal((L, D)) for _ in range(5))
    a = rng.standard_normal(L)
    wq, wk, wv = (0.5 * rng.standard_normal((D, W)) for _ in range(3))
    nw = 1.0 + 0.02 * rng.standard_normal(D)
    return dict(q=q, k=k, v=v, a=a, og=og, wq=wq, wk=wk, wv=wv, norm_w=nw), dy


@pytest.mark.parametrize("flags", FLAG_SETS)
def test_backward_matches_finite_differences(flags):
    x, dy = _head(1)
    eps = 1e-3  # a larger eps keeps the norm's curvature moderate for the differences
    grads = oracle.gbla_head_backward(**x, dy=dy, eps=eps, flags=flags)
    names = dict(q="dq", k="dk", v="dv", a="da", og="dog", wq="dwq", wk="dwk", wv="dwv",
                 norm_w="dnorm_w")

    def loss(xx):
        return float(np.sum(dy * oracle.gbla_head(**xx, eps=eps, flags=flags)))

    h = 1e-5
    for name, gname in names.items():
        base = x[name]
        num = np.empty_like(base)
        for idx in np.ndindex(base.shape):
            xp = {kk: vv.copy() for kk, vv in x.items()}
            xm = {kk: vv.copy() for kk, vv in x.items()}
            xp[name][idx] += h
            xm[name][idx] -= h
            num[idx] = (loss(xp) - loss(xm)) / (2 * h)
        np.testing.assert_allclose(grads[gname], num, rtol=1e-6, atol=1e-8,
                                   err_msg=f"{gname} (flags={flags})")


def _torch_forward(q, k, v, gate, og, conv_w, norm_w, seq_lens, eps, flags):
    """Plain PyTorch fp64 forward of the layer core, written from Sec. 2.1."""
    B, N, H, D = q.shape
    W = conv_w.shape[-1]
    ys = []
    for b in range(B):
        L = int(seq_lens[b])
        rows = []
        for h in range(H):
            def conv(x, s):
                if flags & oracle.NO_CONV:
                    return x
                xt = torch.nn.functional.pad(x.T.unsqueeze(0), (W - 1, 0))
                return torch.nn.functional.conv1d(xt, conv_w[s, h].unsqueeze(1), groups=D)[0].T
            qt, kt, vt = conv(q[b, :L, h], 0), conv(k[b, :L, h], 1), conv(v[b, :L, h], 2)
            phi = lambda x: torch.nn.functional.elu(x) + 1.0
            if flags & oracle.NO_GATE:
                g = torch.full((L,), 1.0 / L, dtype=q.dtype)
            else:
                g = torch.softmax(gate[b, :L, h], dim=0)
            kh = g[:, None] * phi(kt)
            S = kh.T @ vt
            z = kh.sum(0)
            pq = phi(qt)
            O = (pq @ S) / (pq @ z)[:, None]
            if flags & oracle.NO_NORM:
                y = O
            else:
                r = torch.rsqrt((O * O).mean(-1, keepdim=True) + eps)
                y = O * r * norm_w[h] * torch.nn.functional.silu(og[b, :L, h])
            rows.append(y)
        ys.append(rows)
    return ys


@pytest.mark.parametrize("flags", FLAG_SETS)
def test_backward_matches_autograd(flags):
    rng = np.random.default_rng(2)
    B, N, H, D, W = 2, 33, 2, 8, 4
    seq_lens = np.array([33, 20], np.int32)
    arrs = dict(q=rng.standard_normal((B, N, H, D)), k=rng.standard_normal((B, N, H, D)),
                v=rng.standard_normal((B, N, H, D)), gate=rng.standard_normal((B, N, H)),
                out_gate=rng.standard_normal((B, N, H, D)),
                conv_w=0.5 * rng.standard_normal((3, H, D, W)),
                norm_w=1.0 + 0.02 * rng.standard_normal((H, D)))
    dy = rng.standard_normal((B, N, H, D))
    eps = oracle.RMS_EPS
    got = oracle.gbla_backward(**arrs, dy=dy, seq_lens=seq_lens, eps=eps, flags=flags)

    t = {kk: torch.tensor(vv, requires_grad=True) for kk, vv in arrs.items()}
    ys = _torch_forward(t["q"], t["k"], t["v"], t["gate"], t["out_gate"], t["conv_w"],
                        t["norm_w"], seq_lens, eps, flags)
    dyt = torch.tensor(dy)
    loss = sum((ys[b][h] * dyt[b, :int(seq_lens[b]), h]).sum()
               for b in range(B) for h in range(H))
    loss.backward()
    pairs = dict(q="dq", k="dk", v="dv", gate="dgate", out_gate="dout_gate",
                 conv_w="dconv_w", norm_w="dnorm_w")
    for name, gname in pairs.items():
        # an input the variant does not use has no autograd gradient: zero
        ref = t[name].grad.numpy() if t[name].grad is not None else np.zeros_like(arrs[name])
        np.testing.assert_allclose(got[gname], ref, rtol=1e-9, atol=1e-11,
                                   err_msg=f"{gname} (flags={flags})")


def test_gate_gradient_sums_to_zero():
    # y is unchanged by a constant shift of one head's logits (softmax), so the
    # logit gradient of every (b, h) sums to zero
    x, dy = _head(3, L=40, D=8)
    g = oracle.gbla_head_backward(**x, dy=dy)
    assert abs(g["da"].sum()) < 1e-12 * max(1.0, np.abs(g["da"]).sum())


def test_value_scale_invariance_without_eps():
    # with eps = 0, y(c v) = y(v) (O scales with v, RMSNorm removes the scale),
    # so the directional derivative <dv, v> vanishes
    x, dy = _head(4, L=30, D=8)
    x["wv"] = x["wv"]  # v~ is linear in v: the scale passes through the conv
    g = oracle.gbla_head_backward(**x, dy=dy, eps=0.0)
    assert abs(np.sum(g["dv"] * x["v"])) < 1e-10 * np.abs(g["dv"]).sum()


def test_padded_rows_get_no_gradient():
    rng = np.random.default_rng(5)
    B, N, H, D, W = 2, 12, 1, 4, 4
    arrs = dict(q=rng.standard_normal((B, N, H, D)), k=rng.standard_normal((B, N, H, D)),
                v=rng.standard_normal((B, N, H, D)), gate=rng.standard_normal((B, N, H)),
                out_gate=rng.standard_normal((B, N, H, D)),
                conv_w=0.5 * rng.standard_normal((3, H, D, W)),
                norm_w=np.ones((H, D)))
    dy = rng.standard_normal((B, N, H, D))
    got = oracle.gbla_backward(**arrs, dy=dy, seq_lens=[12, 5])
    for name in ("dq", "dk", "dv", "dout_gate"):
        assert np.all(got[name][1, 5:] == 0.0)
    assert np.all(got["dgate"][1, 5:] == 0.0)
