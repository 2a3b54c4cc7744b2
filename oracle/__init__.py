"""fp64 CPU oracle of the GBLA layer-core forward.

TEST INFRASTRUCTURE ONLY.  Only the tests, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this package.  It shares no code
with the CUDA library in ``paper_2606_07317_gb300``; neither imports the other.

The arithmetic lives in ``gbla_oracle.c`` (plain C, double precision), which
follows Sec. 2 (bidirectional linear attention, Eq. bla) and Sec. 2.1 (GBLA:
Conv1D, key gating, gated RMSNorm) of the paper.  This module only compiles
it with gcc and marshals numpy arrays into it.

The bidirectional softmax attention of Sec. 2 (``softmax_attention``), the SA
layer of the paper's hybrid [SA, LA, LA] encoder, is pinned by the
``pin_sa_*`` checks (library softmax and matrix products, torch's own
attention, invariants).

The layer front end (``gbla_project``: the X-space Conv1D and the stacked
Q, K, V, R and w_g projections of Sec. 2.1 items 1-3) and the whole layer
(``gbla_layer``: front end, then the core with its Conv1D off) are pinned by
the ``pin_project_*`` and ``pin_layer_conv_commutes`` checks.

Parity status: every function here is pinned by ``tests/test_oracle_pins.py``
against library routines, closed forms, the quadratic (L x L) form and
invariants.  The paper's own unstated choices (phi, eps, conv tap order, the
norm weight's shape) are readings, listed in the C file's header.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "gbla_oracle.c")
_OUT_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_OUT_DIR, "liboracle.so")

NO_CONV = 1  # identity Conv1D (ablation "W/o Conv1D")
NO_GATE = 2  # uniform key gate (ablation "W/o Key gating")
NO_NORM = 4  # no gated RMSNorm (ablation "W/o Gated RMSNorm")
BLA = NO_CONV | NO_GATE | NO_NORM  # all add-ons off: Eq. bla

RMS_EPS = 1e-6  # RMSNorm epsilon (the paper leaves it unstated; fixed reading)
CONV_W = 4      # Conv1D kernel size used in the paper's experiments

_lock = threading.Lock()
_lib = None

_dp = ctypes.POINTER(ctypes.c_double)


def build(src: str = _SRC, out: str = _LIB_PATH, extra_flags=()) -> str:
    """Compile the oracle into a shared library with gcc and return its path.

    -ffp-contract=off keeps the double arithmetic identical on x86 and Arm.
    """
    os.makedirs(os.path.dirname(out), exist_ok=True)
    tmp = out + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fPIC", "-shared",
           *extra_flags, src, "-o", tmp, "-lm", "-lpthread"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, out)
    return out


def _declare(lib):
    lib.oracle_phi.restype = ctypes.c_double
    lib.oracle_phi.argtypes = [ctypes.c_double]
    lib.oracle_silu.restype = ctypes.c_double
    lib.oracle_silu.argtypes = [ctypes.c_double]
    lib.oracle_conv1d.restype = None
    lib.oracle_conv1d.argtypes = [_dp, ctypes.c_long, ctypes.c_int, ctypes.c_long,
                                  _dp, ctypes.c_int, _dp]
    lib.oracle_softmax.restype = None
    lib.oracle_softmax.argtypes = [_dp, ctypes.c_long, ctypes.c_long, _dp]
    lib.oracle_gated_rmsnorm_row.restype = None
    lib.oracle_gated_rmsnorm_row.argtypes = [_dp, _dp, _dp, ctypes.c_int,
                                             ctypes.c_double, _dp]
    head_common = [_dp, _dp, _dp, _dp, _dp, ctypes.c_long, ctypes.c_long,
                   ctypes.c_long, ctypes.c_int, _dp, _dp, _dp, ctypes.c_int, _dp,
                   ctypes.c_double, ctypes.c_int, _dp]
    lib.oracle_gbla_head.restype = ctypes.c_int
    lib.oracle_gbla_head.argtypes = head_common + [_dp] * 7
    lib.oracle_gbla_head_quadratic.restype = ctypes.c_int
    lib.oracle_gbla_head_quadratic.argtypes = head_common + [_dp]
    lib.oracle_gbla_head_backward.restype = ctypes.c_int
    lib.oracle_gbla_head_backward.argtypes = (
        [_dp, _dp, _dp, _dp, _dp, ctypes.c_long, ctypes.c_long, ctypes.c_long, ctypes.c_int,
         _dp, _dp, _dp, ctypes.c_int, _dp, ctypes.c_double, ctypes.c_int, _dp] + [_dp] * 18)
    lib.oracle_gbla_backward.restype = ctypes.c_int
    lib.oracle_gbla_backward.argtypes = [_dp, _dp, _dp, _dp, _dp, _dp, _dp,
                                         ctypes.POINTER(ctypes.c_int32),
                                         ctypes.c_long, ctypes.c_long, ctypes.c_long,
                                         ctypes.c_int, ctypes.c_int, ctypes.c_double,
                                         ctypes.c_int, _dp] + [_dp] * 7
    lib.oracle_gbla_project.restype = ctypes.c_int
    lib.oracle_gbla_project.argtypes = [_dp, _dp, _dp, ctypes.POINTER(ctypes.c_int32),
                                        ctypes.c_long, ctypes.c_long, ctypes.c_int,
                                        ctypes.c_int, ctypes.c_long, ctypes.c_int] + [_dp] * 6
    lib.oracle_softmax_attention.restype = ctypes.c_int
    lib.oracle_softmax_attention.argtypes = [_dp, _dp, _dp, ctypes.POINTER(ctypes.c_int32),
                                             ctypes.c_long, ctypes.c_long, ctypes.c_long,
                                             ctypes.c_int, ctypes.c_int, _dp, _dp]
    lib.oracle_softmax_attention_rows.restype = ctypes.c_int
    lib.oracle_softmax_attention_rows.argtypes = [_dp, ctypes.c_long, _dp, _dp, ctypes.c_long,
                                                  ctypes.c_int, _dp, _dp]
    lib.oracle_gbla_forward.restype = ctypes.c_int
    lib.oracle_gbla_forward.argtypes = [_dp, _dp, _dp, _dp, _dp, _dp, _dp,
                                        ctypes.POINTER(ctypes.c_int32),
                                        ctypes.c_long, ctypes.c_long, ctypes.c_long,
                                        ctypes.c_int, ctypes.c_int, ctypes.c_double,
                                        ctypes.c_int, ctypes.c_int, _dp]
    return lib


def load(path: str | None = None):
    """Load (building first if needed) the oracle library."""
    global _lib
    with _lock:
        if path is not None:
            return _declare(ctypes.CDLL(path))
        if _lib is None:
            if (not os.path.exists(_LIB_PATH)
                    or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC)):
                build()
            _lib = _declare(ctypes.CDLL(_LIB_PATH))
        return _lib


def _f64(x) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(x, dtype=np.float64))


def _ptr(a: np.ndarray | None):
    if a is None:
        return None
    return a.ctypes.data_as(_dp)


def phi(x: float, lib=None) -> float:
    return (lib or load()).oracle_phi(float(x))


def silu(x: float, lib=None) -> float:
    return (lib or load()).oracle_silu(float(x))


def conv1d(x, w, lib=None) -> np.ndarray:
    """Causal depthwise Conv1D.  x: [L, C], w: [C, W] -> [L, C]."""
    x = _f64(x); w = _f64(w)
    L, C = x.shape
    y = np.empty((L, C), np.float64)
    (lib or load()).oracle_conv1d(_ptr(x), L, C, C, _ptr(w), w.shape[1], _ptr(y))
    return y


def softmax(a, lib=None) -> np.ndarray:
    """Key-gate softmax over the sequence.  a: [L] -> [L]."""
    a = _f64(a)
    g = np.empty(a.shape[0], np.float64)
    (lib or load()).oracle_softmax(_ptr(a), a.shape[0], 1, _ptr(g))
    return g


def gated_rmsnorm_row(O, og, w, eps=RMS_EPS, lib=None) -> np.ndarray:
    O = _f64(O); og = _f64(og); w = _f64(w)
    y = np.empty(O.shape[0], np.float64)
    (lib or load()).oracle_gated_rmsnorm_row(_ptr(O), _ptr(og), _ptr(w), O.shape[0],
                                             float(eps), _ptr(y))
    return y


def gbla_head(q, k, v, a, og, wq, wk, wv, norm_w, eps=RMS_EPS, flags=0,
              intermediates=False, lib=None):
    """One (batch, head): q, k, v, og [L, D]; a [L]; wq/wk/wv [D, W]; norm_w [D].

    Returns y [L, D], or (y, dict of intermediates) when asked.
    """
    q, k, v, og = (_f64(t) for t in (q, k, v, og))
    a = _f64(a); wq, wk, wv = (_f64(t) for t in (wq, wk, wv)); norm_w = _f64(norm_w)
    L, D = q.shape
    W = wq.shape[1]
    y = np.empty((L, D), np.float64)
    inter = None
    if intermediates:
        inter = dict(qt=np.empty((L, D)), kt=np.empty((L, D)), vt=np.empty((L, D)),
                     g=np.empty(L), S=np.empty((D, D)), z=np.empty(D),
                     O=np.empty((L, D)))
    ptrs = ([_ptr(inter[n]) for n in ("qt", "kt", "vt", "g", "S", "z", "O")]
            if inter else [None] * 7)
    rc = (lib or load()).oracle_gbla_head(
        _ptr(q), _ptr(k), _ptr(v), _ptr(a), _ptr(og), D, 1, L, D,
        _ptr(wq), _ptr(wk), _ptr(wv), W, _ptr(norm_w), float(eps), int(flags),
        _ptr(y), *ptrs)
    if rc != 0:
        raise ValueError(f"oracle_gbla_head rejected its arguments ({rc})")
    return (y, inter) if intermediates else y


def gbla_head_quadratic(q, k, v, a, og, wq, wk, wv, norm_w, eps=RMS_EPS, flags=0,
                        lib=None):
    """Same as gbla_head through the explicit L x L matrix; returns (y, O)."""
    q, k, v, og = (_f64(t) for t in (q, k, v, og))
    a = _f64(a); wq, wk, wv = (_f64(t) for t in (wq, wk, wv)); norm_w = _f64(norm_w)
    L, D = q.shape
    y = np.empty((L, D)); O = np.empty((L, D))
    rc = (lib or load()).oracle_gbla_head_quadratic(
        _ptr(q), _ptr(k), _ptr(v), _ptr(a), _ptr(og), D, 1, L, D,
        _ptr(wq), _ptr(wk), _ptr(wv), wq.shape[1], _ptr(norm_w), float(eps),
        int(flags), _ptr(y), _ptr(O))
    if rc != 0:
        raise ValueError(f"oracle_gbla_head_quadratic rejected its arguments ({rc})")
    return y, O


def gbla_forward(q, k, v, gate, out_gate, conv_w, norm_w, seq_lens=None,
                 eps=RMS_EPS, flags=0, n_threads=1, out=None, lib=None):
    """Whole core over [B, N, H, D] arrays; rows t >= seq_lens[b] keep `out`'s values
    (NaN when `out` is not given).  conv_w: [3, H, D, W]; norm_w: [H, D]."""
    q, k, v, og = (_f64(t) for t in (q, k, v, out_gate))
    gate = _f64(gate); conv_w = _f64(conv_w); norm_w = _f64(norm_w)
    B, N, H, D = q.shape
    W = conv_w.shape[-1]
    y = np.full((B, N, H, D), np.nan) if out is None else out
    assert y.dtype == np.float64 and y.flags.c_contiguous and y.shape == q.shape
    sl = None
    if seq_lens is not None:
        sl = np.ascontiguousarray(np.asarray(seq_lens, dtype=np.int32))
    rc = (lib or load()).oracle_gbla_forward(
        _ptr(q), _ptr(k), _ptr(v), _ptr(gate), _ptr(og), _ptr(conv_w), _ptr(norm_w),
        sl.ctypes.data_as(ctypes.POINTER(ctypes.c_int32)) if sl is not None else None,
        B, H, N, D, W, float(eps), int(flags), int(n_threads), _ptr(y))
    if rc != 0:
        raise ValueError(f"oracle_gbla_forward rejected its arguments ({rc})")
    return y


def softmax_attention(q, k, v, seq_lens=None, n_threads=1, out=None, absout=False, lib=None):
    """Bidirectional softmax attention of Sec. 2 over [B, N, H, D] arrays: for
    every valid query i < L_b, sum_j exp(q_i . k_j / sqrt(D)) v_j / sum_j exp(...)
    over the valid keys j < L_b.  Rows t >= L_b keep `out`'s values (NaN when
    `out` is not given).  With absout=True also returns sum_j p_j |v_j| / sum_j p_j
    per output (the scale of the error a relative rounding of the probabilities
    p_j makes)."""
    q, k, v = (_f64(t) for t in (q, k, v))
    B, N, H, D = q.shape
    y = np.full((B, N, H, D), np.nan) if out is None else out
    assert y.dtype == np.float64 and y.flags.c_contiguous and y.shape == q.shape
    a = np.full((B, N, H, D), np.nan) if absout else None
    sl = None
    if seq_lens is not None:
        sl = np.ascontiguousarray(np.asarray(seq_lens, dtype=np.int32))
    rc = (lib or load()).oracle_softmax_attention(
        _ptr(q), _ptr(k), _ptr(v),
        sl.ctypes.data_as(ctypes.POINTER(ctypes.c_int32)) if sl is not None else None,
        B, N, H, D, int(n_threads), _ptr(y), _ptr(a))
    if rc != 0:
        raise ValueError(f"oracle_softmax_attention rejected its arguments ({rc})")
    return (y, a) if absout else y


def softmax_attention_rows(q_rows, k, v, lib=None):
    """Selected query rows q_rows [R, D] of one (batch, head) against its valid
    keys and values k, v [L, D]; returns (out, absout), each [R, D]."""
    q_rows, k, v = (_f64(t) for t in (q_rows, k, v))
    R, D = q_rows.shape
    L = k.shape[0]
    y = np.empty((R, D))
    a = np.empty((R, D))
    rc = (lib or load()).oracle_softmax_attention_rows(_ptr(q_rows), R, _ptr(k), _ptr(v), L, D,
                                                       _ptr(y), _ptr(a))
    if rc != 0:
        raise ValueError(f"oracle_softmax_attention_rows rejected its arguments ({rc})")
    return y, a


def gbla_head_backward(q, k, v, a, og, wq, wk, wv, norm_w, dy, eps=RMS_EPS, flags=0,
                       scales=False, lib=None):
    """Gradients of sum(dy * y) for one (batch, head) (chain rule through the six
    forward steps of Sec. 2.1, reverse order).  Returns a dict with dq, dk, dv, dog
    [L, D], da [L], dwq, dwk, dwv [D, W] and dnorm_w [D]; with ``scales`` also the
    error scales mdq, mdk, mdv, mdog [L, D], mda [L], mdwq, mdwk, mdwv [D, W] and
    mdnorm_w [D] (see oracle_gbla_head_backward in the C file)."""
    q, k, v, og, dy = (_f64(t) for t in (q, k, v, og, dy))
    a = _f64(a); wq, wk, wv = (_f64(t) for t in (wq, wk, wv)); norm_w = _f64(norm_w)
    L, D = q.shape
    W = wq.shape[1]
    out = dict(dq=np.zeros((L, D)), dk=np.zeros((L, D)), dv=np.zeros((L, D)),
               da=np.zeros(L), dog=np.zeros((L, D)), dwq=np.zeros((D, W)),
               dwk=np.zeros((D, W)), dwv=np.zeros((D, W)), dnorm_w=np.zeros(D))
    mags = [None] * 9
    if scales:
        out.update(mdq=np.zeros((L, D)), mdk=np.zeros((L, D)), mdv=np.zeros((L, D)),
                   mda=np.zeros(L), mdog=np.zeros((L, D)), mdwq=np.zeros((D, W)),
                   mdwk=np.zeros((D, W)), mdwv=np.zeros((D, W)), mdnorm_w=np.zeros(D))
        mags = [_ptr(out[n]) for n in ("mdq", "mdk", "mdv", "mda", "mdog", "mdwq", "mdwk",
                                       "mdwv", "mdnorm_w")]
    rc = (lib or load()).oracle_gbla_head_backward(
        _ptr(q), _ptr(k), _ptr(v), _ptr(a), _ptr(og), D, 1, L, D, _ptr(wq), _ptr(wk),
        _ptr(wv), W, _ptr(norm_w), float(eps), int(flags), _ptr(dy),
        *[_ptr(out[n]) for n in ("dq", "dk", "dv", "da", "dog", "dwq", "dwk", "dwv",
                                 "dnorm_w")], *mags)
    if rc != 0:
        raise ValueError(f"oracle_gbla_head_backward rejected its arguments ({rc})")
    return out


def _at(arr, offset):
    """Pointer to element `offset` of a C-contiguous float64 array."""
    return ctypes.cast(arr.ctypes.data + 8 * int(offset), _dp)


def gbla_backward(q, k, v, gate, out_gate, conv_w, norm_w, dy, seq_lens=None,
                  eps=RMS_EPS, flags=0, scales=False, n_threads=1, lib=None):
    """Whole-core backward over [B, N, H, D] arrays: gradients of sum(dy * y).

    Returns a dict: dq, dk, dv, dout_gate [B, N, H, D]; dgate [B, N, H]; dconv_w
    [3, H, D, W]; dnorm_w [H, D].  Rows past seq_lens[b] are zero.  With
    ``scales``, also the error scales mdq, mdk, mdv, mdout_gate [B, N, H, D],
    mdgate [B, N, H] (zero past seq_lens[b]), mdconv_w [3, H, D, W] and
    mdnorm_w [H, D].

    One call of oracle_gbla_head_backward per (batch, head).  With n_threads > 1
    the heads run on that many threads, each head taking its batches in batch
    order, so the tap and norm-weight sums over the batch are added in the same
    order as by oracle_gbla_backward (the serial loop in C) and equal its
    results exactly."""
    q, k, v, og, dy = (_f64(t) for t in (q, k, v, out_gate, dy))
    gate = _f64(gate); conv_w = _f64(conv_w); norm_w = _f64(norm_w)
    B, N, H, D = q.shape
    W = conv_w.shape[-1]
    names = ["dq", "dk", "dv", "dgate", "dout_gate", "dconv_w", "dnorm_w"]
    out = dict(dq=np.zeros_like(q), dk=np.zeros_like(q), dv=np.zeros_like(q),
               dgate=np.zeros_like(gate), dout_gate=np.zeros_like(q),
               dconv_w=np.zeros_like(conv_w), dnorm_w=np.zeros_like(norm_w))
    if scales:
        for n in names:
            out["m" + n] = np.zeros_like(out[n])
    sl = None if seq_lens is None else np.asarray(seq_lens, dtype=np.int64)
    lb = lib or load()
    ld = H * D

    def head(h):
        for b in range(B):
            L = N if sl is None else int(min(max(sl[b], 0), N))
            base, gbase = (b * N * H + h) * D, b * N * H + h
            grads = [_at(out[n], gbase if n == "dgate" else base)
                     for n in ("dq", "dk", "dv", "dgate", "dout_gate")]
            taps = [_at(out["dconv_w"], ((i * H + h) * D) * W) for i in range(3)]
            mags = [None] * 9
            if scales:
                mags = [_at(out["m" + n], gbase if n == "dgate" else base)
                        for n in ("dq", "dk", "dv", "dgate", "dout_gate")]
                mags += [_at(out["mdconv_w"], ((i * H + h) * D) * W) for i in range(3)]
                mags += [_at(out["mdnorm_w"], h * D)]
            rc = lb.oracle_gbla_head_backward(
                _at(q, base), _at(k, base), _at(v, base), _at(gate, gbase), _at(og, base),
                ld, H, L, D, *[_at(conv_w, ((i * H + h) * D) * W) for i in range(3)], W,
                _at(norm_w, h * D), float(eps), int(flags), _at(dy, base),
                *grads, *taps, _at(out["dnorm_w"], h * D), *mags)
            if rc != 0:
                raise ValueError(f"oracle_gbla_head_backward rejected its arguments ({rc})")

    if n_threads > 1 and H > 1:
        from concurrent.futures import ThreadPoolExecutor
        with ThreadPoolExecutor(max_workers=min(n_threads, H)) as ex:
            list(ex.map(head, range(H)))
    else:
        for h in range(H):
            head(h)
    return out


def gbla_backward_serial(q, k, v, gate, out_gate, conv_w, norm_w, dy, seq_lens=None,
                         eps=RMS_EPS, flags=0, lib=None):
    """The same gradients through oracle_gbla_backward, the serial (batch, head)
    loop written in C (pins the Python loop of gbla_backward)."""
    q, k, v, og, dy = (_f64(t) for t in (q, k, v, out_gate, dy))
    gate = _f64(gate); conv_w = _f64(conv_w); norm_w = _f64(norm_w)
    B, N, H, D = q.shape
    W = conv_w.shape[-1]
    out = dict(dq=np.empty_like(q), dk=np.empty_like(q), dv=np.empty_like(q),
               dgate=np.empty_like(gate), dout_gate=np.empty_like(q),
               dconv_w=np.empty_like(conv_w), dnorm_w=np.empty_like(norm_w))
    sl = None
    if seq_lens is not None:
        sl = np.ascontiguousarray(np.asarray(seq_lens, dtype=np.int32))
    rc = (lib or load()).oracle_gbla_backward(
        _ptr(q), _ptr(k), _ptr(v), _ptr(gate), _ptr(og), _ptr(conv_w), _ptr(norm_w),
        sl.ctypes.data_as(ctypes.POINTER(ctypes.c_int32)) if sl is not None else None,
        B, H, N, D, W, float(eps), int(flags), _ptr(dy),
        *[_ptr(out[n]) for n in ("dq", "dk", "dv", "dgate", "dout_gate", "dconv_w",
                                 "dnorm_w")])
    if rc != 0:
        raise ValueError(f"oracle_gbla_backward rejected its arguments ({rc})")
    return out


def gbla_project(x, conv_x, w, H, D, seq_lens=None, absdot=False, lib=None):
    """Layer front end (Sec. 2.1 items 1-3): X~ = Conv1D(X) over the d channels of
    x [B, N, d] with taps conv_x [d, W], then the stacked projections w [F, d],
    F = 4 H D + H (rows: W_Q, W_K, W_V, W_R per head and dim, then w_g per head).

    Returns a dict: q, k, v, out_gate [B, N, H, D], gate [B, N, H] (rows past
    seq_lens[b] are NaN) and, when asked, absdot [B, N, F] = sum_c |x~_c w_fc|.
    """
    x = _f64(x); conv_x = _f64(conv_x); w = _f64(w)
    B, N, d = x.shape
    F = 4 * H * D + H
    if w.shape != (F, d) or conv_x.shape[0] != d:
        raise ValueError("gbla_project: w must be [4*H*D + H, d] and conv_x [d, W]")
    out = {n: np.full((B, N, H, D), np.nan) for n in ("q", "k", "v", "out_gate")}
    out["gate"] = np.full((B, N, H), np.nan)
    ad = np.full((B, N, F), np.nan) if absdot else None
    sl = None
    if seq_lens is not None:
        sl = np.ascontiguousarray(np.asarray(seq_lens, dtype=np.int32))
    rc = (lib or load()).oracle_gbla_project(
        _ptr(x), _ptr(conv_x), _ptr(w),
        sl.ctypes.data_as(ctypes.POINTER(ctypes.c_int32)) if sl is not None else None,
        B, N, d, conv_x.shape[1], H, D,
        *[_ptr(out[n]) for n in ("q", "k", "v", "out_gate", "gate")], _ptr(ad))
    if rc != 0:
        raise ValueError(f"oracle_gbla_project rejected its arguments ({rc})")
    if absdot:
        out["absdot"] = ad
    return out


def gbla_layer(x, conv_x, w, norm_w, H, D, seq_lens=None, store=None, eps=RMS_EPS,
               lib=None):
    """Whole GBLA layer of Sec. 2.1 from the embedded sequence x [B, N, d]: the
    front end (gbla_project) followed by the core with its Conv1D off (the
    Conv1D already ran on X).  `store`, when given, maps each intermediate
    array to the values the layer keeps between the two halves (for example
    rounding to the storage dtype); None keeps them in double precision.
    Returns y [B, N, H, D] (rows past seq_lens[b] are NaN)."""
    pr = gbla_project(x, conv_x, w, H, D, seq_lens=seq_lens, lib=lib)
    if store is not None:
        pr = {n: store(a) for n, a in pr.items()}
    B, N = pr["q"].shape[:2]
    zeros_conv = np.zeros((3, H, D, CONV_W))  # unused with NO_CONV
    inter = {n: np.nan_to_num(pr[n], nan=0.0) for n in pr}
    return gbla_forward(inter["q"], inter["k"], inter["v"], inter["gate"],
                        inter["out_gate"], zeros_conv, norm_w, seq_lens=seq_lens,
                        eps=eps, flags=NO_CONV, lib=lib)
