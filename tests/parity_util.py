"""Helpers shared by the GPU parity tests: oracle runs on the same seeded
inputs and the comparison rules.

Comparison rules (the tolerances the GPU path must meet):
  fp32 storage: max |y - y_ref| / max(|y_ref|, 1) <= 1e-4 (relative error,
                with absolute error used where |y_ref| < 1 because elementwise
                relative error is unbounded near zero).
  bf16 storage: |y - y_ref| <= 2e-2 + ulp_bf16(y_ref) / 2 elementwise: the 2e-2
                computation budget after RMSNorm plus the rounding of the
                stored bf16 value itself (half a bf16 ulp of the true value,
                0.03125 for |y| in [8, 16), larger than 2e-2 on its own).
"""
from __future__ import annotations

import math
import os

import numpy as np
import torch

import oracle

FP32_TOL = 1e-4
BF16_ABS_TOL = 2e-2


def ulp_bf16(x: np.ndarray) -> np.ndarray:
    """Spacing of bf16 numbers at |x| (8 significant bits)."""
    ax = np.abs(x).astype(np.float64)
    ax = np.maximum(ax, np.finfo(np.float32).tiny)
    e = np.floor(np.log2(ax))
    return np.exp2(e - 7)


def to64(t: torch.Tensor) -> np.ndarray:
    return t.detach().to("cpu", torch.float64).numpy()


def compare(y_gpu: np.ndarray, y_ref: np.ndarray, dtype: str) -> dict:
    """Returns error statistics; 'ok' tells whether the rule for dtype holds."""
    assert y_gpu.shape == y_ref.shape
    d = np.abs(y_gpu - y_ref)
    finite = bool(np.all(np.isfinite(y_gpu)))
    stats = {
        "max_abs": float(d.max()) if d.size else 0.0,
        "max_rel_elem": float((d / np.maximum(np.abs(y_ref), 1e-30)).max()) if d.size else 0.0,
        "normwise": float(np.linalg.norm(d) / max(np.linalg.norm(y_ref), 1e-300)) if d.size else 0.0,
        "finite": finite,
    }
    if dtype == "fp32":
        m = float((d / np.maximum(np.abs(y_ref), 1.0)).max()) if d.size else 0.0
        stats["metric"] = m
        stats["ok"] = finite and m <= FP32_TOL
    else:
        bound = BF16_ABS_TOL + 0.5 * ulp_bf16(y_ref)
        excess = float((d - bound).max()) if d.size else -1.0
        stats["metric"] = float(d.max()) if d.size else 0.0
        stats["worst_excess"] = excess
        stats["ok"] = finite and excess <= 0.0
    return stats


def compare_prenorm(y_gpu: np.ndarray, y_ref: np.ndarray, dtype: str) -> dict:
    """Errors of an output without the gated RMSNorm (o = O).  The RMSNorm
    divides O by rms(O), so the bounds on the normalised output carry over to O
    scaled by rms(O): fp32 max |d| <= 1e-4 max|y_ref|; bf16 |d| <= 2e-2 rms(y_ref)
    + half a bf16 ulp of y_ref."""
    assert y_gpu.shape == y_ref.shape
    d = np.abs(y_gpu - y_ref)
    finite = bool(np.all(np.isfinite(y_gpu)))
    scale = float(np.sqrt(np.mean(y_ref ** 2))) if d.size else 0.0
    stats = {"max_abs": float(d.max()) if d.size else 0.0, "rms_ref": scale, "finite": finite}
    if dtype == "fp32":
        m = float(d.max() / max(np.abs(y_ref).max(), 1e-30)) if d.size else 0.0
        stats["metric"] = m
        stats["ok"] = finite and m <= FP32_TOL
    else:
        bound = BF16_ABS_TOL * scale + 0.5 * ulp_bf16(y_ref)
        excess = float((d - bound).max()) if d.size else -1.0
        stats["worst_excess"] = excess
        stats["ok"] = finite and excess <= 0.0
    return stats


def oracle_full(inp: dict, n_threads: int | None = None, flags: int = 0) -> np.ndarray:
    """Oracle over the whole [B, N, H, D] workload (padded rows stay NaN)."""
    sl = inp["seq_lens"]
    return oracle.gbla_forward(
        to64(inp["q"]), to64(inp["k"]), to64(inp["v"]), to64(inp["gate"]),
        to64(inp["out_gate"]), to64(inp["conv_w"]), to64(inp["norm_w"]),
        None if sl is None else sl.cpu().numpy(), flags=flags,
        n_threads=n_threads or os.cpu_count() or 1)


def oracle_rows(inp: dict, n_threads: int | None = None) -> list:
    """Oracle per batch row over its valid tokens: a list of [L_b, H, D] arrays.

    Each row is converted to float64 and run on its own, so a ragged workload
    padded to a long N never needs the padded [B, N, H, D] tensors in float64.
    Rows run concurrently (the C oracle releases the GIL and threads over heads)."""
    import concurrent.futures as cf

    B, N, H, _ = inp["q"].shape
    sl = inp["seq_lens"]
    lens = [N if sl is None else max(0, min(int(sl[b]), N)) for b in range(B)]
    cores = n_threads or os.cpu_count() or 1
    per_call = max(1, min(H, cores))

    def one(b):
        L = lens[b]
        cut = lambda t: to64(t[b:b + 1, :L])  # noqa: E731
        if L == 0:
            return np.zeros((0, H, inp["q"].shape[3]))
        y = oracle.gbla_forward(cut(inp["q"]), cut(inp["k"]), cut(inp["v"]), cut(inp["gate"]),
                                cut(inp["out_gate"]), to64(inp["conv_w"]), to64(inp["norm_w"]),
                                None, n_threads=per_call)
        return y[0]

    with cf.ThreadPoolExecutor(max(1, cores // per_call)) as ex:
        return list(ex.map(one, range(B)))


def log_stats(record: dict) -> None:
    """Appends one JSON line of measured errors to $GBLA_PARITY_LOG, if set."""
    path = os.environ.get("GBLA_PARITY_LOG")
    if path:
        import json
        with open(path, "a") as f:
            f.write(json.dumps(record) + "\n")


def oracle_head(inp: dict, b: int, h: int, L: int | None = None, intermediates=False):
    """Oracle for one (batch, head) over its valid rows."""
    N = inp["q"].shape[1]
    if L is None:
        sl = inp["seq_lens"]
        L = N if sl is None else int(sl[b])
        L = max(0, min(L, N))
    sl_ = slice(0, L)
    cw = inp["conv_w"]
    return oracle.gbla_head(
        to64(inp["q"][b, sl_, h]), to64(inp["k"][b, sl_, h]), to64(inp["v"][b, sl_, h]),
        to64(inp["gate"][b, sl_, h]), to64(inp["out_gate"][b, sl_, h]),
        to64(cw[0, h]), to64(cw[1, h]), to64(cw[2, h]), to64(inp["norm_w"][h]),
        intermediates=intermediates)


def valid_mask(B, N, seq_lens) -> np.ndarray:
    m = np.zeros((B, N), bool)
    for b in range(B):
        L = N if seq_lens is None else max(0, min(int(seq_lens[b]), N))
        m[b, :L] = True
    return m
