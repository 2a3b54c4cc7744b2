"""Seeded synthetic inputs for the GBLA layer core.

This module holds no arithmetic of the method: it only draws random tensors.
Both the CUDA path and the oracle consume what it produces.

The paper trains on proprietary listening histories (Yandex Music) and on the
Amazon review sets; neither is available here, so the inputs are synthetic
stand-ins with the paper's shapes: head dimension 64 (d = 1024, 16 heads),
Conv1D width 4, history lengths up to 32768 (Sec. 3, Table 5).

Recipe (per workload): a ``torch.Generator`` on the target device seeded with
the workload's seed draws, in this order, q, k, v, out_gate ``[B, N, H, D]`` and
the gate logits ``[B, N, H]`` from N(0, 1) in fp32 (then rounded to nearest
bf16 for bf16 workloads), conv taps ``[3, H, D, 4]`` from N(0, 1/4) and the
RMSNorm weight ``[H, D]`` as 1 + N(0, 0.02^2), both kept in fp32.  Ragged
workloads first draw their lengths on the host with numpy
``default_rng(seed).lognormal(ln 4096, 1.0)``, rounded and clipped to
[64, 32768]; N is the longest length and the padding rows hold N(0, 1) values
like the rest.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np
import torch

CONV_WIDTH = 4


@dataclass(frozen=True)
class Workload:
    name: str
    B: int
    H: int
    N: int              # padded length (ragged: longest sequence)
    D: int
    dtype: str          # "fp32" or "bf16"
    seed: int
    ragged: bool = False
    seq_lens: tuple = field(default=None)

    @property
    def torch_dtype(self):
        return torch.float32 if self.dtype == "fp32" else torch.bfloat16

    def lengths(self) -> list[int]:
        return list(self.seq_lens) if self.seq_lens is not None else [self.N] * self.B

    @property
    def valid_tokens(self) -> int:
        """Valid positions summed over the batch (each carries all H heads)."""
        return int(sum(self.lengths()))

    @property
    def bytes_per_token_head(self) -> int:
        """Bytes the core must move per valid (token, head): q, k, v, out_gate and
        o (D values each) plus one gate logit."""
        e = 4 if self.dtype == "fp32" else 2
        return e * (5 * self.D + 1)


def ragged_lengths(B: int, seed: int, median: int = 4096, sigma: float = 1.0,
                   lo: int = 64, hi: int = 32768) -> tuple:
    rng = np.random.default_rng(seed)
    x = rng.lognormal(mean=math.log(median), sigma=sigma, size=B)
    return tuple(int(v) for v in np.clip(np.rint(x), lo, hi))


def _ragged(name, B, H, D, seed):
    sl = ragged_lengths(B, seed)
    return Workload(name, B, H, max(sl), D, "bf16", seed, True, sl)


WORKLOADS = {
    w.name: w for w in [
        Workload("tiny_fp32_b1_h2_n256_d32", 1, 2, 256, 32, "fp32", 0),
        Workload("bf16_b8_h8_n2048_d64", 8, 8, 2048, 64, "bf16", 1),
        Workload("bf16_b4_h8_n8192_d64", 4, 8, 8192, 64, "bf16", 2),
        Workload("bf16_b2_h8_n32768_d64", 2, 8, 32768, 64, "bf16", 3),
        _ragged("bf16_ragged_b32_h8_d128", 32, 8, 128, 4),
        # a smaller ragged D = 128 batch of the same length distribution, for
        # profiler captures that must stay within a few GB of device memory
        _ragged("bf16_ragged_b8_h8_d128", 8, 8, 128, 11),
    ]
}

HEADLINE = "bf16_b2_h8_n32768_d64"


def custom(B, H, N, D, dtype="bf16", seed=0, seq_lens=None, name="custom") -> Workload:
    sl = tuple(int(x) for x in seq_lens) if seq_lens is not None else None
    return Workload(name, B, H, N, D, dtype, seed, sl is not None, sl)


def make_inputs(w: Workload, device="cpu") -> dict:
    """Draw the workload's tensors on `device` (see the module docstring)."""
    dev = torch.device(device)
    g = torch.Generator(device=dev)
    g.manual_seed(w.seed)
    shp = (w.B, w.N, w.H, w.D)

    def normal(shape, std=1.0):
        t = torch.randn(shape, generator=g, device=dev, dtype=torch.float32)
        return t.mul_(std) if std != 1.0 else t

    out = {}
    for name in ("q", "k", "v", "out_gate"):
        out[name] = normal(shp).to(w.torch_dtype)
    out["gate"] = normal((w.B, w.N, w.H)).to(w.torch_dtype)
    out["conv_w"] = normal((3, w.H, w.D, CONV_WIDTH), std=0.5)
    out["norm_w"] = normal((w.H, w.D), std=0.02).add_(1.0)
    out["seq_lens"] = (torch.tensor(w.seq_lens, dtype=torch.int32, device=dev)
                       if w.seq_lens is not None else None)
    return out


# --- layer front end (X-space Conv1D and stacked projections) ---------------
#
# Recipe: a ``torch.Generator`` on the target device seeded with `seed` draws,
# in this order, the embedded sequence x ``[B, N, d]`` from N(0, 1) (rounded to
# nearest bf16), the Conv1D taps on X ``[d, 4]`` from N(0, 1/4) (fp32), the
# stacked projection weights ``[4 H D + H, d]`` from N(0, 1/d) (rounded to
# bf16; an output then has unit variance, as with a standard linear-layer
# initialisation) and the RMSNorm weight ``[H, D]`` as 1 + N(0, 0.02^2).
# The default model width is d = H * D (512 for the 8 x 64 headline core).

def make_layer_inputs(B, N, d, H, D, seed=0, seq_lens=None, device="cpu") -> dict:
    dev = torch.device(device)
    g = torch.Generator(device=dev)
    g.manual_seed(seed)

    def normal(shape, std=1.0):
        t = torch.randn(shape, generator=g, device=dev, dtype=torch.float32)
        return t.mul_(std) if std != 1.0 else t

    out = {"x": normal((B, N, d)).to(torch.bfloat16)}
    out["conv_x"] = normal((d, CONV_WIDTH), std=0.5)
    out["w_proj"] = normal((4 * H * D + H, d), std=1.0 / math.sqrt(d)).to(torch.bfloat16)
    out["norm_w"] = normal((H, D), std=0.02).add_(1.0)
    out["seq_lens"] = (torch.tensor(list(seq_lens), dtype=torch.int32, device=dev)
                       if seq_lens is not None else None)
    return out
