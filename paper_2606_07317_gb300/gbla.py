"""Thin ctypes binding of libgbla (the C ABI declared in include/gbla.h).

Argument marshalling only: every step of the GBLA core runs in the library's
CUDA kernels.  Tensors are torch tensors; device calls take CUDA tensors and
enqueue on the current torch stream (or the stream given).  There is no CPU
fallback: if the library is missing or fails to load, calls raise.
"""
from __future__ import annotations

import ctypes
import os
import threading

import torch

from . import build as _build

GBLA_OK, GBLA_ERR_INVALID_ARG, GBLA_ERR_UNSUPPORTED, GBLA_ERR_ALLOC, GBLA_ERR_CUDA = range(5)
GBLA_FP32, GBLA_BF16 = 0, 1
ALGO_AUTO, ALGO_SIMT, ALGO_TC = 0, 1, 2
# ablation flags (gbla_flags): identity Conv1D, uniform key gate, no gated RMSNorm
FLAG_NO_CONV, FLAG_NO_GATE, FLAG_NO_NORM = 1, 2, 4
FLAG_BLA = FLAG_NO_CONV | FLAG_NO_GATE | FLAG_NO_NORM
CONV_WIDTH = 4

EXPORTED = ["gbla_forward", "gbla_forward_ex", "gbla_forward_variant", "gbla_forward_f32out",
            "gbla_backward", "gbla_backward_variant", "gbla_backward_from_state",
            "gbla_state", "gbla_state_stats", "gbla_combine_states",
            "gbla_readout",
            "gbla_forward_host", "gbla_state_floats", "gbla_rms_eps",
            "gbla_status_string", "gbla_version", "gbla_release", "gbla_launch_count",
            "gbla_state_static_scratch", "gbla_device_error", "gbla_last_cuda_error",
            "gbla_project", "gbla_layer_forward", "gbla_attention_forward"]

_lock = threading.Lock()
_lib = None

_vp = ctypes.c_void_p
_i = ctypes.c_int


class GblaError(RuntimeError):
    def __init__(self, status: int, fn: str):
        self.status = status
        msg = f"{fn}: {status_string(status)} (status {status})"
        if status == GBLA_ERR_CUDA:
            msg += f": {load().gbla_last_cuda_error().decode()}"
        super().__init__(msg)


def lib_path() -> str:
    return _build.LIB_PATH


def load(path: str | None = None):
    """Load libgbla.so (it must have been built; see __graft_entry__.build())."""
    global _lib
    with _lock:
        if _lib is not None and path is None:
            return _lib
        p = path or lib_path()
        if not os.path.exists(p):
            raise RuntimeError(f"CUDA library not built: {p} is missing "
                               "(run `python -c 'import __graft_entry__ as g; g.build()'`)")
        lib = ctypes.CDLL(p)
        fwd = [_vp] * 9 + [_i] * 5
        lib.gbla_forward.argtypes = fwd + [_vp]
        lib.gbla_forward.restype = _i
        lib.gbla_forward_ex.argtypes = fwd + [_i, _vp]
        lib.gbla_forward_ex.restype = _i
        lib.gbla_forward_variant.argtypes = fwd + [_i, ctypes.c_uint32, _vp]
        lib.gbla_forward_variant.restype = _i
        lib.gbla_forward_f32out.argtypes = fwd + [_i, _vp]
        lib.gbla_forward_f32out.restype = _i
        lib.gbla_backward.argtypes = [_vp] * 16 + [_i] * 5 + [_vp]
        lib.gbla_backward.restype = _i
        lib.gbla_backward_variant.argtypes = [_vp] * 16 + [_i] * 5 + [ctypes.c_uint32, _vp]
        lib.gbla_backward_variant.restype = _i
        lib.gbla_backward_from_state.argtypes = [_vp] * 18 + [_i] * 5 + [_vp]
        lib.gbla_backward_from_state.restype = _i
        lib.gbla_project.argtypes = [_vp] * 9 + [_i] * 6 + [_vp]
        lib.gbla_project.restype = _i
        lib.gbla_layer_forward.argtypes = [_vp] * 6 + [_i] * 6 + [_vp]
        lib.gbla_layer_forward.restype = _i
        lib.gbla_attention_forward.argtypes = [_vp] * 5 + [_i] * 5 + [_vp]
        lib.gbla_attention_forward.restype = _i
        lib.gbla_forward_host.argtypes = fwd + [_vp]
        lib.gbla_forward_host.restype = _i
        lib.gbla_state.argtypes = [_vp] * 6 + [_i] * 6 + [_vp]
        lib.gbla_state.restype = _i
        lib.gbla_state_stats.argtypes = [_vp] * 7 + [_i] * 6 + [_vp]
        lib.gbla_state_stats.restype = _i
        lib.gbla_combine_states.argtypes = [_vp, _vp, _i, _vp, _vp, _i, _i, _i, _vp]
        lib.gbla_combine_states.restype = _i
        lib.gbla_readout.argtypes = [_vp] * 7 + [_i] * 6 + [_vp]
        lib.gbla_readout.restype = _i
        lib.gbla_state_static_scratch.argtypes = [_vp] * 6 + [_i] * 5 + [_vp]
        lib.gbla_state_static_scratch.restype = _i
        lib.gbla_state_floats.argtypes = [_i]
        lib.gbla_state_floats.restype = ctypes.c_size_t
        lib.gbla_rms_eps.argtypes = []
        lib.gbla_rms_eps.restype = ctypes.c_float
        lib.gbla_status_string.argtypes = [_i]
        lib.gbla_status_string.restype = ctypes.c_char_p
        lib.gbla_version.argtypes = []
        lib.gbla_version.restype = ctypes.c_char_p
        lib.gbla_release.argtypes = []
        lib.gbla_release.restype = None
        lib.gbla_last_cuda_error.argtypes = []
        lib.gbla_last_cuda_error.restype = ctypes.c_char_p
        lib.gbla_device_error.argtypes = [_i]
        lib.gbla_device_error.restype = ctypes.c_uint32
        lib.gbla_launch_count.argtypes = []
        lib.gbla_launch_count.restype = ctypes.c_uint64
        if path is None:
            _lib = lib
        return lib


def status_string(status: int) -> str:
    return load().gbla_status_string(int(status)).decode()


def rms_eps() -> float:
    return float(load().gbla_rms_eps())


def version() -> str:
    return load().gbla_version().decode()


def launch_count() -> int:
    """Kernels the library has enqueued so far (all devices, all threads)."""
    return int(load().gbla_launch_count())


def device_error(reset: bool = False) -> int:
    """Error bits left by a tensor-core kernel whose bounded wait ran out (0 = none)."""
    return int(load().gbla_device_error(1 if reset else 0))


def state_floats(D: int) -> int:
    return int(load().gbla_state_floats(int(D)))


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.float32:
        return GBLA_FP32
    if t.dtype == torch.bfloat16:
        return GBLA_BF16
    raise TypeError(f"unsupported dtype {t.dtype}")


def _ptr(t):
    if t is None:
        return None
    return t.data_ptr() or None


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return _vp(stream.cuda_stream)


def _check(status: int, fn: str):
    if status != GBLA_OK:
        raise GblaError(status, fn)


def _bhnd(q: torch.Tensor):
    if q.dim() != 4:
        raise ValueError("q must be [B, N, H, D]")
    B, N, H, D = q.shape
    return B, H, N, D


def forward(q, k, v, gate, out_gate, conv_w, norm_w, seq_lens=None, out=None,
            algo: int = ALGO_AUTO, stream=None, flags: int = 0) -> torch.Tensor:
    """o = GBLA core forward; tensors on one CUDA device, layouts of include/gbla.h.
    `flags` (FLAG_*) selects an ablation (gbla_forward_variant); 0 is the full core."""
    B, H, N, D = _bhnd(q)
    if out is None:
        out = torch.empty_like(q)
    if flags:
        st = load().gbla_forward_variant(
            _ptr(q), _ptr(k), _ptr(v), _ptr(gate), _ptr(out_gate), _ptr(conv_w),
            _ptr(norm_w), _ptr(seq_lens), _ptr(out), B, H, N, D, _dtype_code(q), int(algo),
            int(flags), _stream(stream))
        _check(st, "gbla_forward_variant")
        return out
    st = load().gbla_forward_ex(
        _ptr(q), _ptr(k), _ptr(v), _ptr(gate), _ptr(out_gate), _ptr(conv_w),
        _ptr(norm_w), _ptr(seq_lens), _ptr(out), B, H, N, D, _dtype_code(q), int(algo),
        _stream(stream))
    _check(st, "gbla_forward_ex")
    return out


def attention(q, k, v, seq_lens=None, out=None, stream=None) -> torch.Tensor:
    """Bidirectional softmax attention of Sec. 2 (gbla_attention_forward): q, k, v,
    out [B, N, H, D] bf16 (D = 64); rows past seq_lens are not written."""
    B, H, N, D = _bhnd(q)
    if out is None:
        out = torch.empty_like(q)
    st = load().gbla_attention_forward(_ptr(q), _ptr(k), _ptr(v), _ptr(seq_lens), _ptr(out),
                                       B, H, N, D, _dtype_code(q), _stream(stream))
    _check(st, "gbla_attention_forward")
    return out


def forward_f32out(q, k, v, gate, out_gate, conv_w, norm_w, seq_lens=None, out=None,
                   algo: int = ALGO_AUTO, stream=None) -> torch.Tensor:
    """Debug variant of forward (gbla_forward_f32out): the same kernels and arithmetic,
    with o stored in fp32 before the rounding to the input dtype."""
    B, H, N, D = _bhnd(q)
    if out is None:
        out = torch.empty(q.shape, dtype=torch.float32, device=q.device)
    st = load().gbla_forward_f32out(
        _ptr(q), _ptr(k), _ptr(v), _ptr(gate), _ptr(out_gate), _ptr(conv_w),
        _ptr(norm_w), _ptr(seq_lens), _ptr(out), B, H, N, D, _dtype_code(q), int(algo),
        _stream(stream))
    _check(st, "gbla_forward_f32out")
    return out


def backward(q, k, v, gate, out_gate, conv_w, norm_w, seq_lens, dy, stream=None,
             flags: int = 0, state=None, stats=None) -> dict:
    """Gradients of sum(dy * o) (gbla_backward): dq, dk, dv, dout_gate like q; dgate like
    gate; dconv_w [3, H, D, W] and dnorm_w [H, D] fp32.  Rows past seq_lens are 0.
    `flags` (FLAG_*) selects an ablation (gbla_backward_variant); 0 is the full core.
    `state` and `stats`, as state_stats returned them for this forward, skip the state
    pass (gbla_backward_from_state; full core only)."""
    B, H, N, D = _bhnd(q)
    if (state is None) != (stats is None):
        raise ValueError("state and stats go together")
    if state is not None and flags:
        raise ValueError("a saved state serves the full core only (flags 0)")
    g = dict(dq=torch.empty_like(q), dk=torch.empty_like(q), dv=torch.empty_like(q),
             dgate=torch.empty_like(gate), dout_gate=torch.empty_like(q),
             dconv_w=torch.empty_like(conv_w, dtype=torch.float32),
             dnorm_w=torch.empty_like(norm_w, dtype=torch.float32))
    args = (_ptr(q), _ptr(k), _ptr(v), _ptr(gate), _ptr(out_gate), _ptr(conv_w), _ptr(norm_w),
            _ptr(seq_lens), _ptr(dy), _ptr(g["dq"]), _ptr(g["dk"]), _ptr(g["dv"]),
            _ptr(g["dgate"]), _ptr(g["dout_gate"]), _ptr(g["dconv_w"]), _ptr(g["dnorm_w"]),
            B, H, N, D, _dtype_code(q))
    if state is not None:
        if (state.dtype != torch.float32 or stats.dtype != torch.float32
                or tuple(state.shape) != (B, H, D * D + D) or tuple(stats.shape) != (B, H, 2)
                or not state.is_contiguous() or not stats.is_contiguous()):
            raise ValueError("state must be [B, H, D*D + D] and stats [B, H, 2], contiguous fp32")
        a = list(args)
        a[8:8] = [_ptr(state), _ptr(stats)]  # after seq_lens
        st = load().gbla_backward_from_state(*a, _stream(stream))
        _check(st, "gbla_backward_from_state")
    elif flags:
        st = load().gbla_backward_variant(*args, int(flags), _stream(stream))
        _check(st, "gbla_backward_variant")
    else:
        st = load().gbla_backward(*args, _stream(stream))
        _check(st, "gbla_backward")
    return g


def project(x, conv_x, w_proj, H, D, seq_lens=None, out=None, stream=None) -> dict:
    """Layer front end (gbla_project): X~ = Conv1D(x) over the d channels of x [B, N, d],
    then the stacked projections w_proj [4 H D + H, d] (rows W_Q, W_K, W_V, W_R per head
    and dim, then w_g per head).  Returns q, k, v, out_gate [B, N, H, D] and gate
    [B, N, H] (rows past seq_lens are not written; `out` may supply the five tensors)."""
    B, N, d = x.shape
    if out is None:
        out = {n: x.new_empty((B, N, H, D)) for n in ("q", "k", "v", "out_gate")}
        out["gate"] = x.new_empty((B, N, H))
    st = load().gbla_project(
        _ptr(x), _ptr(conv_x), _ptr(w_proj), _ptr(seq_lens), _ptr(out["q"]), _ptr(out["k"]),
        _ptr(out["v"]), _ptr(out["out_gate"]), _ptr(out["gate"]), B, N, d, H, D,
        _dtype_code(x), _stream(stream))
    _check(st, "gbla_project")
    return out


def layer_forward(x, conv_x, w_proj, norm_w, H, D, seq_lens=None, out=None,
                  stream=None) -> torch.Tensor:
    """Whole GBLA layer from x [B, N, d] (gbla_layer_forward): front end, then the core
    with its Conv1D off.  Returns o [B, N, H, D]."""
    B, N, d = x.shape
    if out is None:
        out = x.new_empty((B, N, H, D))
    st = load().gbla_layer_forward(
        _ptr(x), _ptr(conv_x), _ptr(w_proj), _ptr(norm_w), _ptr(seq_lens), _ptr(out),
        B, N, d, H, D, _dtype_code(x), _stream(stream))
    _check(st, "gbla_layer_forward")
    return out


def forward_default(q, k, v, gate, out_gate, conv_w, norm_w, seq_lens, out, stream=None):
    """Direct call of gbla_forward (the AUTO entry point)."""
    B, H, N, D = _bhnd(q)
    st = load().gbla_forward(
        _ptr(q), _ptr(k), _ptr(v), _ptr(gate), _ptr(out_gate), _ptr(conv_w),
        _ptr(norm_w), _ptr(seq_lens), _ptr(out), B, H, N, D, _dtype_code(q),
        _stream(stream))
    _check(st, "gbla_forward")
    return out


def state(k, v, gate, conv_w, seq_lens=None, out=None, algo: int = ALGO_AUTO,
          stream=None) -> torch.Tensor:
    """[B, H, D*D + D] fp32: S (row-major) then z per (batch, head)."""
    B, H, N, D = _bhnd(k)
    if out is None:
        out = torch.empty((B, H, D * D + D), dtype=torch.float32, device=k.device)
    st = load().gbla_state(_ptr(k), _ptr(v), _ptr(gate), _ptr(conv_w), _ptr(seq_lens),
                           _ptr(out), B, H, N, D, _dtype_code(k), int(algo),
                           _stream(stream))
    _check(st, "gbla_state")
    return out


def state_stats(k, v, gate, conv_w, seq_lens=None, algo: int = ALGO_AUTO, stream=None):
    """gbla_state_stats: (state [B, H, D*D + D], stats [B, H, 2]) fp32, stats = (max gate
    logit, sum of exp(logit - max)) over each sequence's valid positions."""
    B, H, N, D = _bhnd(k)
    out = torch.empty((B, H, D * D + D), dtype=torch.float32, device=k.device)
    stats = torch.empty((B, H, 2), dtype=torch.float32, device=k.device)
    st = load().gbla_state_stats(_ptr(k), _ptr(v), _ptr(gate), _ptr(conv_w), _ptr(seq_lens),
                                 _ptr(out), _ptr(stats), B, H, N, D, _dtype_code(k), int(algo),
                                 _stream(stream))
    _check(st, "gbla_state_stats")
    return out, stats


def combine_states(states, stats, stream=None):
    """gbla_combine_states: states [P, B, H, D*D + D] and stats [P, B, H, 2] (fp32, one
    CUDA device) of P disjoint token segments -> (state, stats) of the whole sequences."""
    P, B, H, F = states.shape
    D = int(round((F + 0.25) ** 0.5 - 0.5))
    if D * D + D != F or tuple(stats.shape) != (P, B, H, 2):
        raise ValueError("states must be [P, B, H, D*D + D] and stats [P, B, H, 2]")
    states, stats = states.contiguous(), stats.contiguous()
    out = torch.empty((B, H, F), dtype=torch.float32, device=states.device)
    out_stats = torch.empty((B, H, 2), dtype=torch.float32, device=states.device)
    st = load().gbla_combine_states(_ptr(states), _ptr(stats), P, _ptr(out), _ptr(out_stats),
                                    B, H, D, _stream(stream))
    _check(st, "gbla_combine_states")
    return out, out_stats


def readout(q, out_gate, conv_w, norm_w, state_t, seq_lens=None, out=None,
            algo: int = ALGO_AUTO, stream=None) -> torch.Tensor:
    B, H, N, D = _bhnd(q)
    if out is None:
        out = torch.empty_like(q)
    st = load().gbla_readout(_ptr(q), _ptr(out_gate), _ptr(conv_w), _ptr(norm_w),
                             _ptr(seq_lens), _ptr(state_t), _ptr(out), B, H, N, D,
                             _dtype_code(q), int(algo), _stream(stream))
    _check(st, "gbla_readout")
    return out


def forward_host(q, k, v, gate, out_gate, conv_w, norm_w, seq_lens=None, out=None,
                 stream=None) -> torch.Tensor:
    """Host-memory entry point: CPU tensors (pinned for full copy speed) in and out."""
    B, H, N, D = _bhnd(q)
    if out is None:
        out = torch.empty_like(q)
    st = load().gbla_forward_host(
        _ptr(q), _ptr(k), _ptr(v), _ptr(gate), _ptr(out_gate), _ptr(conv_w),
        _ptr(norm_w), _ptr(seq_lens), _ptr(out), B, H, N, D, _dtype_code(q),
        _stream(stream))
    _check(st, "gbla_forward_host")
    return out


def state_static_scratch(k, v, gate, conv_w, seq_lens=None, out=None,
                         stream=None) -> torch.Tensor:
    """gbla_state without any GPU allocation: for callers that cannot allocate
    device memory (its partial sums live in a fixed array inside the library;
    see include/gbla.h for the size limit and the rule against overlapping
    calls)."""
    B, H, N, D = _bhnd(k)
    if out is None:
        out = torch.empty((B, H, D * D + D), dtype=torch.float32, device=k.device)
    st = load().gbla_state_static_scratch(_ptr(k), _ptr(v), _ptr(gate), _ptr(conv_w),
                                          _ptr(seq_lens), _ptr(out), B, H, N, D,
                                          _dtype_code(k), _stream(stream))
    _check(st, "gbla_state_static_scratch")
    return out
