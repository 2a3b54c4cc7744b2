"""The C-ABI library loads and exports every entry point include/gbla.h
declares; host-side validation rejects bad arguments before touching a GPU.
CPU only: no call here enqueues GPU work."""
import ctypes
import os
import re

import pytest

import oracle
from paper_2606_07317_gb300 import build, gbla

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADERS = [os.path.join(ROOT, "include", f) for f in os.listdir(os.path.join(ROOT, "include"))
           if f.endswith(".h")]


def _declared():
    names = set()
    for h in HEADERS:
        text = open(h).read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        names |= set(re.findall(r"\b(gbla_[a-z0-9_]+)\s*\(", text))
    return sorted(names)


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(build.LIB_PATH):
        build.build()
    return gbla.load()


def test_every_declared_symbol_is_exported(lib):
    declared = _declared()
    assert declared, "no declarations parsed"
    raw = ctypes.CDLL(build.LIB_PATH)
    missing = [n for n in declared if not hasattr(raw, n)]
    assert not missing, missing
    assert set(gbla.EXPORTED) <= set(declared)


def test_constants(lib):
    assert gbla.rms_eps() == pytest.approx(oracle.RMS_EPS, rel=1e-7)
    assert gbla.state_floats(64) == 64 * 64 + 64
    assert gbla.state_floats(0) == 0
    assert gbla.version().count(".") == 2
    for s in range(5):
        assert gbla.status_string(s)
    assert gbla.status_string(99) == "unknown status"


def _fwd(lib, ptrs, B=1, H=1, N=4, D=64, dtype=gbla.GBLA_BF16, algo=gbla.ALGO_AUTO):
    return lib.gbla_forward_ex(*ptrs, B, H, N, D, dtype, algo, None)


P16 = 0x10000  # a 16-byte aligned fake address; validation fails before any use


def test_null_pointer_rejected(lib):
    ptrs = [P16] * 9
    ptrs[7] = None  # seq_lens may be NULL
    for i in [0, 1, 2, 3, 4, 5, 6, 8]:
        bad = list(ptrs)
        bad[i] = None
        assert _fwd(lib, bad) == gbla.GBLA_ERR_INVALID_ARG, i


def test_bad_sizes_rejected(lib):
    ptrs = [P16] * 9
    assert _fwd(lib, ptrs, B=-1) == gbla.GBLA_ERR_INVALID_ARG
    assert _fwd(lib, ptrs, N=-5) == gbla.GBLA_ERR_INVALID_ARG
    assert _fwd(lib, ptrs, D=48) == gbla.GBLA_ERR_UNSUPPORTED
    assert _fwd(lib, ptrs, D=256) == gbla.GBLA_ERR_UNSUPPORTED
    assert _fwd(lib, ptrs, dtype=7) == gbla.GBLA_ERR_UNSUPPORTED
    assert _fwd(lib, ptrs, B=70000) == gbla.GBLA_ERR_INVALID_ARG


def test_empty_is_ok_without_touching_pointers(lib):
    assert _fwd(lib, [None] * 9, B=0) == gbla.GBLA_OK
    assert _fwd(lib, [None] * 9, N=0) == gbla.GBLA_OK
    assert _fwd(lib, [None] * 9, H=0) == gbla.GBLA_OK


def test_misaligned_rejected(lib):
    ptrs = [P16 + i * 0x100000 for i in range(9)]
    for i in [0, 1, 2, 3, 4, 5, 6, 8]:
        bad = list(ptrs)
        bad[i] = bad[i] + 2
        assert _fwd(lib, bad) == gbla.GBLA_ERR_INVALID_ARG, i
    bad = list(ptrs)
    bad[7] = bad[7] + 2  # seq_lens needs 4-byte alignment
    assert _fwd(lib, bad) == gbla.GBLA_ERR_INVALID_ARG


def test_overlapping_output_rejected(lib):
    ptrs = [P16 + i * 0x100000 for i in range(9)]
    ptrs[8] = ptrs[2] + 16  # o inside v
    assert _fwd(lib, ptrs) == gbla.GBLA_ERR_INVALID_ARG


def test_unknown_algo_rejected(lib):
    ptrs = [P16 + i * 0x100000 for i in range(9)]
    assert _fwd(lib, ptrs, algo=9) == gbla.GBLA_ERR_UNSUPPORTED


def test_state_and_readout_validation(lib):
    # gbla_state(k, v, gate, conv_w, seq_lens, state, B, H, N, D, dtype, algo, stream)
    assert lib.gbla_state(None, P16, P16, P16, None, P16, 1, 1, 4, 64, 1, 0, None) == \
        gbla.GBLA_ERR_INVALID_ARG
    assert lib.gbla_state(P16, P16, P16, P16, None, P16, 1, 1, 4, 40, 1, 0, None) == \
        gbla.GBLA_ERR_UNSUPPORTED
    # gbla_readout(q, og, conv_w, norm_w, seq_lens, state, o, ...)
    assert lib.gbla_readout(P16, P16, P16, P16, None, None, P16, 1, 1, 4, 64, 1, 0, None) == \
        gbla.GBLA_ERR_INVALID_ARG
    assert lib.gbla_forward_host(None, P16, P16, P16, P16, P16, P16, None, P16,
                                 1, 1, 4, 64, 1, None) == gbla.GBLA_ERR_INVALID_ARG


def test_backward_from_state_validates_saved_state(lib):
    # q k v gate out_gate conv_w norm_w seq_lens state stats dy dq dk dv dgate dout_gate
    # dconv_w dnorm_w: distinct aligned fake addresses, seq_lens NULL
    base = [P16 + i * 0x100000 for i in range(18)]
    base[7] = None
    for i, bad in [(8, None), (8, base[8] + 4), (9, None), (9, base[9] + 8)]:
        ptrs = list(base)
        ptrs[i] = bad
        st = lib.gbla_backward_from_state(*ptrs, 1, 1, 4, 64, gbla.GBLA_BF16, None)
        assert st == gbla.GBLA_ERR_INVALID_ARG, (i, bad)


def test_backward_saved_state_arguments_checked_on_host():
    """The binding rejects a saved state without its statistics (or the reverse),
    with an ablation, or of the wrong shape or dtype, before calling the library."""
    import torch
    q = torch.zeros((1, 8, 2, 64), dtype=torch.bfloat16)
    g = torch.zeros((1, 8, 2), dtype=torch.bfloat16)
    cw, nw = torch.zeros((3, 2, 64, 4)), torch.zeros((2, 64))
    state, stats = torch.zeros((1, 2, 64 * 64 + 64)), torch.zeros((1, 2, 2))
    args = (q, q, q, g, q, cw, nw, None, q)
    for kw in (dict(state=state), dict(stats=stats),
               dict(flags=gbla.FLAG_NO_GATE, state=state, stats=stats),
               dict(state=state[:, :1], stats=stats),
               dict(state=state.double(), stats=stats),
               dict(state=state, stats=stats[..., :1])):
        with pytest.raises(ValueError):
            gbla.backward(*args, **kw)
