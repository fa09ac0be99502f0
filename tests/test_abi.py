"""The C-ABI library builds, loads and exports every declared symbol; host-side
validation rejects bad arguments before any launch (CPU only, no kernel runs)."""

import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADERS = [os.path.join(ROOT, "include", h) for h in ("bcmt.h", "bcmt_testing.h")]


@pytest.fixture(scope="module")
def C():
    from paper_2608_13578_gb300 import build
    build.build()
    from paper_2608_13578_gb300 import bcmt
    return bcmt


def declared_functions():
    names = set()
    for h in HEADERS:
        src = open(h).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        for m in re.finditer(r"\b(bcmt_[a-z_]+)\s*\(", src):
            names.add(m.group(1))
    return sorted(names)


def test_every_declared_symbol_is_exported(C):
    names = declared_functions()
    assert "bcmt_forward" in names and "bcmt_backward" in names
    lib = ctypes.CDLL(C.LIB_PATH)
    for n in names:
        assert hasattr(lib, n), n
    assert set(names) == set(C.EXPORTED)


def test_workspace_sizes_host_only(C):
    p = C.make_params(8, 1024, 512, 8, 64, "bf16")
    ws, sc = C.bcmt_workspace_size(p), C.bcmt_scratch_size(p)
    n = 8 * 1024
    # at least Q/K/V, Concat(heads), H and G in bf16
    assert ws >= n * 512 * 2 * 6
    assert sc >= n * 512 * 2 * 6
    ph = C.make_params(8, 1024, 512, 8, 64, "bf16", flags=C.BCMT_FLAG_HONLY)
    assert C.bcmt_workspace_size(ph) < ws
    bad = C.make_params(8, 1024, 500, 8, 64, "bf16")
    assert C.bcmt_workspace_size(bad) == 0


@pytest.mark.parametrize("field,value,code", [
    ("D", 96, "BCMT_ERR_SHAPE"),       # not a multiple of 64
    ("H", 3, "BCMT_ERR_SHAPE"),        # D % H != 0
    ("H", 1, "BCMT_ERR_SHAPE"),        # head width 128 < ... D=256 -> 256 > 128
    ("L", 0, "BCMT_ERR_SHAPE"),
    ("L", 4096, "BCMT_ERR_UNSUPPORTED"),
    ("T", 0, "BCMT_ERR_SHAPE"),
    ("B", 0, "BCMT_ERR_SHAPE"),
    ("dtype", 7, "BCMT_ERR_ARG"),
    ("flags", 64, "BCMT_ERR_ARG"),
])
def test_forward_rejects_bad_params(C, field, value, code):
    p = C.make_params(2, 64, 256, 4, 16, "bf16")
    setattr(p, field, value)
    dummy = 1 << 20  # never dereferenced: validation fails first
    with pytest.raises(C.BCMTError) as e:
        C.bcmt_forward(p, dummy, None, None, None, dummy, dummy, dummy, dummy, dummy, dummy,
                       dummy, dummy, 0)
    assert e.value.code == getattr(C, code), C.bcmt_last_error()


def test_forward_rejects_null_and_misaligned(C):
    p = C.make_params(2, 64, 256, 4, 16, "bf16")
    a = 1 << 20
    with pytest.raises(C.BCMTError) as e:
        C.bcmt_forward(p, None, None, None, None, a, a, a, a, a, a, a, a, 0)
    assert e.value.code == C.BCMT_ERR_ARG and "x" in C.bcmt_last_error()
    with pytest.raises(C.BCMTError) as e:
        C.bcmt_forward(p, a + 8, None, None, None, a, a, a, a, a, a, a, a, 0)
    assert e.value.code == C.BCMT_ERR_ALIGN
    # the Q/K/V entry needs q, k, v
    pq = C.make_params(2, 64, 256, 4, 16, "bf16", input_is_x=False)
    with pytest.raises(C.BCMTError) as e:
        C.bcmt_forward(pq, a, None, a, a, None, a, a, a, a, a, a, a, 0)
    assert e.value.code == C.BCMT_ERR_ARG and "q" in C.bcmt_last_error()


def test_backward_rejects_missing_gradients(C):
    p = C.make_params(2, 64, 256, 4, 16, "fp32")
    a = 1 << 20
    with pytest.raises(C.BCMTError) as e:
        C.bcmt_backward(p, a, a, None, None, a, a, a, a, a, a, a, a, a, None, None, a, a, a, a,
                        None, 0)
    assert e.value.code == C.BCMT_ERR_ARG and "dw_g" in C.bcmt_last_error()
