"""Python binding of the BCMT CUDA library (``include/bcmt.h``).

Argument marshalling only: every step of the mixer runs in the library's CUDA
kernels.  The functions below carry the C names; tensors are passed as device
pointers (``torch.Tensor`` arguments are converted with ``data_ptr()``, plain
ints are taken as raw device addresses, ``None`` is NULL) and the stream as a
``torch.cuda.Stream`` or a raw ``cudaStream_t`` int.  PyTorch is used only for
device memory and streams.

Importing this module loads ``_lib/libbcmt.so`` and raises if it is missing:
there is no CPU fallback.
"""

from __future__ import annotations

import ctypes
import os
from typing import Dict, Optional, Tuple

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "_lib", "libbcmt.so")

BCMT_OK, BCMT_ERR_ARG, BCMT_ERR_SHAPE, BCMT_ERR_ALIGN, BCMT_ERR_CUDA, BCMT_ERR_TIMEOUT, \
    BCMT_ERR_UNSUPPORTED = range(7)
BCMT_F32, BCMT_BF16 = 0, 1
BCMT_FLAG_HONLY, BCMT_FLAG_CHECK, BCMT_FLAG_PROFILE = 1, 2, 4

STATUS_NAMES = {0: "BCMT_OK", 1: "BCMT_ERR_ARG", 2: "BCMT_ERR_SHAPE", 3: "BCMT_ERR_ALIGN",
                4: "BCMT_ERR_CUDA", 5: "BCMT_ERR_TIMEOUT", 6: "BCMT_ERR_UNSUPPORTED"}


class BCMTError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"{STATUS_NAMES.get(code, code)}: {msg}")
        self.code = code


class bcmt_params(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int), ("T", ctypes.c_int), ("D", ctypes.c_int),
                ("H", ctypes.c_int), ("L", ctypes.c_int), ("dtype", ctypes.c_int),
                ("input_is_x", ctypes.c_int), ("flags", ctypes.c_uint)]


def make_params(B, T, D, H, L, dtype="bf16", input_is_x=True, flags=0) -> bcmt_params:
    dt = {"fp32": BCMT_F32, "bf16": BCMT_BF16, BCMT_F32: BCMT_F32, BCMT_BF16: BCMT_BF16}[dtype]
    return bcmt_params(B, T, D, H, L, dt, 1 if input_is_x else 0, flags)


_VP = ctypes.c_void_p
_P = ctypes.POINTER(bcmt_params)


def _load():
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(
            f"{LIB_PATH} is missing: build it with `python -m paper_2608_13578_gb300.build`")
    lib = ctypes.CDLL(LIB_PATH)
    lib.bcmt_workspace_size.argtypes = [_P]
    lib.bcmt_workspace_size.restype = ctypes.c_size_t
    lib.bcmt_scratch_size.argtypes = [_P]
    lib.bcmt_scratch_size.restype = ctypes.c_size_t
    lib.bcmt_forward.argtypes = [_P] + [_VP] * 13
    lib.bcmt_forward.restype = ctypes.c_int
    lib.bcmt_backward.argtypes = [_P] + [_VP] * 21
    lib.bcmt_backward.restype = ctypes.c_int
    lib.bcmt_device_status.argtypes = [_VP]
    lib.bcmt_device_status.restype = ctypes.c_int
    lib.bcmt_last_error.argtypes = []
    lib.bcmt_last_error.restype = ctypes.c_char_p
    lib.bcmt_profile_read.argtypes = [ctypes.POINTER(ctypes.c_char_p), ctypes.POINTER(ctypes.c_int),
                                      ctypes.POINTER(ctypes.c_double), ctypes.c_int]
    lib.bcmt_profile_read.restype = ctypes.c_int
    lib.bcmt_profile_reset.argtypes = []
    lib.bcmt_profile_reset.restype = None
    lib.bcmt_decode_state_size.argtypes = [_P]
    lib.bcmt_decode_state_size.restype = ctypes.c_size_t
    lib.bcmt_decode_reset.argtypes = [_P, _VP, _VP]
    lib.bcmt_decode_reset.restype = ctypes.c_int
    lib.bcmt_decode_step.argtypes = [_P, _VP, ctypes.c_long] + [_VP] * 9
    lib.bcmt_decode_step.restype = ctypes.c_int
    lib.bcmt_attention_backward_noalloc.argtypes = [_P, _VP, _VP, _VP, ctypes.c_long, _VP, _VP,
                                                    _VP, _VP, _VP, _VP, ctypes.c_long, _VP]
    lib.bcmt_attention_backward_noalloc.restype = ctypes.c_int
    lib.bcmt_test_set_tensor_cores.argtypes = [ctypes.c_int, ctypes.c_int]
    lib.bcmt_test_set_tensor_cores.restype = ctypes.c_int
    lib.bcmt_test_gemm.argtypes = [ctypes.c_int] * 6 + [_VP, ctypes.c_long, ctypes.c_long, _VP,
                                                        ctypes.c_long, ctypes.c_long, _VP,
                                                        ctypes.c_long, ctypes.c_int, _VP]
    lib.bcmt_test_gemm.restype = ctypes.c_int
    _gi = [ctypes.c_int] * 3 + [_VP, ctypes.c_long, _VP, ctypes.c_long, _VP, ctypes.c_int]
    lib.bcmt_test_gemm_group.argtypes = ([ctypes.c_int] * 3 + [_VP, ctypes.c_long, _VP, ctypes.c_long,
                                                               _VP] + _gi + _gi + [_VP])
    lib.bcmt_test_gemm_group.restype = ctypes.c_int
    lib.bcmt_test_attn.argtypes = [ctypes.c_int, ctypes.c_int, _P, _VP, _VP, _VP, ctypes.c_long,
                                   _VP, _VP, _VP, _VP, _VP, _VP, _VP, ctypes.c_long, _VP]
    lib.bcmt_test_attn.restype = ctypes.c_int
    lib.bcmt_test_wait_expiry.argtypes = [ctypes.c_longlong, _VP]
    lib.bcmt_test_wait_expiry.restype = ctypes.c_int
    return lib


LIB = _load()

# Symbols include/bcmt.h and include/bcmt_testing.h declare.
EXPORTED = ("bcmt_workspace_size", "bcmt_scratch_size", "bcmt_forward", "bcmt_backward",
            "bcmt_device_status", "bcmt_last_error", "bcmt_profile_read", "bcmt_profile_reset",
            "bcmt_attention_backward_noalloc",
            "bcmt_decode_state_size", "bcmt_decode_reset", "bcmt_decode_step",
            "bcmt_test_set_tensor_cores", "bcmt_test_gemm", "bcmt_test_gemm_group", "bcmt_test_attn",
            "bcmt_test_wait_expiry")


def _ptr(t) -> Optional[int]:
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream(s) -> Optional[int]:
    if s is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(s, int):
        return s
    return s.cuda_stream


def _check(code: int):
    if code != BCMT_OK:
        raise BCMTError(code, bcmt_last_error())


def bcmt_last_error() -> str:
    return LIB.bcmt_last_error().decode()


def bcmt_workspace_size(p: bcmt_params) -> int:
    return LIB.bcmt_workspace_size(ctypes.byref(p))


def bcmt_scratch_size(p: bcmt_params) -> int:
    return LIB.bcmt_scratch_size(ctypes.byref(p))


def bcmt_forward(p: bcmt_params, x, q, k, v, w_qkv, w_o, w_p, w_m, w_g, decay, y, workspace,
                 stream=None) -> None:
    _check(LIB.bcmt_forward(ctypes.byref(p), _ptr(x), _ptr(q), _ptr(k), _ptr(v), _ptr(w_qkv),
                            _ptr(w_o), _ptr(w_p), _ptr(w_m), _ptr(w_g), _ptr(decay), _ptr(y),
                            _ptr(workspace), _stream(stream)))


def bcmt_backward(p: bcmt_params, dy, x_or_q, k, v, w_qkv, w_o, w_p, w_m, w_g, decay, workspace,
                  scratch, dx_or_dq, dk, dv, dw_qkv, dw_o, dw_p, dw_m, dw_g, stream=None,
                  d_decay=None) -> None:
    """d_decay (fp32 [D], optional): gradient for a learned per-channel decay."""
    _check(LIB.bcmt_backward(ctypes.byref(p), _ptr(dy), _ptr(x_or_q), _ptr(k), _ptr(v),
                             _ptr(w_qkv), _ptr(w_o), _ptr(w_p), _ptr(w_m), _ptr(w_g), _ptr(decay),
                             _ptr(workspace), _ptr(scratch), _ptr(dx_or_dq), _ptr(dk), _ptr(dv),
                             _ptr(dw_qkv), _ptr(dw_o), _ptr(dw_p), _ptr(dw_m), _ptr(dw_g),
                             _ptr(d_decay), _stream(stream)))


def bcmt_device_status(stream=None) -> None:
    _check(LIB.bcmt_device_status(_stream(stream)))


def bcmt_decode_state_size(p: bcmt_params) -> int:
    return LIB.bcmt_decode_state_size(ctypes.byref(p))


def bcmt_decode_reset(p: bcmt_params, state, stream=None) -> None:
    _check(LIB.bcmt_decode_reset(ctypes.byref(p), _ptr(state), _stream(stream)))


def bcmt_decode_step(p: bcmt_params, state, pos: int, x_t, w_qkv, w_o, w_p, w_m, w_g, decay, y_t,
                     stream=None) -> None:
    _check(LIB.bcmt_decode_step(ctypes.byref(p), _ptr(state), pos, _ptr(x_t), _ptr(w_qkv),
                                _ptr(w_o), _ptr(w_p), _ptr(w_m), _ptr(w_g), _ptr(decay),
                                _ptr(y_t), _stream(stream)))


def bcmt_attention_backward_noalloc(p: bcmt_params, q, k, v, ld, o, lse, dO, dq, dk, dv, ld_d,
                                    stream=None) -> None:
    """Attention backward whose scratch is a device array inside the library
    (for callers that cannot allocate device memory); see include/bcmt.h."""
    _check(LIB.bcmt_attention_backward_noalloc(ctypes.byref(p), _ptr(q), _ptr(k), _ptr(v), ld,
                                               _ptr(o), _ptr(lse), _ptr(dO), _ptr(dq), _ptr(dk),
                                               _ptr(dv), ld_d, _stream(stream)))


def bcmt_profile_reset() -> None:
    LIB.bcmt_profile_reset()


def bcmt_profile_read(cap: int = 64) -> Dict[str, Tuple[int, float]]:
    names = (ctypes.c_char_p * cap)()
    cnt = (ctypes.c_int * cap)()
    ms = (ctypes.c_double * cap)()
    n = LIB.bcmt_profile_read(names, cnt, ms, cap)
    if n < 0:
        raise BCMTError(BCMT_ERR_CUDA, "profile read failed")
    return {names[i].decode(): (cnt[i], ms[i]) for i in range(min(n, cap))}


def bcmt_test_set_tensor_cores(gemm_on: bool, attn_on: bool) -> int:
    return LIB.bcmt_test_set_tensor_cores(int(gemm_on), int(attn_on))


def bcmt_test_gemm(impl, dtype, dtype_out, M, N, K, A, sam, sak, B, sbk, sbn, C, ldc, splits=1,
                   stream=None) -> int:
    r = LIB.bcmt_test_gemm(impl, dtype, dtype_out, M, N, K, _ptr(A), sam, sak, _ptr(B), sbk, sbn,
                           _ptr(C), ldc, splits, _stream(stream))
    if r < 0:
        raise BCMTError(BCMT_ERR_CUDA, bcmt_last_error())
    return r


def bcmt_test_gemm_group(M0, N0, K0, A0, lda0, B0t, ldb0t, C0, M1, N1, K1, A1t, lda1t, B1, ldb1,
                         part1, splits1, M2=0, N2=0, K2=0, A2t=None, lda2t=0, B2=None, ldb2=0,
                         part2=None, splits2=1, stream=None) -> int:
    r = LIB.bcmt_test_gemm_group(M0, N0, K0, _ptr(A0), lda0, _ptr(B0t), ldb0t, _ptr(C0), M1, N1, K1,
                                 _ptr(A1t), lda1t, _ptr(B1), ldb1, _ptr(part1), splits1, M2, N2,
                                 K2, _ptr(A2t), lda2t, _ptr(B2), ldb2, _ptr(part2), splits2,
                                 _stream(stream))
    if r < 0:
        raise BCMTError(BCMT_ERR_CUDA, bcmt_last_error())
    return r


def bcmt_test_attn(impl, backward, p: bcmt_params, q, k, v, ld, o, lse, dO=None, drow=None,
                   dq=None, dk=None, dv=None, ld_d=0, stream=None) -> None:
    r = LIB.bcmt_test_attn(impl, backward, ctypes.byref(p), _ptr(q), _ptr(k), _ptr(v), ld, _ptr(o),
                           _ptr(lse), _ptr(dO), _ptr(drow), _ptr(dq), _ptr(dk), _ptr(dv), ld_d,
                           _stream(stream))
    if r != 0:
        raise BCMTError(BCMT_ERR_CUDA, bcmt_last_error())


def bcmt_test_wait_expiry(cycles: int, stream=None) -> None:
    """Launches a wait that nothing ends, bounded by ``cycles`` SM clock
    cycles; afterwards bcmt_device_status() reports BCMT_ERR_TIMEOUT."""
    if LIB.bcmt_test_wait_expiry(cycles, _stream(stream)) != 0:
        raise BCMTError(BCMT_ERR_CUDA, bcmt_last_error())
