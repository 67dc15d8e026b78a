"""Python binding of libmosaic.so (include/mosaic.h).

Argument marshalling only: every function has the name of the C entry point
it calls, takes torch tensors (or None) for device buffers, passes their
device addresses and the current CUDA stream, and raises MosaicError on a
non-OK status.  All arithmetic happens in the library's kernels.  Ring
buffers are int32 tensors holding uint32 bit patterns; bf16 digit planes are
int16 tensors holding bf16 bit patterns.

There is no fallback: if the library is missing, ``lib()`` raises.
"""
from __future__ import annotations

import ctypes
import os

from . import build as _build

OK = 0
STATUS = {0: "ok", 1: "invalid argument", 2: "invalid shape", 3: "misaligned", 4: "unsupported",
          5: "CUDA error", 6: "workspace too small", 7: "device wait timed out"}

GEMM_AUTO, GEMM_TC, GEMM_MMA_S8, GEMM_IMAD = 0, 1, 2, 3
SKINNY_MAX_M = 16   # MOSAIC_SKINNY_MAX_M: token counts the streaming product serves
STREAMW_MAX_M = 64  # MOSAIC_STREAMW_MAX_M: up to here the tensor-core product streams B as uint32
OP_RING_GEMM, OP_MASK_CHAINS, OP_MASK_WEIGHT, OP_MASK_ACTIVATION, OP_UNMASK = 1, 2, 3, 4, 5
OP_FREIVALDS_CHECK, OP_ACTIVATION_PLANES, OP_UNMASK_PLANES = 6, 7, 8
TAG_M, TAG_N, TAG_L, TAG_S, TAG_EW, TAG_R, TAG_T, TAG_EX, TAG_SIGN, TAG_CHECK = range(1, 11)


class MosaicError(RuntimeError):
    def __init__(self, fn, status):
        super().__init__(f"{fn} failed: {STATUS.get(status, status)} ({status})")
        self.status = status


class mosaic_params(ctypes.Structure):
    _fields_ = [("kappa", ctypes.c_uint32), ("d", ctypes.c_uint32), ("r", ctypes.c_uint32 * 3),
                ("t", ctypes.c_uint32 * 3), ("sigma", ctypes.c_float), ("qbits", ctypes.c_uint32),
                ("rounds", ctypes.c_uint32), ("act_nested", ctypes.c_uint32)]


class mosaic_key(ctypes.Structure):
    _fields_ = [("key", ctypes.c_uint32 * 8)]


MASK_CHAINS, MASK_WEIGHT, MASK_ACTIVATION = 1, 2, 3


class mosaic_mask_io(ctypes.Structure):
    _fields_ = [("W", ctypes.c_void_p), ("ldw", ctypes.c_int64), ("n", ctypes.c_int64),
                ("P", ctypes.c_void_p), ("C", ctypes.c_void_p), ("CT", ctypes.c_void_p),
                ("sign_words", ctypes.c_void_p), ("s_w", ctypes.c_void_p), ("L", ctypes.c_void_p),
                ("S_idx", ctypes.c_void_p), ("S_val", ctypes.c_void_p), ("Wp", ctypes.c_void_p),
                ("Wp_planes", ctypes.c_void_p), ("J", ctypes.c_void_p), ("cj_planes", ctypes.c_void_p),
                ("pass_dev", ctypes.c_void_p), ("Ux_tm", ctypes.c_void_p), ("K_tm", ctypes.c_void_p)]


class mosaic_kernel_time(ctypes.Structure):
    _fields_ = [("name", ctypes.c_char * 64), ("launches", ctypes.c_uint64), ("ms", ctypes.c_double)]


_lib = None
_P, _I64, _U32, _U64, _INT, _F32 = (ctypes.c_void_p, ctypes.c_int64, ctypes.c_uint32,
                                    ctypes.c_uint64, ctypes.c_int, ctypes.c_float)
_SZ = ctypes.c_size_t
_PP = ctypes.POINTER(mosaic_params)
_PK = ctypes.POINTER(mosaic_key)

_SIGS = {
    "mosaic_default_params": ([_PP], None),
    "mosaic_kernel_launches": ([], ctypes.c_uint64),
    "mosaic_kernel_timing": ([_INT], _INT),
    "mosaic_int_mix_rate": ([_P, _SZ, ctypes.POINTER(ctypes.c_double), _P], _INT),
    "mosaic_smem_read_rate": ([_P, _SZ, ctypes.POINTER(ctypes.c_double), _P], _INT),
    "mosaic_kernel_times": ([ctypes.POINTER(mosaic_kernel_time), _INT, _INT], _INT),
    "mosaic_status_string": ([_INT], ctypes.c_char_p),
    "mosaic_qmax": ([_I64, _U32], ctypes.c_int32),
    "mosaic_gaussian_table": ([_F32, _P, _INT], _INT),
    "mosaic_prg_uniform": ([_PK, _U32, _U64, _U32, _I64, _I64, _P, _I64, _P], _INT),
    "mosaic_prg_gaussian": ([_PK, _U32, _U64, _U32, _F32, _I64, _P, _P], _INT),
    "mosaic_prg_sparse": ([_PK, _U32, _U64, _U32, _I64, _U32, _U32, _P, _P, _P, _P], _INT),
    "mosaic_hadamard": ([_P, _I64, _P, _I64, _I64, _I64, _P, _P], _INT),
    "mosaic_encode": ([_P, _I64, _I64, _I64, _I64, ctypes.c_int32, _INT, _P, _P, _I64, _P, _I64,
                       _P, _P, _P], _INT),
    "mosaic_digit_split": ([_P, _I64, _I64, _I64, _P, _P], _INT),
    "mosaic_gemm_variant_available": ([_INT], _INT),
    "mosaic_ring_gemm": ([_P, _I64, _P, _I64, _P, _I64, _I64, _I64, _I64, _INT, _P, _SZ, _P], _INT),
    "mosaic_ring_gemm_planes": ([_P, _I64, _I64, _P, _I64, _I64, _P, _I64, _I64, _I64, _I64, _INT,
                                 _P], _INT),
    "mosaic_mask_chains": ([_PP, _PK, _U64, _I64, _P, _P, _P, _P, _SZ, _P], _INT),
    "mosaic_mask_weight": ([_PP, _PK, _U64, _P, _I64, _I64, _I64, _I64, _P, _P, _P, _P, _P, _P, _P,
                            _P, _P, _P, _INT, _P, _SZ, _P], _INT),
    "mosaic_mask_activation": ([_PP, _PK, _U64, _I64, _I64, _I64, _P, _P, _P, _P, _INT, _P, _SZ,
                                _P], _INT),
    "mosaic_unmask": ([_PP, _I64, _I64, _P, _I64, _P, _P, _P, _P, _P, _P, _P, _P, _P, _I64, _INT,
                       _P, _SZ, _P], _INT),
    "mosaic_workspace_bytes": ([_INT, _I64, _I64, _I64, _PP], _SZ),
    "mosaic_device_status": ([_P], _INT),
    "mosaic_unmask_noalloc": ([_PP, _I64, _I64, _P, _I64, _P, _P, _P, _P, _P, _P, _P, _P, _P, _I64,
                               _INT, _P], _INT),
    "mosaic_prepare_activation": ([_PP, _I64, _I64, _P, _P, _P, _P], _INT),
    "mosaic_mask_activation_planes": ([_PP, _PK, _U64, _I64, _I64, _I64, _P, _P, _P, _P, _P, _INT, _P,
                                       _SZ, _P], _INT),
    "mosaic_mask_activation_ex": ([_PP, _PK, _U64, _P, _I64, _I64, _I64, _P, _P, _P, _P, _P, _INT, _P, _SZ,
                                   _P], _INT),
    "mosaic_mask_activation_phase": ([_PP, _PK, _U64, _P, _I64, _I64, _I64, _P, _P, _P, _P, _P, _INT, _P, _SZ,
                                      _INT, _P], _INT),
    "mosaic_advance_pass": ([_P, _U64, _P], _INT),
    "mosaic_mask": ([_INT, _PP, _PK, _U64, _I64, _I64, _I64, ctypes.POINTER(mosaic_mask_io), _INT, _P, _SZ,
                     _P], _INT),
    "mosaic_prepare_unmask": ([_PP, _I64, _P, _P, _P], _INT),
    "mosaic_unmask_planes": ([_PP, _I64, _I64, _P, _I64, _P, _P, _P, _P, _P, _P, _P, _P, _P, _P, _I64,
                              _INT, _P, _SZ, _P], _INT),
    "mosaic_selftest_wait": ([_I64, _P], _INT),
    "mosaic_rmsnorm": ([_P, _I64, _I64, _I64, _F32, _P, _I64, _P], _INT),
    "mosaic_swiglu": ([_P, _I64, _I64, _I64, _P, _I64, _P], _INT),
    "mosaic_freivalds_setup": ([_PP, _PK, _U64, _INT, _P, _I64, _I64, _I64, _P, _P, _P], _INT),
    "mosaic_freivalds_check": ([_INT, _P, _P, _I64, _I64, _I64, _P, _I64, _P, _I64, _P, _P, _P, _SZ,
                                _P], _INT),
}

EXPORTS = tuple(_SIGS)


def library_path() -> str:
    return _build.LIB


def lib():
    """Loads libmosaic.so; raises if it has not been built."""
    global _lib
    if _lib is None:
        path = _build.LIB
        if not os.path.exists(path):
            raise RuntimeError(f"libmosaic.so not found at {path}: run "
                               "paper_2607_29221_gb300.build.build() first")
        L = ctypes.CDLL(path)
        for name, (args, res) in _SIGS.items():
            f = getattr(L, name)
            f.argtypes = args
            f.restype = res
        _lib = L
    return _lib


# ---------------------------------------------------------------------------
def default_params(**over) -> mosaic_params:
    p = mosaic_params()
    lib().mosaic_default_params(ctypes.byref(p))
    for k, v in over.items():
        if k in ("r", "t"):
            arr = getattr(p, k)
            for i in range(3):
                arr[i] = v[i] if i < len(v) else 0
        else:
            setattr(p, k, v)
    return p


def make_key(words) -> mosaic_key:
    k = mosaic_key()
    for i in range(8):
        k.key[i] = int(words[i]) & 0xFFFFFFFF
    return k


def _ptr(t):
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream(stream):
    if stream is not None:
        return stream if isinstance(stream, int) else stream.cuda_stream
    import torch
    return torch.cuda.current_stream().cuda_stream


def _call(name, *args):
    st = getattr(lib(), name)(*args)
    if st != OK:
        raise MosaicError(name, st)


# ---------------------------------------------------------------------------
def mosaic_kernel_launches() -> int:
    return int(lib().mosaic_kernel_launches())


def mosaic_kernel_timing(enable: bool) -> bool:
    """Turns per-kernel event timing on or off; returns the previous setting."""
    return bool(lib().mosaic_kernel_timing(1 if enable else 0))


def mosaic_kernel_times(reset: bool = True) -> dict:
    """{"<role>:<kernel>": (launches, total ms)} of the launches timed so far."""
    n = int(lib().mosaic_kernel_times(None, 0, 0))
    if n < 0:
        raise MosaicError("mosaic_kernel_times", -1)
    buf = (mosaic_kernel_time * max(n, 1))()
    n = int(lib().mosaic_kernel_times(buf, n, 1 if reset else 0))
    if n < 0:
        raise MosaicError("mosaic_kernel_times", -1)
    return {buf[i].name.decode(): (int(buf[i].launches), float(buf[i].ms)) for i in range(min(n, len(buf)))}


def mosaic_int_mix_rate(scratch, stream=None) -> float:
    """Measured ChaCha20 mix (add / xor / rotate) rate of the device, ops/s."""
    out = ctypes.c_double(0.0)
    _call("mosaic_int_mix_rate", _ptr(scratch), scratch.numel() * scratch.element_size(), ctypes.byref(out),
          _stream(stream))
    return float(out.value)


def mosaic_smem_read_rate(scratch, stream=None) -> float:
    """Measured shared-memory read rate of the device with the tiled gather's
    access (whole 128-byte lines, 16-byte loads), bytes/s."""
    out = ctypes.c_double(0.0)
    _call("mosaic_smem_read_rate", _ptr(scratch), scratch.numel() * scratch.element_size(), ctypes.byref(out),
          _stream(stream))
    return float(out.value)


def mosaic_qmax(n_pad: int, qbits: int = 16) -> int:
    return int(lib().mosaic_qmax(n_pad, qbits))


def mosaic_gaussian_table(sigma: float):
    import numpy as np
    buf = np.zeros(256, np.uint64)
    B = lib().mosaic_gaussian_table(sigma, buf.ctypes.data_as(ctypes.c_void_p), 256)
    if B < 0:
        raise MosaicError("mosaic_gaussian_table", 1)
    return buf[: 2 * B + 1].copy()


def mosaic_gemm_variant_available(variant: int) -> bool:
    return bool(lib().mosaic_gemm_variant_available(variant))


def mosaic_device_status(stream=None):
    _call("mosaic_device_status", _stream(stream))


def mosaic_selftest_wait(limit_us: int, stream=None):
    """Launches a bounded wait that runs out after limit_us (the timeout path's
    self-test); the next mosaic_device_status raises MOSAIC_ERR_TIMEOUT."""
    _call("mosaic_selftest_wait", limit_us, _stream(stream))


def mosaic_workspace_bytes(op: int, m: int, n_pad: int, l: int, params: mosaic_params = None) -> int:
    return int(lib().mosaic_workspace_bytes(op, m, n_pad, l,
                                            None if params is None else ctypes.byref(params)))


def mosaic_prg_uniform(key, tag, stream_id, rounds, rows, cols, out, ldo=None, stream=None):
    _call("mosaic_prg_uniform", ctypes.byref(key), tag, stream_id, rounds, rows, cols, _ptr(out),
          cols if ldo is None else ldo, _stream(stream))


def mosaic_prg_gaussian(key, tag, stream_id, rounds, sigma, count, out, stream=None):
    _call("mosaic_prg_gaussian", ctypes.byref(key), tag, stream_id, rounds, sigma, count, _ptr(out),
          _stream(stream))


def mosaic_prg_sparse(key, tag, stream_id, rounds, rows, r, t, idx, val, fail=None, stream=None):
    _call("mosaic_prg_sparse", ctypes.byref(key), tag, stream_id, rounds, rows, r, t, _ptr(idx),
          _ptr(val), _ptr(fail), _stream(stream))


def mosaic_hadamard(x, ldx, y, rows, n, n_pad, sign_words=None, stream=None):
    _call("mosaic_hadamard", _ptr(x), ldx, _ptr(y), rows, n, n_pad, _ptr(sign_words),
          _stream(stream))


def mosaic_encode(x, ldx, rows, n, n_pad, qmax, rotate, sign_words, mask, ldm, out, ldo, scale,
                  planes=None, stream=None):
    _call("mosaic_encode", _ptr(x), ldx, rows, n, n_pad, qmax, rotate, _ptr(sign_words), _ptr(mask),
          ldm, _ptr(out), ldo, _ptr(scale), _ptr(planes), _stream(stream))


def mosaic_digit_split(a, lda, rows, cols, planes, stream=None):
    _call("mosaic_digit_split", _ptr(a), lda, rows, cols, _ptr(planes), _stream(stream))


def mosaic_ring_gemm(A, lda, B, ldb, C, ldc, M, N, K, variant=GEMM_AUTO, ws=None, ws_bytes=0,
                     stream=None):
    if ws is not None and not ws_bytes:
        ws_bytes = ws.numel() * ws.element_size()
    _call("mosaic_ring_gemm", _ptr(A), lda, _ptr(B), ldb, _ptr(C), ldc, M, N, K, variant, _ptr(ws),
          ws_bytes, _stream(stream))


def mosaic_ring_gemm_planes(Ap, ldpa, a_plane, Bp, ldpb, b_plane, C, ldc, M, N, K,
                            variant=GEMM_TC, stream=None):
    _call("mosaic_ring_gemm_planes", _ptr(Ap), ldpa, a_plane, _ptr(Bp), ldpb, b_plane, _ptr(C), ldc,
          M, N, K, variant, _stream(stream))


def mosaic_mask_chains(params, key, chain_id, n_pad, P, C, CT, ws, stream=None):
    _call("mosaic_mask_chains", ctypes.byref(params), ctypes.byref(key), chain_id, n_pad, _ptr(P),
          _ptr(C), _ptr(CT), _ptr(ws), 0 if ws is None else ws.numel() * ws.element_size(),
          _stream(stream))


def mosaic_mask_weight(params, key, matrix_id, W, ldw, m, n, n_pad, P, CT, sign_words, s_w, L,
                       S_idx, S_val, Wp, Wp_planes, J, variant, ws, stream=None):
    _call("mosaic_mask_weight", ctypes.byref(params), ctypes.byref(key), matrix_id, _ptr(W), ldw, m,
          n, n_pad, _ptr(P), _ptr(CT), _ptr(sign_words), _ptr(s_w), _ptr(L), _ptr(S_idx),
          _ptr(S_val), _ptr(Wp), _ptr(Wp_planes), _ptr(J), variant, _ptr(ws),
          0 if ws is None else ws.numel() * ws.element_size(), _stream(stream))


def mosaic_mask_activation(params, key, pass_id, m, n_pad, l, C, J, Ux_tm, K_tm, variant, ws,
                           stream=None):
    _call("mosaic_mask_activation", ctypes.byref(params), ctypes.byref(key), pass_id, m, n_pad, l,
          _ptr(C), _ptr(J), _ptr(Ux_tm), _ptr(K_tm), variant, _ptr(ws),
          0 if ws is None else ws.numel() * ws.element_size(), _stream(stream))


def mosaic_unmask(params, l, m, Z, ldz, K_tm, L, S_idx, S_val, s_w, s_x, bias, Y, Yhat, ldy,
                  variant, ws, stream=None):
    _call("mosaic_unmask", ctypes.byref(params), l, m, _ptr(Z), ldz, _ptr(K_tm), _ptr(L),
          _ptr(S_idx), _ptr(S_val), _ptr(s_w), _ptr(s_x), _ptr(bias), _ptr(Y), _ptr(Yhat), ldy,
          variant, _ptr(ws), 0 if ws is None else ws.numel() * ws.element_size(), _stream(stream))


def mosaic_unmask_noalloc(params, l, m, Z, ldz, K_tm, L, S_idx, S_val, s_w, s_x, bias, Y, Yhat, ldy,
                          variant, stream=None):
    """mosaic_unmask without a workspace: for callers that cannot allocate
    device memory, the scratch is a fixed 16 MiB array inside the library
    (l * m <= 2^22).  Calls whose GPU work overlaps share that array and race."""
    _call("mosaic_unmask_noalloc", ctypes.byref(params), l, m, _ptr(Z), ldz, _ptr(K_tm), _ptr(L),
          _ptr(S_idx), _ptr(S_val), _ptr(s_w), _ptr(s_x), _ptr(bias), _ptr(Y), _ptr(Yhat), ldy,
          variant, _stream(stream))


def mosaic_rmsnorm(x, ldx, rows, n, eps, y, ldy, stream=None):
    _call("mosaic_rmsnorm", _ptr(x), ldx, rows, n, eps, _ptr(y), ldy, _stream(stream))


def mosaic_swiglu(gu, ldg, rows, ffn, out, ldo, stream=None):
    _call("mosaic_swiglu", _ptr(gu), ldg, rows, ffn, _ptr(out), ldo, _stream(stream))


def mosaic_freivalds_setup(params, key, matrix_id, k, Wm, ldw, m, n_pad, a, Ychk, stream=None):
    _call("mosaic_freivalds_setup", ctypes.byref(params), ctypes.byref(key), matrix_id, k, _ptr(Wm), ldw,
          m, n_pad, _ptr(a), _ptr(Ychk), _stream(stream))


def mosaic_freivalds_check(k, a, Ychk, m, n_pad, l, Z, ldz, Xp, ldx, bad, n_bad, ws, stream=None):
    _call("mosaic_freivalds_check", k, _ptr(a), _ptr(Ychk), m, n_pad, l, _ptr(Z), ldz, _ptr(Xp), ldx,
          _ptr(bad), _ptr(n_bad), _ptr(ws), 0 if ws is None else ws.numel() * ws.element_size(),
          _stream(stream))


def mosaic_prepare_activation(params, m, n_pad, C, J, cj_planes, stream=None):
    _call("mosaic_prepare_activation", ctypes.byref(params), m, n_pad, _ptr(C), _ptr(J), _ptr(cj_planes),
          _stream(stream))


def mosaic_mask_activation_planes(params, key, pass_id, m, n_pad, l, C, J, cj_planes, Ux_tm, K_tm, variant,
                                  ws, stream=None):
    _call("mosaic_mask_activation_planes", ctypes.byref(params), ctypes.byref(key), pass_id, m, n_pad, l,
          _ptr(C), _ptr(J), _ptr(cj_planes), _ptr(Ux_tm), _ptr(K_tm), variant, _ptr(ws),
          0 if ws is None else ws.numel() * ws.element_size(), _stream(stream))


def mosaic_prepare_unmask(params, m, L, L_planes, stream=None):
    _call("mosaic_prepare_unmask", ctypes.byref(params), m, _ptr(L), _ptr(L_planes), _stream(stream))


def mosaic_unmask_planes(params, l, m, Z, ldz, K_tm, L, L_planes, S_idx, S_val, s_w, s_x, bias, Y, Yhat,
                         ldy, variant, ws, stream=None):
    _call("mosaic_unmask_planes", ctypes.byref(params), l, m, _ptr(Z), ldz, _ptr(K_tm), _ptr(L),
          _ptr(L_planes), _ptr(S_idx), _ptr(S_val), _ptr(s_w), _ptr(s_x), _ptr(bias), _ptr(Y), _ptr(Yhat),
          ldy, variant, _ptr(ws), 0 if ws is None else ws.numel() * ws.element_size(), _stream(stream))


def mosaic_mask_activation_ex(params, key, pass_id, pass_dev, m, n_pad, l, C, J, cj_planes, Ux_tm, K_tm,
                              variant, ws, stream=None):
    _call("mosaic_mask_activation_ex", ctypes.byref(params), ctypes.byref(key), pass_id, _ptr(pass_dev), m,
          n_pad, l, _ptr(C), _ptr(J), _ptr(cj_planes), _ptr(Ux_tm), _ptr(K_tm), variant, _ptr(ws),
          0 if ws is None else ws.numel() * ws.element_size(), _stream(stream))


INITX_DRAWS, INITX_COMPOSE, INITX_ALL = 1, 2, 3


def mosaic_mask_activation_phase(params, key, pass_id, pass_dev, m, n_pad, l, C, J, cj_planes, Ux_tm, K_tm,
                                 variant, ws, phase, stream=None):
    _call("mosaic_mask_activation_phase", ctypes.byref(params), ctypes.byref(key), pass_id, _ptr(pass_dev), m,
          n_pad, l, _ptr(C), _ptr(J), _ptr(cj_planes), _ptr(Ux_tm), _ptr(K_tm), variant, _ptr(ws),
          0 if ws is None else ws.numel() * ws.element_size(), phase, _stream(stream))


def mosaic_mask(kind, params, key, stream_id, rows, n_pad, l, io: dict, variant=GEMM_AUTO, ws=None,
                stream=None):
    """io: field name of mosaic_mask_io -> tensor (device buffers) or int (ldw, n)."""
    s = mosaic_mask_io()
    for name, _ in mosaic_mask_io._fields_:
        v = io.get(name)
        if v is not None:                 # fields left out stay 0 / NULL
            setattr(s, name, v if isinstance(v, int) else _ptr(v))
    _call("mosaic_mask", kind, ctypes.byref(params), ctypes.byref(key), stream_id, rows, n_pad, l,
          ctypes.byref(s), variant, _ptr(ws), 0 if ws is None else ws.numel() * ws.element_size(),
          _stream(stream))


def mosaic_advance_pass(pass_dev, delta=1, stream=None):
    _call("mosaic_advance_pass", _ptr(pass_dev), delta, _stream(stream))
