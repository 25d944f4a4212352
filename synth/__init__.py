"""Seeded synthetic inputs for the DAS hot path (host side, plus device fill).

The arithmetic lives in synth_core.h; this module only loads the two shared
libraries and shapes their output.  It holds none of the method's arithmetic,
so both the CPU oracle's tests and the CUDA path's tests and benchmark use it.
"""
import ctypes
import os

import numpy as np

from .build import DEV_LIB, HOST_LIB, build_dev, build_host

# tensor ids, as in synth_core.h
T_KCACHE, T_VCACHE, T_Q, T_KBLK, T_VBLK, T_KNEW, T_VNEW = 1, 2, 3, 4, 5, 6, 7
T_LOGITS, T_DRAFT, T_ACCEPT, T_PREFIX, T_BLOCK, T_FILL = 8, 9, 10, 11, 12, 13

_host = None
_dev = None


def host_lib():
    global _host
    if _host is None:
        build_host()
        lib = ctypes.CDLL(HOST_LIB)
        i, u64, d, p = ctypes.c_int, ctypes.c_uint64, ctypes.c_double, ctypes.c_void_p
        lib.synth_matured_block.argtypes = [u64, i, i, i, i, i, i, i, i, i, i, i, p, i]
        lib.synth_matured_block.restype = i
        lib.synth_normal_block.argtypes = [u64, i, i, i, i, i, i, i, i, d, p, i]
        lib.synth_normal_block.restype = i
        lib.synth_uniform_int.argtypes = [u64, i, u64, ctypes.c_int64, ctypes.c_int64]
        lib.synth_uniform_int.restype = ctypes.c_int64
        lib.synth_accept_inputs.argtypes = [u64, i, i, i, p, p, p]
        lib.synth_accept_inputs.restype = i
        lib.synth_e4m3_codes.argtypes = [u64, i, u64, ctypes.c_size_t, p]
        lib.synth_e4m3_codes.restype = None
        _host = lib
    return _host


def dev_lib():
    """The device fill library (needs a GPU to run, not to load)."""
    global _dev
    if _dev is None:
        build_dev()
        lib = ctypes.CDLL(DEV_LIB)
        i, u64, p = ctypes.c_int, ctypes.c_uint64, ctypes.c_void_p
        lib.synth_dev_fill_matured.argtypes = [p, u64, i, i, i, i, i, i, i, i, i, p]
        lib.synth_dev_fill_matured.restype = i
        lib.synth_dev_fill_filler.argtypes = [p, ctypes.c_size_t, u64, p]
        lib.synth_dev_fill_filler.restype = i
        _dev = lib
    return _dev


def _threads():
    try:
        return max(1, len(os.sched_getaffinity(0)))
    except AttributeError:
        return os.cpu_count() or 1


def matured_block(seed, tensor, is_value, depth, R, layer, b, t0, t1, h0, h1, D, nthreads=None):
    """bf16 bits [t1-t0][h1-h0][D] of a matured tensor at stored depth `depth`."""
    out = np.empty((t1 - t0, h1 - h0, D), dtype=np.uint16)
    rc = host_lib().synth_matured_block(seed, tensor, int(is_value), depth, R, layer, b, t0, t1,
                                        h0, h1, D, out.ctypes.data, nthreads or _threads())
    if rc:
        raise ValueError("coordinates outside the generator's counter layout")
    return out


def normal_block(seed, tensor, layer, b, t0, t1, h0, h1, D, divisor=1.0, nthreads=None):
    """bf16 bits [t1-t0][h1-h0][D] of N(0,1)/divisor."""
    out = np.empty((t1 - t0, h1 - h0, D), dtype=np.uint16)
    rc = host_lib().synth_normal_block(seed, tensor, layer, b, t0, t1, h0, h1, D, float(divisor),
                                       out.ctypes.data, nthreads or _threads())
    if rc:
        raise ValueError("coordinates outside the generator's counter layout")
    return out


T_KLOW, T_VLOW = 14, 15


def e4m3_codes(seed, tensor, shape, c0=0):
    """uint8 e4m3 codes of the given shape (random sign, exponent field 4..9,
    random mantissa; never NaN) from tensor stream `tensor`."""
    n = int(np.prod(shape))
    out = np.empty(n, dtype=np.uint8)
    host_lib().synth_e4m3_codes(seed, tensor, c0, n, out.ctypes.data)
    return out.reshape(shape)


def uniform_int(seed, tensor, idx, lo, hi):
    return int(host_lib().synth_uniform_int(seed, tensor, idx, lo, hi))


def accept_inputs(seed, B, W, vocab):
    """(accept_star int32 [B], draft int32 [B][W], logits float32 [B][W][vocab])."""
    a = np.empty(B, dtype=np.int32)
    d = np.empty((B, W), dtype=np.int32)
    lg = np.empty((B, W, vocab), dtype=np.float32)
    if host_lib().synth_accept_inputs(seed, B, W, vocab, a.ctypes.data, d.ctypes.data,
                                      lg.ctypes.data):
        raise ValueError("bad accept-input shape")
    return a, d, lg


def bf16_bits_to_float(bits):
    """bf16 bits (uint16) -> float32, exact."""
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)
