"""fp64 CPU oracle of the DAS hot path (ctypes loader for das_oracle.c).

TEST INFRASTRUCTURE ONLY: the test suite, the smoke check and the benchmark's
CPU-baseline leg may use it; the CUDA library never does.  It shares no code
with the CUDA path; only the seeded input generator (package `synth`) feeds
both.

Functions (each follows the paper; see das_oracle.c):
  attend_seq       Eqs. 2-3 for one sequence and layer, on given slabs
  attention        Eqs. 2-3 over a whole depth-indexed cache (Eq. 4 depths)
  greedy_accept    Sec. 3.4 acceptance
  kv_append        Sec. 3.4 / App. B.1 commit
All pinned by tests/test_oracle_pins.py (no function is left unpinned).
"""
import ctypes
import os

import numpy as np

from .build import LIB, build

_lib = None


def lib():
    global _lib
    if _lib is None:
        build()
        L = ctypes.CDLL(LIB)
        i, d, p = ctypes.c_int, ctypes.c_double, ctypes.c_void_p
        L.das_oracle_attend_seq.argtypes = [i, i, i, i, i, i, p, p, p, p, p, i, i, i, d, p, p, i, i]
        L.das_oracle_attend_seq.restype = None
        L.das_oracle_attention.argtypes = [p, p, i, i, i, i, i, i, i, i, i, p, p, i, p, p, p, i, d,
                                           i, p, p, i]
        L.das_oracle_attention.restype = i
        L.das_oracle_greedy_accept.argtypes = [p, p, i, i, i, p, p, p]
        L.das_oracle_greedy_accept.restype = None
        L.das_oracle_kv_append.argtypes = [p, p, i, i, i, i, i, i, p, p, p, i, p, p]
        L.das_oracle_kv_append.restype = None
        L.das_oracle_wave_readout.argtypes = [p, i, i, i, p, i]
        L.das_oracle_wave_readout.restype = None
        L.das_oracle_e4m3_decode_n.argtypes = [p, p, ctypes.c_size_t]
        L.das_oracle_e4m3_decode_n.restype = None
        L.das_oracle_e4m3_from_bf16_n.argtypes = [p, p, ctypes.c_size_t]
        L.das_oracle_e4m3_from_bf16_n.restype = None
        L.das_oracle_kv_append_f8.argtypes = [p, p, p, p, i, i, i, i, i, i, p, p, p, i, p, p]
        L.das_oracle_kv_append_f8.restype = None
        _lib = L
    return _lib


def _threads():
    try:
        return max(1, len(os.sched_getaffinity(0)))
    except AttributeError:
        return os.cpu_count() or 1


def _u16(a):
    return np.ascontiguousarray(a, dtype=np.uint16)


def attend_seq(q, k_pre, v_pre, k_blk, v_blk, block_len=None, prefix_range=None, use_block=True,
               scale=None, heads=None):
    """One sequence, one layer.  q [T][Hq][D], k_pre/v_pre [P][Hkv][D],
    k_blk/v_blk [T][Hkv][D], all bf16 bits.  Returns out [T][Hq][D] and
    lse [Hq][T] in float64."""
    q, k_pre, v_pre, k_blk, v_blk = map(_u16, (q, k_pre, v_pre, k_blk, v_blk))
    T, Hq, D = q.shape
    P, Hkv = k_pre.shape[0], k_pre.shape[1]
    lo, hi = (0, P) if prefix_range is None else prefix_range
    h_lo, h_hi = (0, Hq) if heads is None else heads
    out = np.zeros((T, Hq, D))
    lse = np.full((Hq, T), -np.inf)
    lib().das_oracle_attend_seq(P, T, T if block_len is None else block_len, Hq, Hkv, D,
                                q.ctypes.data, k_pre.ctypes.data, v_pre.ctypes.data,
                                k_blk.ctypes.data, v_blk.ctypes.data, lo, hi, int(use_block),
                                1.0 / np.sqrt(D) if scale is None else float(scale),
                                out.ctypes.data, lse.ctypes.data, h_lo, h_hi)
    return out, lse


def attention(K, V, layer, key_depth, value_depth, prefix_len, block_len, q, k_blk, v_blk,
              scale=None, use_block=True, nthreads=None):
    """Whole cache.  K, V bf16 bits [R][L][B][cap][Hkv][D]; q [B][T][Hq][D];
    k_blk, v_blk [B][T][Hkv][D].  Returns out [B][T][Hq][D], lse [B][Hq][T]."""
    K, V, q, k_blk, v_blk = map(_u16, (K, V, q, k_blk, v_blk))
    R, L, B, cap, Hkv, D = K.shape
    T, Hq = q.shape[1], q.shape[2]
    pl = np.ascontiguousarray(prefix_len, dtype=np.int32)
    bl = np.ascontiguousarray(block_len, dtype=np.int32)
    out = np.zeros((B, T, Hq, D))
    lse = np.full((B, Hq, T), -np.inf)
    rc = lib().das_oracle_attention(K.ctypes.data, V.ctypes.data, R, L, B, cap, Hkv, D, layer,
                                    key_depth, value_depth, pl.ctypes.data, bl.ctypes.data, T,
                                    q.ctypes.data, k_blk.ctypes.data, v_blk.ctypes.data, Hq,
                                    0.0 if scale is None else float(scale), int(use_block),
                                    out.ctypes.data, lse.ctypes.data, nthreads or _threads())
    if rc:
        raise ValueError("oracle: arguments outside the definition")
    return out, lse


def greedy_accept(logits, draft):
    """logits float32 [B][W][V], draft int32 [B][W] ->
    (accepted [B], target_ids [B][W], next_token [B]) int32."""
    lg = np.ascontiguousarray(logits, dtype=np.float32)
    dr = np.ascontiguousarray(draft, dtype=np.int32)
    B, W, Vv = lg.shape
    acc = np.zeros(B, dtype=np.int32)
    tid = np.zeros((B, W), dtype=np.int32)
    nxt = np.zeros(B, dtype=np.int32)
    lib().das_oracle_greedy_accept(lg.ctypes.data, dr.ctypes.data, B, W, Vv, acc.ctypes.data,
                                   tid.ctypes.data, nxt.ctypes.data)
    return acc, tid, nxt


def e4m3_decode(codes):
    """e4m3 codes (uint8) -> float64 values, exactly."""
    c = np.ascontiguousarray(codes, dtype=np.uint8)
    out = np.empty(c.shape, dtype=np.float64)
    lib().das_oracle_e4m3_decode_n(c.ctypes.data, out.ctypes.data, c.size)
    return out


def e4m3_from_bf16(bits):
    """bf16 bits -> e4m3 codes: nearest, ties to even, saturating at +-448."""
    b = np.ascontiguousarray(bits, dtype=np.uint16)
    out = np.empty(b.shape, dtype=np.uint8)
    lib().das_oracle_e4m3_from_bf16_n(b.ctypes.data, out.ctypes.data, b.size)
    return out


def _bf16_bits_exact(x):
    """float64 values that are exactly bf16 (e4m3 values are) -> bf16 bits."""
    f = np.ascontiguousarray(x, dtype=np.float32)
    u = f.view(np.uint32)
    if np.any((u & 0xFFFF) != 0):
        raise ValueError("oracle: value is not a bf16 value")
    return (u >> 16).astype(np.uint16)


def widen_f8_cache(top, low):
    """The depth-indexed bf16 cache [R][L][B][cap][Hkv][D] that an e4m3 cache
    (top: bf16 bits [L][B][cap][Hkv][D] of depth R; low: e4m3 codes
    [R-1][L][B][cap][Hkv][D]) stores, every value widened exactly."""
    top = np.ascontiguousarray(top, dtype=np.uint16)
    R = 1 + (0 if low is None else low.shape[0])
    full = np.empty((R,) + top.shape, dtype=np.uint16)
    full[R - 1] = top
    if R > 1:
        full[:R - 1] = _bf16_bits_exact(e4m3_decode(low))
    return full


def attention_f8(k_top, v_top, k_low, v_low, layer, key_depth, value_depth, prefix_len,
                 block_len, q, k_blk, v_blk, scale=None, nthreads=None):
    """Eqs. 2-3 on an e4m3 cache: the attention of the values it stores."""
    return attention(widen_f8_cache(k_top, k_low), widen_f8_cache(v_top, v_low), layer,
                     key_depth, value_depth, prefix_len, block_len, q, k_blk, v_blk, scale=scale,
                     nthreads=nthreads)


def kv_append_f8(k_top, v_top, k_low, v_low, k_new, v_new, accepted, prefix_len):
    """The commit into an e4m3 cache; returns new (k_top, v_top, k_low, v_low,
    prefix_len, error_flag) without touching the inputs."""
    kt, vt = (np.array(x, dtype=np.uint16, copy=True) for x in (k_top, v_top))
    kl, vl = (np.array(x, dtype=np.uint8, copy=True) for x in (k_low, v_low))
    kn, vn = _u16(k_new), _u16(v_new)
    R, L, B, W, Hkv, D = kn.shape
    cap = kt.shape[2]
    acc = np.ascontiguousarray(accepted, dtype=np.int32)
    pl = np.array(prefix_len, dtype=np.int32, copy=True)
    flag = np.zeros(1, dtype=np.int32)
    lib().das_oracle_kv_append_f8(kt.ctypes.data, vt.ctypes.data, kl.ctypes.data, vl.ctypes.data,
                                  R, L, B, cap, Hkv, D, kn.ctypes.data, vn.ctypes.data,
                                  acc.ctypes.data, W, pl.ctypes.data, flag.ctypes.data)
    return kt, vt, kl, vl, pl, int(flag[0])


def wave_readout(logits, tokens):
    """Eq. 6 shifted readout: tokens' = tokens with tokens'[b][i+1] =
    argmax logits[b][i] for i < W (first maximum).  logits float32 [B][W][V],
    tokens int32 [B][S], S >= W + 1; the input is not modified."""
    lg = np.ascontiguousarray(logits, dtype=np.float32)
    tk = np.array(tokens, dtype=np.int32, copy=True, order="C")
    B, W, Vv = lg.shape
    if tk.shape[0] != B or tk.shape[1] < W + 1:
        raise ValueError("oracle: tokens must be [B][>= W+1]")
    lib().das_oracle_wave_readout(lg.ctypes.data, B, W, Vv, tk.ctypes.data, tk.shape[1])
    return tk


def wave_width(gamma, w_init, j):
    """Active width of refinement round j (Eq. 5): W_j = min(gamma, W_init + j)."""
    return min(gamma, w_init + j)


def kv_append(K, V, k_new, v_new, accepted, prefix_len):
    """Returns (K', V', prefix_len', error_flag) without touching the inputs.
    K, V [R][L][B][cap][Hkv][D]; k_new, v_new [R][L][B][W][Hkv][D] (bf16 bits)."""
    K2, V2 = np.array(K, dtype=np.uint16, copy=True), np.array(V, dtype=np.uint16, copy=True)
    kn, vn = _u16(k_new), _u16(v_new)
    R, L, B, cap, Hkv, D = K2.shape
    W = kn.shape[3]
    acc = np.ascontiguousarray(accepted, dtype=np.int32)
    pl = np.array(prefix_len, dtype=np.int32, copy=True)
    flag = np.zeros(1, dtype=np.int32)
    lib().das_oracle_kv_append(K2.ctypes.data, V2.ctypes.data, R, L, B, cap, Hkv, D,
                               kn.ctypes.data, vn.ctypes.data, acc.ctypes.data, W, pl.ctypes.data,
                               flag.ctypes.data)
    return K2, V2, pl, int(flag[0])
