"""The seeded input generator (no GPU): its primitives against exact or
library references, its distributions, and the depth-maturation law."""
import ctypes
import math

import numpy as np
import pytest

import synth
from synth import workloads as wl_mod


def _lib():
    L = synth.host_lib()
    p, sz = ctypes.c_void_p, ctypes.c_size_t
    L.synth_bf16_array.argtypes = [p, sz, p]
    L.synth_ln_array.argtypes = [p, sz, p]
    L.synth_cos_turn_array.argtypes = [p, sz, p]
    L.synth_normal_array.argtypes = [ctypes.c_uint64, ctypes.c_int, ctypes.c_uint64, sz, p]
    return L


def bf16_exact(x):
    """Nearest bfloat16 (ties to even), choosing among neighbouring bf16
    patterns by exact rational distance."""
    from fractions import Fraction
    out = np.empty(x.shape, dtype=np.uint16)
    for i, v in enumerate(x.tolist()):
        b = int(np.array([v], dtype=np.float32).view(np.uint32)[0]) >> 16
        sign = b & 0x8000
        best = None
        for c in range(max(0, (b & 0x7FFF) - 2), (b & 0x7FFF) + 3):
            c |= sign
            cv = float(np.array([c << 16], dtype=np.uint32).view(np.float32)[0])
            key = (abs(Fraction(cv) - Fraction(v)), c & 1)
            if best is None or key < best[0]:
                best = (key, c)
        out[i] = best[1]
    return out


def test_bf16_rounding_is_nearest_even():
    L = _lib()
    rng = np.random.default_rng(0)
    x = np.concatenate([rng.normal(0, 3, 20000), rng.normal(0, 1e-30, 200),
                        # exact ties between two bf16 values
                        (np.arange(1, 200) * 2 + 1) * 2.0 ** -8 + 1.0,
                        -((np.arange(1, 200) * 2 + 1) * 2.0 ** -8 + 1.0)])
    out = np.empty(x.shape, dtype=np.uint16)
    L.synth_bf16_array(x.ctypes.data, x.size, out.ctypes.data)
    np.testing.assert_array_equal(out, bf16_exact(x))


def test_ln_and_cos_series_accuracy():
    L = _lib()
    rng = np.random.default_rng(1)
    u = np.concatenate([rng.random(100000), 2.0 ** -np.arange(1, 54), [1.0]])
    u = u[u > 0]
    ln = np.empty_like(u)
    L.synth_ln_array(u.ctypes.data, u.size, ln.ctypes.data)
    ref = np.log(u)
    assert np.max(np.abs(ln - ref) / np.maximum(np.abs(ref), 1e-300)) < 1e-15
    assert ln[-1] == 0.0
    t = rng.random(100000)
    c = np.empty_like(t)
    L.synth_cos_turn_array(t.ctypes.data, t.size, c.ctypes.data)
    assert np.max(np.abs(c - np.cos(2 * np.pi * t))) < 2e-15


def test_normal_moments_and_independence():
    L = _lib()
    n = 400000
    x = np.empty(n)
    L.synth_normal_array(7, synth.T_Q, 0, n, x.ctypes.data)
    assert abs(x.mean()) < 0.01 and abs(x.var() - 1) < 0.01
    assert abs(np.mean(x ** 3)) < 0.02 and abs(np.mean(x ** 4) - 3) < 0.05
    assert abs(np.corrcoef(x[:-1], x[1:])[0, 1]) < 0.01
    y = np.empty(n)
    L.synth_normal_array(8, synth.T_Q, 0, n, y.ctypes.data)
    assert abs(np.corrcoef(x, y)[0, 1]) < 0.01
    z = np.empty(n)
    L.synth_normal_array(7, synth.T_Q, 0, n, z.ctypes.data)
    assert np.array_equal(x, z)


def test_maturation_law():
    """K_d - K_R has std (1-d/R)^3, V_d - V_R has std (1-d/R)^1.5, d = R is X_R."""
    R, D = 32, 128
    for is_v, tensor, power in [(0, synth.T_KCACHE, 3.0), (1, synth.T_VCACHE, 1.5)]:
        base = synth.bf16_bits_to_float(synth.matured_block(3, tensor, is_v, R, R, 0, 0, 0, 2000, 0, 2, D))
        for d in (1, 4, 16):
            xd = synth.bf16_bits_to_float(synth.matured_block(3, tensor, is_v, d, R, 0, 0, 0, 2000, 0, 2, D))
            diff = (xd.astype(np.float64) - base).ravel()
            c = (1 - d / R) ** power
            assert abs(diff.std() / c - 1) < 0.03
        assert abs(base.std() - 1) < 0.02


def test_workload_lengths():
    b = wl_mod.WORKLOADS["batched"]
    P, T = b.prefix_lens(), b.block_lens()
    assert P.min() >= 1024 and P.max() <= 8192 and len(set(P.tolist())) > 8
    assert set(T.tolist()) <= {4, 8, 16} and len(set(T.tolist())) >= 2
    assert np.array_equal(P, b.prefix_lens())
    assert wl_mod.WORKLOADS["long"].prefix_bytes_per_layer() == 512 * 2 ** 20
    assert wl_mod.WORKLOADS["decode"].prefix_bytes_per_layer() == 64 * 2 ** 20
