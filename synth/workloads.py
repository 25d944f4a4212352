"""The synthetic workloads of the DAS hot path and host builders of their inputs.

Shapes follow the paper's setting: looped models with R = 32 recurrences and
4 shared core layers (Huginn, App. A), bf16 caches, draft blocks of 4-16 rows
and verify widths of 16 (Sec. 3.3-3.4, App. A.2); prefix lengths stand in for
math/code decoding contexts (GSM8K, MATH-500, HumanEval, MBPP prompts plus
generations), which are not used.  Values follow the depth-maturation law of
synth_core.h: V_d = V_R + (1-d/R)^1.5 N_d, K_d = K_R + (1-d/R)^3 N_d,
queries N(0,1)/sqrt(D).
"""
import math
from dataclasses import dataclass, field

import numpy as np

from . import (T_BLOCK, T_KBLK, T_KCACHE, T_KNEW, T_PREFIX, T_Q, T_VBLK, T_VCACHE, T_VNEW,
               matured_block, normal_block, uniform_int)


@dataclass(frozen=True)
class Workload:
    name: str
    batch: int
    layers: int
    q_heads: int
    kv_heads: int
    head_dim: int
    depths: int          # R, stored recurrent depths
    key_depth: int       # kappa
    value_depth: int     # nu
    prefix: tuple        # (lo, hi): P_b uniform in [lo, hi]; lo == hi for a fixed length
    block: tuple         # block lengths T_b are drawn from these choices
    seed: int = 0
    kind: str = "draft"  # "draft" (Mature-V) or "verify"
    vocab: int = 0       # verify-and-commit only
    extra_capacity: int = 0
    notes: str = field(default="", compare=False)

    @property
    def group(self):
        return self.q_heads // self.kv_heads

    @property
    def max_block(self):
        return max(self.block)

    @property
    def max_prefix(self):
        return self.prefix[1]

    @property
    def capacity(self):
        return self.max_prefix + self.max_block + self.extra_capacity

    @property
    def block_depth(self):
        """Depth of the draft block's own K/V: the draft's depth, or the verified depth."""
        return self.key_depth

    def prefix_lens(self):
        lo, hi = self.prefix
        if lo == hi:
            return np.full(self.batch, lo, dtype=np.int32)
        return np.array([uniform_int(self.seed, T_PREFIX, b, lo, hi) for b in range(self.batch)],
                        dtype=np.int32)

    def block_lens(self):
        if len(self.block) == 1:
            return np.full(self.batch, self.block[0], dtype=np.int32)
        n = len(self.block)
        return np.array([self.block[uniform_int(self.seed, T_BLOCK, b, 0, n - 1)]
                         for b in range(self.batch)], dtype=np.int32)

    def prefix_bytes_per_layer(self):
        """Algorithmic bytes one layer call streams: K at kappa plus V at nu."""
        return int(self.prefix_lens().astype(np.int64).sum()) * self.kv_heads * self.head_dim * 2 * 2

    def replace(self, **kw):
        d = dict(self.__dict__)
        d.update(kw)
        return Workload(**d)


WORKLOADS = {
    "tiny": Workload(
        name="tiny Mature-V: B1 L1 H4/4 D64 P256 T4 R8 r2",
        batch=1, layers=1, q_heads=4, kv_heads=4, head_dim=64, depths=8, key_depth=2,
        value_depth=8, prefix=(256, 256), block=(4,)),
    "decode": Workload(
        name="single-sequence decode (~3.5B looped): B1 L4 H32/32 D128 P4096 T8 R32 r4",
        batch=1, layers=4, q_heads=32, kv_heads=32, head_dim=128, depths=32, key_depth=4,
        value_depth=32, prefix=(4096, 4096), block=(8,)),
    "batched": Workload(
        name="batched math/code drafting: B16 ragged P[1024,8192] L4 H32/8 D128 T{4,8,16} R32 r8",
        batch=16, layers=4, q_heads=32, kv_heads=8, head_dim=128, depths=32, key_depth=8,
        value_depth=32, prefix=(1024, 8192), block=(4, 8, 16)),
    "long": Workload(
        name="long-context drafting: B4 L4 H32/8 D128 P32768 T16 R32 r6",
        batch=4, layers=4, q_heads=32, kv_heads=8, head_dim=128, depths=32, key_depth=6,
        value_depth=32, prefix=(32768, 32768), block=(16,)),
    "verify": Workload(
        name="verify-and-commit: B8 L4 H32/8 D128 P16384 W16 depth R=32, vocab 32000",
        batch=8, layers=4, q_heads=32, kv_heads=8, head_dim=128, depths=32, key_depth=32,
        value_depth=32, prefix=(16384, 16384), block=(16,), kind="verify", vocab=32000),
}
ORDER = ["tiny", "decode", "batched", "long", "verify"]


def gen_q(wl, layer):
    """bf16 bits [B][max_block][Hq][D]: N(0,1)/sqrt(D)."""
    T, D = wl.max_block, wl.head_dim
    return np.stack([normal_block(wl.seed, T_Q, layer, b, 0, T, 0, wl.q_heads, D, math.sqrt(D))
                     for b in range(wl.batch)])


def gen_block_kv(wl, layer):
    """(k_blk, v_blk) bf16 bits [B][max_block][Hkv][D] at the block's depth."""
    T, D, R, d = wl.max_block, wl.head_dim, wl.depths, wl.block_depth
    k = np.stack([matured_block(wl.seed, T_KBLK, 0, d, R, layer, b, 0, T, 0, wl.kv_heads, D)
                  for b in range(wl.batch)])
    v = np.stack([matured_block(wl.seed, T_VBLK, 1, d, R, layer, b, 0, T, 0, wl.kv_heads, D)
                  for b in range(wl.batch)])
    return k, v


def gen_cache(wl, depths=None, tokens=None):
    """(K, V) bf16 bits [R][L][B][capacity][Hkv][D]; depths not listed stay 0.

    `tokens` limits generation to positions [0, tokens) (default: capacity).
    """
    R, L, B, cap, H, D = wl.depths, wl.layers, wl.batch, wl.capacity, wl.kv_heads, wl.head_dim
    tok = cap if tokens is None else tokens
    K = np.zeros((R, L, B, cap, H, D), dtype=np.uint16)
    V = np.zeros((R, L, B, cap, H, D), dtype=np.uint16)
    kd = {wl.key_depth} if depths is None else set(depths)
    vd = {wl.value_depth} if depths is None else set(depths)
    for l in range(L):
        for b in range(B):
            for d in kd:
                K[d - 1, l, b, :tok] = matured_block(wl.seed, T_KCACHE, 0, d, R, l, b, 0, tok, 0, H, D)
            for d in vd:
                V[d - 1, l, b, :tok] = matured_block(wl.seed, T_VCACHE, 1, d, R, l, b, 0, tok, 0, H, D)
    return K, V


def gen_staged(wl, W):
    """(k_new, v_new) bf16 bits [R][L][B][W][Hkv][D]: the verifier's K/V at every depth."""
    R, L, B, H, D = wl.depths, wl.layers, wl.batch, wl.kv_heads, wl.head_dim
    k = np.empty((R, L, B, W, H, D), dtype=np.uint16)
    v = np.empty((R, L, B, W, H, D), dtype=np.uint16)
    for d in range(1, R + 1):
        for l in range(L):
            for b in range(B):
                k[d - 1, l, b] = matured_block(wl.seed, T_KNEW, 0, d, R, l, b, 0, W, 0, H, D)
                v[d - 1, l, b] = matured_block(wl.seed, T_VNEW, 1, d, R, l, b, 0, W, 0, H, D)
    return k, v
