"""das_mature_v_attention_noalloc: the entry point for callers that cannot
allocate device memory when they call (a serving loop with a fixed memory
plan, a plugin handed only its tensors, a host that forbids cudaMalloc after
start-up).  Its split-K scratch is a fixed array inside the library, so its
results must match the fp64 oracle within the parity tolerance, and the
ordinary (workspace) entry point's, call after call, with nothing allocated
by the caller; its status word must stay clean.

This file is collected last on purpose: if it fails, a run that stops at the
first failure has already run every other test."""
import ctypes

import numpy as np
import pytest
import torch

import oracle
from synth import workloads as wl_mod
from tests.gpu_util import (LSE_ABS, assert_close, dev_bf16, dev_i32, parity_errors,
                            record_parity)

pytestmark = pytest.mark.gpu


def test_noalloc_matches_oracle_and_workspace_entry_point_twice():
    import paper_2609_34538_gb300 as das
    wl = wl_mod.Workload(name="no-alloc", batch=3, layers=2, q_heads=8, kv_heads=2, head_dim=128,
                         depths=8, key_depth=2, value_depth=8, prefix=(100, 3000), block=(4, 8))
    K, V = wl_mod.gen_cache(wl, depths=[2, 8])
    P, T = wl.prefix_lens(), wl.block_lens()
    cache = das.DepthKVCache(dev_bf16(K), dev_bf16(V))
    pl, bl = dev_i32(P), dev_i32(T)
    assert das.das_workspace_size(cache, wl.q_heads, wl.max_block) <= (32 << 20)
    ws = das.new_workspace(cache, wl.q_heads, wl.max_block)
    for layer in (1, 0):  # two calls in a row, different inputs
        qh = wl_mod.gen_q(wl, layer)
        kbh, vbh = wl_mod.gen_block_kv(wl, layer)
        q, kb, vb = dev_bf16(qh), dev_bf16(kbh), dev_bf16(vbh)
        ro, rl = oracle.attention(K, V, layer, 2, 8, P, T, qh, kbh, vbh)
        wo, wlse = das.das_mature_v_attention(cache, layer, 2, 8, pl, bl, q, kb, vb, ws)
        out = torch.full_like(q, float("nan"))
        lse = torch.full((wl.batch, wl.q_heads, wl.max_block), float("nan"), device="cuda")
        das.das_mature_v_attention_noalloc(cache, layer, 2, 8, pl, bl, q, kb, vb, out=out, lse=lse)
        torch.cuda.synchronize()
        assert das.noalloc_status() == 0
        o, l = out.float().cpu().numpy(), lse.cpu().numpy()
        assert_close(o, ro, l, rl, where=f"[no-alloc vs oracle, layer {layer}]")
        # against the workspace entry point: the same kernels on the same inputs
        a, r, le = parity_errors(o, wo.float().cpu().numpy(), l, wlse.cpu().numpy())
        record_parity(f"[no-alloc vs workspace entry point, layer {layer}]", a, r, le)
        assert a <= 1e-2 and r <= 1e-2 and le <= LSE_ABS
        assert np.array_equal(np.isneginf(l), np.isneginf(wlse.cpu().numpy()))
    assert das.workspace_status(ws) == 0


def test_noalloc_rejects_mismatched_outputs_before_launch():
    import paper_2609_34538_gb300 as das
    wl = wl_mod.Workload(name="no-alloc", batch=2, layers=1, q_heads=4, kv_heads=2, head_dim=64,
                         depths=2, key_depth=1, value_depth=2, prefix=(10, 10), block=(4,))
    cache = das.DepthKVCache.empty(2, 1, 2, wl.capacity, 2, 64)
    pl, bl = dev_i32(wl.prefix_lens()), dev_i32(wl.block_lens())
    q = torch.zeros((2, 4, 4, 64), dtype=torch.bfloat16, device="cuda")
    kb = torch.zeros((2, 4, 2, 64), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(ValueError):  # out not shaped like q
        das.das_mature_v_attention_noalloc(cache, 0, 1, 2, pl, bl, q, kb, kb,
                                           out=torch.empty_like(q[:1]))
    with pytest.raises(ValueError):  # lse not [B][Hq][max_block]
        das.das_mature_v_attention_noalloc(cache, 0, 1, 2, pl, bl, q, kb, kb,
                                           lse=torch.empty((2, 4, 3), device="cuda"))
    with pytest.raises(ValueError):  # block K/V not [B][max_block][Hkv][D]
        das.das_mature_v_attention_noalloc(cache, 0, 1, 2, pl, bl, q, kb[:, :3], kb)


def test_noalloc_rejects_shapes_beyond_its_scratch():
    import paper_2609_34538_gb300 as das
    # a descriptor only: the size check returns before anything is read or launched
    big = das.das_kv_cache(256, 256, 2, 1, 1000, 64, 8, 128)
    need = das.LIB.das_workspace_size(ctypes.byref(big), 32, 16)
    assert need > (32 << 20)
    null = ctypes.c_void_p(256)
    rc = das.LIB.das_mature_v_attention_noalloc(ctypes.byref(big), 0, 1, 2, null, null, 16, null,
                                                null, null, 32, 0.0, null, null, ctypes.c_void_p(0))
    assert rc == das.DAS_ERR_WORKSPACE
