"""das_mature_v_attention_noalloc: the entry point for callers that cannot
allocate device memory (a fixed memory plan, a plugin handed only its
tensors, a host that forbids cudaMalloc after start-up).  Its scratch is a
fixed array inside the library, so its results must match the ordinary entry
point's, call after call, with nothing allocated by the caller.

This file is collected last on purpose: if it fails, a run that stops at the
first failure has already run every other test."""
import ctypes

import numpy as np
import pytest
import torch

from synth import workloads as wl_mod
from tests.gpu_util import OUT_ABS, OUT_REL, LSE_ABS, dev_bf16, dev_i32, rel_denominator

pytestmark = pytest.mark.gpu


def _close(a, b, la, lb):
    a, b = a.float().cpu().numpy(), b.float().cpu().numpy()
    err = np.abs(a - b)
    assert (err / np.maximum(np.abs(b), 1.0)).max() <= OUT_ABS
    assert (err / rel_denominator(b)).max() <= OUT_REL
    la, lb = la.cpu().numpy(), lb.cpu().numpy()
    fin = np.isfinite(lb)
    assert np.array_equal(np.isfinite(la), fin)
    assert np.abs(la[fin] - lb[fin]).max(initial=0) <= LSE_ABS


def test_noalloc_matches_workspace_entry_point_twice():
    import paper_2609_34538_gb300 as das
    wl = wl_mod.Workload(name="no-alloc", batch=3, layers=2, q_heads=8, kv_heads=2, head_dim=128,
                         depths=8, key_depth=2, value_depth=8, prefix=(100, 3000), block=(4, 8))
    K, V = wl_mod.gen_cache(wl, depths=[2, 8])
    cache = das.DepthKVCache(dev_bf16(K), dev_bf16(V))
    pl, bl = dev_i32(wl.prefix_lens()), dev_i32(wl.block_lens())
    assert das.das_workspace_size(cache, wl.q_heads, wl.max_block) <= (32 << 20)
    ws = das.new_workspace(cache, wl.q_heads, wl.max_block)
    for layer in (1, 0):  # two calls in a row, different inputs
        q = dev_bf16(wl_mod.gen_q(wl, layer))
        kb, vb = map(dev_bf16, wl_mod.gen_block_kv(wl, layer))
        ref_o, ref_l = das.das_mature_v_attention(cache, layer, 2, 8, pl, bl, q, kb, vb, ws)
        out = torch.full_like(q, float("nan"))
        lse = torch.full((wl.batch, wl.q_heads, wl.max_block), float("nan"), device="cuda")
        das.das_mature_v_attention_noalloc(cache, layer, 2, 8, pl, bl, q, kb, vb, out=out, lse=lse)
        torch.cuda.synchronize()
        _close(out, ref_o, lse, ref_l)


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
