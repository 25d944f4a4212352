"""Helpers shared by the GPU tests: device upload of generator output, the
oracle comparison and the tolerance of the float outputs."""
import numpy as np
import torch

import oracle
import synth
from synth import workloads as wl_mod

# Tolerances: bf16 outputs max abs 1e-2 (relative to max(1, |o|) above 1,
# where bf16 spacing alone exceeds it) and max rel 1e-2, fp32 LSE max abs
# 1e-4.  The relative error of an element is taken against the larger of its
# own magnitude and the RMS of its reference row (the head_dim values of one
# query row): the kernel rounds the softmax weights P to bf16 for the tensor-
# core P.V product (relative error <= 2^-9 per weight), which perturbs an
# output by a fraction of the row's scale, not of the element itself.
OUT_ABS, OUT_REL, LSE_ABS = 1e-2, 1e-2, 1e-4


def rel_denominator(o):
    rms = np.sqrt(np.mean(np.square(o), axis=-1, keepdims=True))
    return np.maximum(np.abs(o), np.maximum(rms, 1e-30))


def dev_bf16(bits):
    a = np.ascontiguousarray(bits, dtype=np.uint16).view(np.int16)
    return torch.from_numpy(a).view(torch.bfloat16).cuda()


def dev_i32(x):
    return torch.from_numpy(np.ascontiguousarray(x, dtype=np.int32)).cuda()


def host_bits(t):
    return t.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def assert_close(out_gpu, out_ref, lse_gpu=None, lse_ref=None, where=""):
    g = np.asarray(out_gpu, dtype=np.float64)
    o = np.asarray(out_ref, dtype=np.float64)
    assert np.all(np.isfinite(g)), f"non-finite output {where}"
    err = np.abs(g - o)
    rel = err / rel_denominator(o)
    # abs error against max(1, |o|): bf16 spacing alone is 2^-7 at |o| = 2
    scaled = err / np.maximum(np.abs(o), 1.0)
    assert scaled.max(initial=0) <= OUT_ABS, f"max abs {err.max():.3e} {where}"
    assert rel.max(initial=0) <= OUT_REL, f"max rel {rel.max():.3e} {where}"
    if lse_gpu is not None:
        lg = np.asarray(lse_gpu, dtype=np.float64)
        lo = np.asarray(lse_ref, dtype=np.float64)
        inf = np.isneginf(lo)
        assert np.array_equal(np.isneginf(lg), inf), f"lse -inf pattern differs {where}"
        d = np.abs(lg[~inf] - lo[~inf])
        assert d.max(initial=0) <= LSE_ABS, f"lse max abs {d.max(initial=0):.3e} {where}"


def run_small(wl, layer=0, key_depth=None, value_depth=None, prefix=None, block=None,
              scale=0.0, poison_tail=False, verify=False):
    """Run one attention call on host-generated inputs and compare with the
    oracle.  Returns (out, lse, workspace) from the GPU."""
    import paper_2609_34538_gb300 as das
    kap = wl.key_depth if key_depth is None else key_depth
    nu = wl.value_depth if value_depth is None else value_depth
    pl = wl.prefix_lens() if prefix is None else np.asarray(prefix, dtype=np.int32)
    bl = wl.block_lens() if block is None else np.asarray(block, dtype=np.int32)
    K, V = wl_mod.gen_cache(wl, depths=sorted({kap, nu}))
    if poison_tail:  # positions past the prefix hold NaN: they must never be used
        for b in range(wl.batch):
            K[:, :, b, pl[b]:] = 0x7FC0
            V[:, :, b, pl[b]:] = 0x7FC0
    q = wl_mod.gen_q(wl, layer)
    kb, vb = wl_mod.gen_block_kv(wl, layer)
    if poison_tail:
        for b in range(wl.batch):
            kb[b, bl[b]:] = 0x7FC0
            vb[b, bl[b]:] = 0x7FC0
            q[b, bl[b]:] = 0x7FC0
    ref_o, ref_l = oracle.attention(K, V, layer, kap, nu, pl, bl, q, kb, vb,
                                    scale=scale if scale > 0 else None)
    cache = das.DepthKVCache(dev_bf16(K), dev_bf16(V))
    ws = das.new_workspace(cache, wl.q_heads, wl.max_block)
    args = (dev_i32(pl), dev_i32(bl), dev_bf16(q), dev_bf16(kb), dev_bf16(vb), ws)
    if verify:
        assert kap == nu
        out, lse = das.das_verify_attention(cache, layer, kap, *args, softmax_scale=scale)
    else:
        out, lse = das.das_mature_v_attention(cache, layer, kap, nu, *args, softmax_scale=scale)
    torch.cuda.synchronize()
    assert_close(out.float().cpu().numpy(), ref_o, lse.cpu().numpy(), ref_l,
                 where=f"[{wl.name} layer {layer} kappa {kap} nu {nu}]")
    return out, lse, ws
