"""Helpers shared by the GPU tests: device upload of generator output, the
oracle comparison and the tolerance of the float outputs."""
import json
import os

import numpy as np
import torch

import oracle
import synth
from synth import workloads as wl_mod

# Tolerances (stated for the method's bf16 outputs and fp32 lse): every
# element's raw error |g - o| <= 1e-2, plus half a bf16 ulp of |o| where
# |o| >= 4 (there the rounding of the output to bf16 alone, up to half an ulp
# = 2^-6 in [4, 8), can exceed 1e-2; below 4 it is at most 2^-7 in [2, 4),
# under 1e-2, and the raw bound holds as stated); relative error <= 1e-2 against the larger
# of |o| and the RMS of the reference row (the head_dim values of one query
# row: the kernel rounds the softmax weights P to bf16 for the tensor-core
# P.V product, relative error <= 2^-9 per weight, which perturbs an output by
# a fraction of the row's scale, not of the element); lse max abs 1e-4.
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


def half_ulp_bf16(o):
    """Half the bf16 spacing at |o| (8 significant bits): 2^(e - 8) for |o| in
    [2^e, 2^(e+1)); 0 at 0."""
    a = np.abs(np.asarray(o, dtype=np.float64))
    e = np.floor(np.log2(np.where(a > 0, a, 1.0)))
    return np.where(a > 0, np.exp2(e - 8), 0.0)


def abs_bound(o):
    """Allowed raw error per element: 1e-2, plus half a bf16 ulp where |o| >= 4."""
    return OUT_ABS + np.where(np.abs(o) >= 4.0, half_ulp_bf16(o), 0.0)


def parity_errors(out_gpu, out_ref, lse_gpu=None, lse_ref=None):
    """(max raw abs error, max relative error, max lse error or None)."""
    g = np.asarray(out_gpu, dtype=np.float64)
    o = np.asarray(out_ref, dtype=np.float64)
    err = np.abs(g - o)
    lse_err = None
    if lse_gpu is not None:
        lg = np.asarray(lse_gpu, dtype=np.float64)
        lo = np.asarray(lse_ref, dtype=np.float64)
        fin = ~np.isneginf(lo)
        lse_err = float(np.abs(lg[fin] - lo[fin]).max(initial=0.0))
    return float(err.max(initial=0.0)), float((err / rel_denominator(o)).max(initial=0.0)), lse_err


def record_parity(where, abs_err, rel_err, lse_err):
    """Print one parity case's measured errors; with PARITY_LOG set, also
    append them as a JSON line to that file."""
    print(f"parity {where}: max abs {abs_err:.3e} max rel {rel_err:.3e} "
          f"lse {lse_err if lse_err is None else f'{lse_err:.3e}'}")
    path = os.environ.get("PARITY_LOG")
    if path:
        with open(path, "a") as f:
            f.write(json.dumps({"case": where, "max_abs": abs_err, "max_rel": rel_err,
                                "lse_max_abs": lse_err}) + "\n")


def assert_close(out_gpu, out_ref, lse_gpu=None, lse_ref=None, where=""):
    g = np.asarray(out_gpu, dtype=np.float64)
    o = np.asarray(out_ref, dtype=np.float64)
    assert np.all(np.isfinite(g)), f"non-finite output {where}"
    err = np.abs(g - o)
    a, r, le = parity_errors(g, o, lse_gpu, lse_ref)
    record_parity(where, a, r, le)
    worst = np.unravel_index(np.argmax(err - abs_bound(o)), err.shape) if err.size else ()
    assert np.all(err <= abs_bound(o)), \
        f"max abs {a:.3e} (worst over bound at {worst}: |o| = {abs(o[worst]) if err.size else 0:.3f}) {where}"
    assert r <= OUT_REL, f"max rel {r:.3e} {where}"
    if lse_gpu is not None:
        lg = np.asarray(lse_gpu, dtype=np.float64)
        lo = np.asarray(lse_ref, dtype=np.float64)
        inf = np.isneginf(lo)
        assert np.array_equal(np.isneginf(lg), inf), f"lse -inf pattern differs {where}"
        assert le <= LSE_ABS, f"lse max abs {le:.3e} {where}"


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
    # no wait ran out (attention pipeline or the merge's partial counters)
    assert das.workspace_status(ws) & 1 == 0
    return out, lse, ws
