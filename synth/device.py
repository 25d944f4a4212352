"""Full-size synthetic inputs built in device memory.

The cache of a workload is allocated in its real layout,
[depths][layers][batch][capacity][kv_heads][head_dim] bf16 for K and V, and
filled on the GPU: depths that a call reads get the exact generator values
(bit-identical to the host generator), the other depths cheap filler.  Small
per-call tensors (queries, block K/V, lengths, logits) come from the host
generator.
"""
import numpy as np
import torch

from . import T_KCACHE, T_KNEW, T_VCACHE, T_VNEW, dev_lib
from . import accept_inputs
from .workloads import gen_block_kv, gen_q


def _check(rc, what):
    if rc != 0:
        raise RuntimeError(f"{what}: CUDA error {rc}")


def _stream():
    return torch.cuda.current_stream().cuda_stream


def fill_matured(t, seed, tensor, is_value, depth, R):
    """t: bf16 [layers][batch][positions][heads][D] slab of stored depth `depth`."""
    L, B, cap, H, D = t.shape
    _check(dev_lib().synth_dev_fill_matured(t.data_ptr(), seed, tensor, is_value, depth, R, L, B,
                                            cap, H, D, _stream()), "fill_matured")


def fill_filler(t, seed):
    _check(dev_lib().synth_dev_fill_filler(t.data_ptr(), t.numel(), seed, _stream()),
           "fill_filler")


def build_cache(wl, key_depths=None, value_depths=None, device="cuda"):
    """(K, V) on the device; exact values at the given depths (default: the
    workload's kappa for K and nu for V), filler elsewhere."""
    kd = {wl.key_depth} if key_depths is None else set(key_depths)
    vd = {wl.value_depth} if value_depths is None else set(value_depths)
    shape = (wl.depths, wl.layers, wl.batch, wl.capacity, wl.kv_heads, wl.head_dim)
    K = torch.empty(shape, dtype=torch.bfloat16, device=device)
    V = torch.empty(shape, dtype=torch.bfloat16, device=device)
    for d in range(1, wl.depths + 1):
        if d in kd:
            fill_matured(K[d - 1], wl.seed, T_KCACHE, 0, d, wl.depths)
        else:
            fill_filler(K[d - 1], wl.seed * 1000 + d)
        if d in vd:
            fill_matured(V[d - 1], wl.seed, T_VCACHE, 1, d, wl.depths)
        else:
            fill_filler(V[d - 1], wl.seed * 1000 + 100 + d)
    return K, V


def build_staged(wl, W, device="cuda"):
    """The verifier's K/V of W inputs at every depth: [R][L][B][W][Hkv][D] each."""
    shape = (wl.depths, wl.layers, wl.batch, W, wl.kv_heads, wl.head_dim)
    kn = torch.empty(shape, dtype=torch.bfloat16, device=device)
    vn = torch.empty(shape, dtype=torch.bfloat16, device=device)
    for d in range(1, wl.depths + 1):
        fill_matured(kn[d - 1], wl.seed, T_KNEW, 0, d, wl.depths)
        fill_matured(vn[d - 1], wl.seed, T_VNEW, 1, d, wl.depths)
    return kn, vn


def upload_bf16(bits, device="cuda"):
    a = np.ascontiguousarray(bits, dtype=np.uint16).view(np.int16)
    return torch.from_numpy(a).view(torch.bfloat16).to(device)


def layer_inputs(wl, layer, device="cuda"):
    """(q, k_blk, v_blk) of one layer call, on the device."""
    q = upload_bf16(gen_q(wl, layer), device)
    kb, vb = gen_block_kv(wl, layer)
    return q, upload_bf16(kb, device), upload_bf16(vb, device)


def accept_tensors(wl, device="cuda"):
    """(accept_star, draft int32 [B][W], logits fp32 [B][W][vocab]) on the device."""
    a, d, lg = accept_inputs(wl.seed, wl.batch, wl.max_block, wl.vocab)
    return a, torch.from_numpy(d).to(device), torch.from_numpy(lg).to(device)
