"""The e4m3 cache variant (depths below R stored as 8-bit floats; not in the
paper): das_mature_v_attention_f8 against the oracle on the stored values,
for every combination of e4m3 / bf16 keys and values, and das_kv_append_f8
bit-exact against the oracle's rounding."""
import numpy as np
import pytest
import torch

import oracle
import synth
from synth import workloads as wl_mod
from tests.gpu_util import assert_close, dev_bf16, dev_i32, host_bits

pytestmark = pytest.mark.gpu


def small(**kw):
    base = dict(name="f8", batch=2, layers=2, q_heads=8, kv_heads=2, head_dim=128, depths=6,
                key_depth=2, value_depth=6, prefix=(700, 700), block=(8,))
    base.update(kw)
    return wl_mod.Workload(**base)


def host_f8_cache(wl):
    R = wl.depths
    K, V = wl_mod.gen_cache(wl, depths=[R])
    low = (R - 1, wl.layers, wl.batch, wl.capacity, wl.kv_heads, wl.head_dim)
    return (K[R - 1].copy(), V[R - 1].copy(), synth.e4m3_codes(wl.seed, synth.T_KLOW, low),
            synth.e4m3_codes(wl.seed, synth.T_VLOW, low))


def every_code(shape, shift):
    """Codes cycling through all 254 finite e4m3 codes (subnormals included)."""
    finite = np.array([c for c in range(256) if c not in (0x7F, 0xFF)], dtype=np.uint8)
    n = int(np.prod(shape))
    return finite[(np.arange(n) * 7 + shift) % finite.size].reshape(shape)


def ranged_q(q):
    """Query rows over a range of magnitudes, exactly in bf16: row (b, i, h)
    scaled by 2^k, k cycling through -8..3; every third row's odd elements
    scaled by a further 2^-12 (far below the row's largest element); one row
    of zeros per sequence."""
    x = synth.bf16_bits_to_float(q).astype(np.float64)
    B, T, H, D = x.shape
    for b in range(B):
        for i in range(T):
            for h in range(H):
                r = (b * T + i) * H + h
                x[b, i, h] *= 2.0 ** (r % 12 - 8)
                if r % 3 == 0:
                    x[b, i, h, 1::2] *= 2.0 ** -12
        x[b, 0, H - 1] = 0.0
    bits = (x.astype(np.float32).view(np.uint32) >> 16).astype(np.uint16)
    assert np.array_equal(synth.bf16_bits_to_float(bits), x.astype(np.float32))  # exact
    return bits


def run_f8(wl, kap, nu, layer=1, prefix=None, block=None, poison_tail=False, scale=0.0,
           all_codes=False, zero_q=False, q_fn=None):
    import paper_2609_34538_gb300 as das
    kt, vt, kl, vl = host_f8_cache(wl)
    if all_codes:
        kl, vl = every_code(kl.shape, 0), every_code(vl.shape, 101)
    pl = wl.prefix_lens() if prefix is None else np.asarray(prefix, np.int32)
    bl = wl.block_lens() if block is None else np.asarray(block, np.int32)
    if poison_tail:  # positions past the prefix hold NaN: never read
        for b in range(wl.batch):
            kl[:, :, b, pl[b]:] = 0x7F
            vl[:, :, b, pl[b]:] = 0x7F
            kt[:, b, pl[b]:] = 0x7FC0
            vt[:, b, pl[b]:] = 0x7FC0
    q = wl_mod.gen_q(wl, layer)
    if zero_q:
        q = np.zeros_like(q)
    if q_fn is not None:
        q = q_fn(q)
    kb, vb = wl_mod.gen_block_kv(wl, layer)
    ref_o, ref_l = oracle.attention_f8(kt, vt, kl, vl, layer, kap, nu, pl, bl, q, kb, vb,
                                       scale=scale if scale > 0 else None)
    up8 = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()
    cache = das.DepthKVCacheF8(dev_bf16(kt), dev_bf16(vt), up8(kl), up8(vl))
    ws = das.new_workspace_f8(cache, wl.q_heads, wl.max_block)
    out, lse = das.das_mature_v_attention_f8(cache, layer, kap, nu, dev_i32(pl), dev_i32(bl),
                                             dev_bf16(q), dev_bf16(kb), dev_bf16(vb), ws,
                                             softmax_scale=scale)
    torch.cuda.synchronize()
    assert_close(out.float().cpu().numpy(), ref_o, lse.cpu().numpy(), ref_l,
                 where=f"[f8 kappa {kap} nu {nu}]")
    assert das.workspace_status(ws) == 0


@pytest.mark.parametrize("kap,nu", [(2, 6), (3, 3), (6, 2), (6, 6), (1, 5)])
def test_read_policies_on_e4m3_cache(kap, nu):
    """Mature-V (e4m3 keys, bf16 values), a low-depth verify (both e4m3),
    Deep K (bf16 keys, e4m3 values), Deep K/V (both bf16) and another
    e4m3-key case."""
    run_f8(small(), kap, nu)


@pytest.mark.parametrize("P", [0, 1, 63, 64, 65, 1000])
def test_prefix_lengths_e4m3(P):
    run_f8(small(prefix=(P, P)), 2, 6, prefix=[P, max(P - 1, 0)], block=[8, 5])


@pytest.mark.parametrize("D", [64, 128])
def test_head_dims_e4m3(D):
    run_f8(small(head_dim=D), 2, 6)
    run_f8(small(head_dim=D), 3, 3)


def test_nan_past_the_prefix_is_never_read_e4m3():
    run_f8(small(prefix=(300, 300)), 2, 6, prefix=[300, 129], block=[8, 3], poison_tail=True)
    run_f8(small(prefix=(300, 300)), 4, 4, prefix=[300, 129], block=[8, 3], poison_tail=True)


def test_every_e4m3_code_is_widened_exactly():
    """Keys and values that run through every finite code, subnormals and
    +-448 included.  e4m3 keys are checked through the scores; e4m3 values
    with zero queries, where every softmax weight is exactly 1 and each
    output is the mean of the stored values (with random queries, values of
    +-448 and random signs make the outputs small averages of large terms, and
    the bf16 rounding of the weights, relative to the values, dominates)."""
    run_f8(small(prefix=(1500, 1500)), 2, 6, all_codes=True)
    for kap, nu in [(6, 3), (4, 4), (2, 6)]:
        run_f8(small(prefix=(1500, 1500)), kap, nu, all_codes=True, zero_q=True)


def test_query_magnitudes_e4m3_keys():
    """e4m3 keys with bf16 values at D = 128 are scored by e4m3 products of
    the query split into two e4m3 parts under a per-row power of two: query
    rows over 2^-8..2^3, rows with elements 2^-12 of their largest, and zero
    rows, against the oracle on the bf16 queries."""
    run_f8(small(), 2, 6, q_fn=ranged_q)
    run_f8(small(), 2, 6, q_fn=ranged_q, scale=1.0)
    run_f8(small(head_dim=64), 2, 6, q_fn=ranged_q)


@pytest.mark.parametrize("kap,nu", [(2, 6), (3, 3)])
def test_ragged_batch_past_32_e4m3(kap, nu):
    """40 sequences of ragged prefixes 0..300 (some empty) and blocks of 0, 1
    or 8 rows: a CTA's range holds many segments, so both query buffers turn
    over many times (the split parts and every softmax warp's read of e are
    released through qempty), consecutive block tiles reuse the bf16 key
    buffer (bkfree), and the plan is made after the dependency wait (more than
    32 sequences)."""
    wl = small(batch=40, layers=1, q_heads=4, kv_heads=2, prefix=(0, 300), block=(0, 1, 8))
    P, T = wl.prefix_lens(), wl.block_lens()
    P[::7] = 0  # empty prefixes: pairs of a block tile alone
    assert (T == 0).any() and (T == 8).any()
    run_f8(wl, kap, nu, layer=0, prefix=P, block=T)


def test_split_across_many_ctas_e4m3():
    run_f8(small(batch=1, kv_heads=1, q_heads=4, prefix=(20000, 20000), block=(16,)), 2, 6)


def test_sharp_scale_e4m3():
    run_f8(small(), 2, 6, scale=1.0)


def test_append_e4m3_bit_exact():
    import paper_2609_34538_gb300 as das
    wl = small(batch=3, prefix=(40, 40), block=(8,))
    R, L, B, W = wl.depths, wl.layers, wl.batch, 6
    kt, vt, kl, vl = host_f8_cache(wl)
    kn = np.stack([synth.matured_block(wl.seed + 7, synth.T_KNEW, 0, d, R, l, b, 0, W, 0,
                                       wl.kv_heads, wl.head_dim)
                   for d in range(1, R + 1) for l in range(L) for b in range(B)])
    kn = kn.reshape(R, L, B, W, wl.kv_heads, wl.head_dim)
    vn = np.ascontiguousarray(kn[::-1])
    acc = np.array([0, 3, W], np.int32)
    pl = np.array([40, 10, 5], np.int32)
    ekt, evt, ekl, evl, epl, eflag = oracle.kv_append_f8(kt, vt, kl, vl, kn, vn, acc, pl)
    up8 = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()
    cache = das.DepthKVCacheF8(dev_bf16(kt), dev_bf16(vt), up8(kl), up8(vl))
    dpl, flag = dev_i32(pl), torch.zeros(1, dtype=torch.int32, device="cuda")
    das.das_kv_append_f8(cache, dev_bf16(kn), dev_bf16(vn), dev_i32(acc), dpl, flag)
    torch.cuda.synchronize()
    assert int(flag.item()) == eflag
    assert np.array_equal(dpl.cpu().numpy(), epl)
    assert np.array_equal(host_bits(cache.k_top), ekt) and np.array_equal(host_bits(cache.v_top), evt)
    assert np.array_equal(cache.k_low.cpu().numpy(), ekl)
    assert np.array_equal(cache.v_low.cpu().numpy(), evl)
