"""Full-size workloads, in the launch configuration the benchmark times: every
layer call runs on the real cache layout (all R depths allocated); sampled
(sequence, kv head) groups are recomputed by the oracle from host-generated
slabs, and every output is checked for the properties that hold at any size.
The device-filled cache is also checked bit for bit against the host
generator on the sampled slabs."""
import numpy as np
import pytest
import torch

import oracle
import synth
from synth import device as sdev
from synth import workloads as wl_mod
from tests.gpu_util import assert_close, dev_i32, host_bits

pytestmark = [pytest.mark.gpu, pytest.mark.slow]


def _pairs(wl, layer, n):
    """n distinct (sequence, kv head) pairs of the layer, seeded (all pairs if
    there are at most n)."""
    rng = np.random.default_rng(100 + layer)
    allp = [(b, h) for b in range(wl.batch) for h in range(wl.kv_heads)]
    if len(allp) <= n:
        return allp
    return [allp[i] for i in sorted(rng.choice(len(allp), size=n, replace=False))]


def _samples(wl):
    """Sampled pairs per layer: 16 where the oracle is quick (prefixes up to
    8192), 4 on the 16k and 32k prefixes."""
    return 4 if wl.max_prefix > 10000 else 16


@pytest.mark.parametrize("name", ["decode", "batched", "long", "verify"])
def test_full_size_sampled(name):
    import paper_2609_34538_gb300 as das
    wl = wl_mod.WORKLOADS[name]
    K, V = sdev.build_cache(wl)
    cache = das.DepthKVCache(K, V)
    ws = das.new_workspace(cache, wl.q_heads, wl.max_block)
    P, T = wl.prefix_lens(), wl.block_lens()
    pl, bl = dev_i32(P), dev_i32(T)
    G, D, R = wl.group, wl.head_dim, wl.depths
    try:
        for layer in range(wl.layers):
            q, kb, vb = sdev.layer_inputs(wl, layer)
            if wl.kind == "verify":
                out, lse = das.das_verify_attention(cache, layer, wl.key_depth, pl, bl, q, kb, vb, ws)
            else:
                out, lse = das.das_mature_v_attention(cache, layer, wl.key_depth, wl.value_depth,
                                                      pl, bl, q, kb, vb, ws)
            torch.cuda.synchronize()
            o = out.float().cpu().numpy()
            l = lse.cpu().numpy()
            assert np.all(np.isfinite(o))
            for b in range(wl.batch):
                assert np.all(o[b, T[b]:] == 0) and np.all(np.isneginf(l[b, :, T[b]:]))
                assert np.all(np.isfinite(l[b, :, :T[b]]))
            qh, kbh, vbh = host_bits(q), host_bits(kb), host_bits(vb)
            for b, h in _pairs(wl, layer, _samples(wl)):
                kp = synth.matured_block(wl.seed, synth.T_KCACHE, 0, wl.key_depth, R, layer, b, 0,
                                         int(P[b]), h, h + 1, D)
                vp = synth.matured_block(wl.seed, synth.T_VCACHE, 1, wl.value_depth, R, layer, b,
                                         0, int(P[b]), h, h + 1, D)
                # the device-filled cache holds exactly the host generator's values
                assert np.array_equal(host_bits(K[wl.key_depth - 1, layer, b, :P[b], h:h + 1]), kp)
                assert np.array_equal(host_bits(V[wl.value_depth - 1, layer, b, :P[b], h:h + 1]), vp)
                ro, rl = oracle.attend_seq(qh[b, :, h * G:(h + 1) * G], kp, vp,
                                           kbh[b, :, h:h + 1], vbh[b, :, h:h + 1],
                                           block_len=int(T[b]))
                assert_close(o[b, :, h * G:(h + 1) * G], ro, l[b, h * G:(h + 1) * G], rl,
                             where=f"[{name} layer {layer} b {b} kv head {h}]")
        assert das.workspace_status(ws) == 0
    finally:
        del cache, K, V
        torch.cuda.empty_cache()


def test_full_size_accept_and_append():
    """Verify-and-commit: accept over [8, 16, 32000] logits, then the append of
    accepted K/V at all 32 depths into the full cache; appended windows and the
    positions around them are compared byte for byte with the oracle."""
    import paper_2609_34538_gb300 as das
    wl = wl_mod.WORKLOADS["verify"]
    W = wl.max_block
    K, V = sdev.build_cache(wl, key_depths=[], value_depths=[])  # filler everywhere
    kn, vn = sdev.build_staged(wl, W)
    a_star, draft, logits = sdev.accept_tensors(wl)
    cache = das.DepthKVCache(K, V)
    P = wl.prefix_lens()
    pl = dev_i32(P)
    try:
        lo, hi = max(0, int(P.min()) - 2), int(P.max()) + W + 0
        hi = min(hi + 2, wl.capacity)
        before_k = host_bits(K[:, :, :, lo:hi])
        before_v = host_bits(V[:, :, :, lo:hi])
        acc, tid, nxt = das.das_greedy_accept(logits, draft)
        flag = torch.zeros(1, dtype=torch.int32, device="cuda")
        das.das_kv_append(cache, kn, vn, acc, pl, flag)
        torch.cuda.synchronize()
        oa, ot, on = oracle.greedy_accept(logits.cpu().numpy(), draft.cpu().numpy())
        assert np.array_equal(acc.cpu().numpy(), oa) and np.array_equal(acc.cpu().numpy(), a_star)
        assert np.array_equal(tid.cpu().numpy(), ot) and np.array_equal(nxt.cpu().numpy(), on)
        # oracle append on the window [lo, hi) of every slab
        K2, V2, pl2, f2 = oracle.kv_append(before_k, before_v, host_bits(kn), host_bits(vn), oa,
                                           P - lo)
        assert np.array_equal(host_bits(K[:, :, :, lo:hi]), K2)
        assert np.array_equal(host_bits(V[:, :, :, lo:hi]), V2)
        assert np.array_equal(pl.cpu().numpy(), pl2 + lo) and int(flag.item()) == f2 == 0
    finally:
        del cache, K, V, kn, vn
        torch.cuda.empty_cache()


@pytest.mark.parametrize("name", ["decode", "long"])
def test_full_size_sampled_e4m3(name):
    """The e4m3 cache variant at full size, configured as the benchmark's
    e4m3 probe: keys at depth r = 1 stored as e4m3 codes (host generator),
    values at depth R = 2 as bf16 (device fill, checked bit for bit against
    the host generator on the sampled slabs).  Sampled (sequence, kv head)
    groups are recomputed by the oracle from the widened keys; every output
    is checked for the properties that hold at any size."""
    import paper_2609_34538_gb300 as das
    wl = wl_mod.WORKLOADS[name].replace(depths=2, key_depth=1, value_depth=2)
    L, B, cap, H, D, G = wl.layers, wl.batch, wl.capacity, wl.kv_heads, wl.head_dim, wl.group
    cache = das.DepthKVCacheF8.empty(2, L, B, cap, H, D)
    codes = synth.e4m3_codes(wl.seed, synth.T_KLOW, (1, L, B, cap, H, D))
    cache.k_low.copy_(torch.from_numpy(codes))
    sdev.fill_matured(cache.v_top, wl.seed, synth.T_VCACHE, 1, 2, 2)
    ws = das.new_workspace_f8(cache, wl.q_heads, wl.max_block)
    P, T = wl.prefix_lens(), wl.block_lens()
    pl, bl = dev_i32(P), dev_i32(T)
    try:
        for layer in range(L):
            q, kb, vb = sdev.layer_inputs(wl, layer)
            out, lse = das.das_mature_v_attention_f8(cache, layer, 1, 2, pl, bl, q, kb, vb, ws)
            torch.cuda.synchronize()
            o = out.float().cpu().numpy()
            l = lse.cpu().numpy()
            assert np.all(np.isfinite(o))
            for b in range(B):
                assert np.all(o[b, T[b]:] == 0) and np.all(np.isneginf(l[b, :, T[b]:]))
                assert np.all(np.isfinite(l[b, :, :T[b]]))
            qh, kbh, vbh = host_bits(q), host_bits(kb), host_bits(vb)
            for b, h in _pairs(wl, layer, _samples(wl)):
                kc = codes[0, layer, b, :P[b], h:h + 1]
                kp = oracle.widen_f8_cache(np.zeros(kc.shape, np.uint16), kc[None])[0]
                vp = synth.matured_block(wl.seed, synth.T_VCACHE, 1, 2, 2, layer, b, 0, int(P[b]),
                                         h, h + 1, D)
                assert np.array_equal(host_bits(cache.v_top[layer, b, :P[b], h:h + 1]), vp)
                ro, rl = oracle.attend_seq(qh[b, :, h * G:(h + 1) * G], kp, vp,
                                           kbh[b, :, h:h + 1], vbh[b, :, h:h + 1],
                                           block_len=int(T[b]))
                assert_close(o[b, :, h * G:(h + 1) * G], ro, l[b, h * G:(h + 1) * G], rl,
                             where=f"[{name} e4m3 keys, layer {layer} b {b} kv head {h}]")
        assert das.workspace_status(ws) == 0
    finally:
        del cache
        torch.cuda.empty_cache()
