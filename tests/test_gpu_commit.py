"""Bit-exact parity of das_greedy_accept and das_kv_append with the oracle."""
import numpy as np
import pytest
import torch

import oracle
import synth
from synth import workloads as wl_mod
from tests.gpu_util import assert_close, dev_bf16, dev_i32, host_bits

pytestmark = pytest.mark.gpu


def gpu_accept(logits, draft):
    import paper_2609_34538_gb300 as das
    acc, tid, nxt = das.das_greedy_accept(torch.from_numpy(logits).cuda(),
                                          torch.from_numpy(draft).cuda())
    torch.cuda.synchronize()
    return acc.cpu().numpy(), tid.cpu().numpy(), nxt.cpu().numpy()


def check_accept(logits, draft):
    g = gpu_accept(np.ascontiguousarray(logits, np.float32), np.ascontiguousarray(draft, np.int32))
    o = oracle.greedy_accept(logits, draft)
    for a, b, name in zip(g, o, ["accepted", "target_ids", "next_token"]):
        assert np.array_equal(a, b), name
    return g


def test_accept_verify_workload():
    """[8, 16, 32000] fp32 logits ~ N(0, 4) with planted acceptance lengths."""
    a_star, draft, logits = synth.accept_inputs(0, 8, 16, 32000)
    acc, _, _ = check_accept(logits, draft)
    assert np.array_equal(acc, a_star)


@pytest.mark.parametrize("B,W,V", [(1, 1, 2), (3, 5, 1001), (2, 16, 7), (4, 32, 50257), (1, 3, 4),
                                   (2, 100, 3001), (1, 1024, 64), (5, 8, 32000), (1, 2, 131072)])
def test_accept_shapes(B, W, V):
    a_star, draft, logits = synth.accept_inputs(B * 100 + W, B, W, V)
    check_accept(logits, draft)


@pytest.mark.parametrize("B,W,V", [(1, 8, 32000), (2, 16, 32000), (7, 16, 32000), (3, 4, 4099),
                                   (6, 5, 50257), (1, 1, 32000), (100, 1, 4096), (4, 3, 131072),
                                   (8, 16, 32000), (16, 8, 32000)])
def test_accept_single_kernel_shapes(B, W, V):
    """Shapes whose sequences fit one cluster of W k <= 16 CTAs (k CTAs per
    row).  They run as one kernel when the device holds all B clusters at
    once, else as the two-kernel form: on a 152-SM GB300 (7 resident clusters
    of 16 CTAs, 15 of 8) all but the last two run as one kernel, with k = 2,
    1, 1, 4, 3, 8, 1 and 5.  Bit-exact either way, planted acceptance
    lengths 0..W."""
    a_star, draft, logits = synth.accept_inputs(B * 1000 + W, B, W, V)
    acc, _, _ = check_accept(logits, draft)
    assert np.array_equal(acc, a_star)


@pytest.mark.parametrize("B,W", [(1, 1), (1, 2), (2, 4), (6, 5), (1, 8), (8, 16)])
@pytest.mark.parametrize("V", [4099, 4096])
def test_accept_ties_at_every_split(B, W, V):
    """Every row holds its maximum on both sides of the slice boundary of
    every k-way split, k = 2..8 (slices of ceil(V / k) columns, rounded up to
    whole float4s when V % 4 == 0): whatever k either form of the kernel
    picks, equal maxima sit in several CTAs' slices, and the smallest index
    (the left side of the 8-way boundary) must win."""
    logits = np.zeros((B, W, V), dtype=np.float32)
    cols = []
    for k in range(2, 9):
        sl = -(-V // k)
        if V % 4 == 0:
            sl = -(-sl // 4) * 4
        cols += [sl - 1, sl]
    logits[:, :, cols] = 7.0
    first = min(cols)
    draft = np.full((B, W), first, dtype=np.int32)
    draft[:, W - 1] = first + 1  # the last proposal is rejected
    acc, tid, nxt = check_accept(logits, draft)
    assert np.all(tid == first) and np.all(acc == W - 1) and np.all(nxt == first)


def test_accept_ties_and_infinities():
    """Equal maxima go to the smallest index; rows of -inf give index 0."""
    B, W, V = 3, 4, 4099
    logits = np.zeros((B, W, V), dtype=np.float32)
    logits[0, 0, [5, 9, 4000]] = 3.0
    logits[0, 1, [4098, 4097]] = 1.0
    logits[1, :, :] = -np.inf
    logits[2, 2, 17] = np.inf
    logits[2, 2, 18] = np.inf
    draft = np.array([[5, 4097, 0, 0], [0, 0, 0, 1], [0, 0, 17, 3]], dtype=np.int32)
    acc, tid, nxt = check_accept(logits, draft)
    assert tid[0, 0] == 5 and tid[0, 1] == 4097 and np.all(tid[1] == 0) and tid[2, 2] == 17
    assert list(acc) == [4, 3, 3]


@pytest.mark.parametrize("B,W", [(1, 7), (8, 7), (32, 7), (2, 4), (6, 5)])
@pytest.mark.parametrize("V", [4099, 4096])
def test_accept_ties_across_slices(B, W, V):
    """Equal maxima on both sides of a boundary between two CTAs' vocabulary
    slices: a row is scanned by k CTAs (k = SMs / rows, 1..8, or fewer in
    the one-kernel form; slices of ceil(V / k) columns, rounded up to whole
    float4s when V % 4 == 0).  Row r of every sequence holds a tie
    straddling the boundary of an (r + 2)-way split, so whatever k the
    launch picks (up to W + 1), some row's tie crosses CTAs; the smaller
    index wins either way.  On a 152-SM GB300: B 1 W 7, B 2 W 4 and B 6 W 5
    run as one kernel with k = 2, 4 and 3; B 8 and 32 at W 7 as two kernels
    with k = 2 and 1."""
    logits = np.zeros((B, W, V), dtype=np.float32)
    draft = np.zeros((B, W), dtype=np.int32)
    first = []
    for r in range(W):
        k = r + 2
        s = -(-V // k)
        if V % 4 == 0:
            s = -(-s // 4) * 4
        logits[:, r, [s - 1, s]] = 5.0
        draft[:, r] = s - 1
        first.append(s - 1)
    acc, tid, _ = check_accept(logits, draft)
    assert np.all(tid == np.array(first)[None, :]) and np.all(acc == W)


def _append_case(R, L, B, cap, H, D, W, pl, acc, seed):
    import paper_2609_34538_gb300 as das
    rng = np.random.default_rng(seed)
    K = rng.integers(0, 65535, (R, L, B, cap, H, D), dtype=np.uint16)
    V = rng.integers(0, 65535, (R, L, B, cap, H, D), dtype=np.uint16)
    kn = rng.integers(0, 65535, (R, L, B, W, H, D), dtype=np.uint16)
    vn = rng.integers(0, 65535, (R, L, B, W, H, D), dtype=np.uint16)
    cache = das.DepthKVCache(dev_bf16(K), dev_bf16(V))
    plg, flag = dev_i32(pl), torch.zeros(1, dtype=torch.int32, device="cuda")
    das.das_kv_append(cache, dev_bf16(kn), dev_bf16(vn), dev_i32(acc), plg, flag)
    torch.cuda.synchronize()
    K2, V2, pl2, f2 = oracle.kv_append(K, V, kn, vn, acc, pl)
    assert np.array_equal(host_bits(cache.k), K2) and np.array_equal(host_bits(cache.v), V2)
    assert np.array_equal(plg.cpu().numpy(), pl2) and int(flag.item()) == f2
    return f2


def test_append_bit_exact_every_count():
    """a = 0 (anchor only) .. a = W (all accepted), various offsets; every byte
    of the cache, including sentinels around the written ranges, checked."""
    W = 6
    acc = np.array([0, 1, 3, W - 1, W, 2, 0], dtype=np.int32)
    pl = np.array([0, 5, 17, 40, 0, 33, 49], dtype=np.int32)
    assert _append_case(3, 2, 7, 50, 2, 64, W, pl, acc, 1) == 0


def test_append_overflow_flags_and_skips():
    acc = np.array([3, 0, 5], dtype=np.int32)
    pl = np.array([30, 31, 20], dtype=np.int32)
    assert _append_case(2, 1, 3, 32, 1, 128, 8, pl, acc, 2) == 1


def test_verify_accept_append_chain_on_device():
    """Verify -> accept -> append with no host round trip: accepted counts flow
    from das_greedy_accept into das_kv_append on the device."""
    import paper_2609_34538_gb300 as das
    wl = wl_mod.WORKLOADS["verify"].replace(batch=3, layers=2, depths=4, key_depth=4,
                                            value_depth=4, prefix=(90, 90), vocab=500)
    W = wl.max_block
    a_star, draft, logits = synth.accept_inputs(5, wl.batch, W, wl.vocab)
    K, V = wl_mod.gen_cache(wl, depths=range(1, wl.depths + 1), tokens=90)
    kn, vn = wl_mod.gen_staged(wl, W)
    cache = das.DepthKVCache(dev_bf16(K), dev_bf16(V))
    ws = das.new_workspace(cache, wl.q_heads, W)
    pl = dev_i32(wl.prefix_lens())
    bl = dev_i32(wl.block_lens())
    q = dev_bf16(wl_mod.gen_q(wl, 1))
    kb, vb = map(dev_bf16, wl_mod.gen_block_kv(wl, 1))
    das.das_verify_attention(cache, 1, wl.depths, pl, bl, q, kb, vb, ws)
    acc, tid, nxt = das.das_greedy_accept(torch.from_numpy(logits).cuda(),
                                          torch.from_numpy(draft).cuda())
    flag = torch.zeros(1, dtype=torch.int32, device="cuda")
    das.das_kv_append(cache, dev_bf16(kn), dev_bf16(vn), acc, pl, flag)
    torch.cuda.synchronize()
    oa, _, _ = oracle.greedy_accept(logits, draft)
    K2, V2, pl2, f2 = oracle.kv_append(K, V, kn, vn, oa, wl.prefix_lens())
    assert np.array_equal(acc.cpu().numpy(), a_star)
    assert np.array_equal(host_bits(cache.k), K2) and np.array_equal(host_bits(cache.v), V2)
    assert np.array_equal(pl.cpu().numpy(), pl2) and int(flag.item()) == f2 == 0


def test_attention_right_after_append_sees_the_new_lengths():
    """append -> attention -> append -> ... in one stream with no host round
    trip: each attention call plans its split from prefix_len, which the
    append just before it bumps on the device, and must attend over exactly
    the updated prefix (the cached rows the append wrote included)."""
    import paper_2609_34538_gb300 as das
    rounds = 6
    wl = wl_mod.WORKLOADS["verify"].replace(batch=3, layers=1, depths=2, key_depth=2,
                                            value_depth=2, prefix=(90, 200), vocab=500)
    W = wl.max_block
    wl = wl.replace(extra_capacity=rounds * W)
    pl0 = np.array([90, 130, 200], dtype=np.int32)
    K, V = wl_mod.gen_cache(wl, depths=range(1, wl.depths + 1), tokens=int(pl0.max()))
    kn, vn = wl_mod.gen_staged(wl, W)
    rng = np.random.default_rng(11)
    accs = rng.integers(0, W + 1, size=(rounds, wl.batch)).astype(np.int32)
    cache = das.DepthKVCache(dev_bf16(K), dev_bf16(V))
    ws = das.new_workspace(cache, wl.q_heads, W)
    pl, bl = dev_i32(pl0), dev_i32(wl.block_lens())
    q = dev_bf16(wl_mod.gen_q(wl, 0))
    kb, vb = map(dev_bf16, wl_mod.gen_block_kv(wl, 0))
    kn_d, vn_d = dev_bf16(kn), dev_bf16(vn)
    acc_d = torch.from_numpy(accs).cuda()
    flag = torch.zeros(1, dtype=torch.int32, device="cuda")
    torch.cuda.synchronize()
    outs = []
    for i in range(rounds):
        das.das_kv_append(cache, kn_d, vn_d, acc_d[i], pl, flag)
        o, l = das.das_verify_attention(cache, 0, wl.depths, pl, bl, q, kb, vb, ws)
        outs.append((o, l))
    torch.cuda.synchronize()
    assert int(flag.item()) == 0 and das.workspace_status(ws) == 0
    Kh, Vh, plh = K, V, pl0
    for i in range(rounds):
        Kh, Vh, plh, f = oracle.kv_append(Kh, Vh, kn, vn, accs[i], plh)
        assert f == 0
        ref_o, ref_l = oracle.attention(Kh, Vh, 0, wl.depths, wl.depths, plh, wl.block_lens(),
                                        wl_mod.gen_q(wl, 0), *wl_mod.gen_block_kv(wl, 0))
        o, l = outs[i]
        assert_close(o.float().cpu().numpy(), ref_o, l.cpu().numpy(), ref_l,
                     where=f"[round {i} prefix {plh.tolist()}]")
    assert np.array_equal(pl.cpu().numpy(), plh)
