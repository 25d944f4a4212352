"""Parity of das_mature_v_attention / das_verify_attention with the fp64
oracle on seeded inputs, over shapes that span several tiles, splits across
CTAs, ragged tails and the degenerate cases of the method."""
import numpy as np
import pytest
import torch

import oracle
from synth import workloads as wl_mod
from tests.gpu_util import assert_close, dev_bf16, dev_i32, run_small

pytestmark = pytest.mark.gpu

TINY = wl_mod.WORKLOADS["tiny"]


def small(**kw):
    base = dict(name="small", batch=1, layers=2, q_heads=2, kv_heads=2, head_dim=128, depths=8,
                key_depth=2, value_depth=8, prefix=(100, 100), block=(4,))
    base.update(kw)
    return wl_mod.Workload(**base)


def test_tiny_workload():
    """B1 L1 H4/4 D64 P256 T4 R8, Mature-V (r, R) = (2, 8)."""
    run_small(TINY)


@pytest.mark.parametrize("P", [0, 1, 63, 64, 65, 200, 1000])
def test_prefix_lengths(P):
    run_small(small(prefix=(P, P)), layer=1)


@pytest.mark.parametrize("G,T", [(1, 1), (1, 16), (4, 4), (4, 8), (4, 12), (4, 16), (8, 8),
                                 (1, 64), (2, 32), (1, 17), (2, 16), (1, 32)])
def test_rows_per_kv_head(G, T):
    """1..64 rows per kv head: up to 16 and up to 32 rows take four and two
    copies of the rows, more the 64-row layout."""
    run_small(small(q_heads=2 * G, kv_heads=2, prefix=(300, 300), block=(T,)))


@pytest.mark.parametrize("D", [64, 128])
def test_head_dims(D):
    run_small(small(head_dim=D, q_heads=8, kv_heads=2, prefix=(777, 777), block=(8,)))


@pytest.mark.parametrize("q_heads", [8, 2])
def test_ragged_batch_with_empty_rows(q_heads):
    """Mixed prefix and block lengths, including P = 0 and T = 0; 64 and 16
    rows per kv head at the longest block."""
    wl = small(batch=6, q_heads=q_heads, kv_heads=2, block=(16,), prefix=(0, 600))
    run_small(wl, prefix=[0, 1, 600, 64, 333, 0], block=[16, 0, 3, 8, 1, 0])


@pytest.mark.parametrize("B", [33, 70])
def test_more_than_32_sequences(B):
    """Batches past one warp's 32 lanes: the split is planned after the
    dependency wait over several 32-sequence chunks, and walks cross from one
    chunk's sequences into the next; ragged lengths including P = 0 and T = 0."""
    rng = np.random.default_rng(B)
    prefix = rng.integers(0, 300, size=B).astype(np.int32)
    block = rng.integers(0, 9, size=B).astype(np.int32)
    prefix[::7] = 0
    block[::11] = 0
    wl = small(batch=B, q_heads=4, kv_heads=2, head_dim=64, prefix=(0, 300), block=(8,))
    run_small(wl, prefix=prefix, block=block)


def test_split_across_many_ctas():
    """More tiles than CTAs for one pair: hundreds of partials merged."""
    run_small(small(batch=1, kv_heads=1, q_heads=4, prefix=(20000, 20000), block=(16,)))
    run_small(small(batch=2, kv_heads=2, q_heads=8, prefix=(5000, 5000), block=(8,)))


@pytest.mark.parametrize("P", [5760, 5761, 9000])
def test_weighted_split_threshold(P):
    """8 pairs on 152 CTAs: the split weights block tiles (extra weight 3)
    once the weighted list holds at least (2 + 3) positions per CTA,
    8 (ceil(P / 64) + 1) + 3 * 8 >= 5 * 152, i.e. P >= 5761; both sides of
    the threshold."""
    run_small(small(batch=1, kv_heads=8, q_heads=8, prefix=(P, P), block=(8,)))


def test_many_pairs():
    """1600 (sequence, kv head) pairs over 152 CTAs, ragged lengths: ranges
    that cross many pairs, a merge grid of thousands of CTAs."""
    rng = np.random.default_rng(5)
    B = 200
    prefix = rng.integers(0, 200, size=B).astype(np.int32)
    block = rng.integers(1, 5, size=B).astype(np.int32)
    wl = small(batch=B, q_heads=8, kv_heads=8, head_dim=64, prefix=(0, 200), block=(4,))
    run_small(wl, prefix=prefix, block=block)


def test_one_workspace_across_shapes():
    """A workspace sized for the largest of three shapes serves all of them in
    turn, twice: nothing a call leaves in it but the status word affects the
    next call, whatever its shape."""
    import paper_2609_34538_gb300 as das
    shapes = [small(batch=4, q_heads=16, kv_heads=8, prefix=(900, 3000), block=(8,)),
              small(batch=1, q_heads=4, kv_heads=1, prefix=(20000, 20000), block=(16,)),
              small(batch=2, q_heads=8, kv_heads=2, prefix=(5000, 5000), block=(4,))]
    cases = []
    for wl in shapes:
        K, V = wl_mod.gen_cache(wl, depths=[2, 8])
        P, T = wl.prefix_lens(), wl.block_lens()
        q = wl_mod.gen_q(wl, 1)
        kb, vb = wl_mod.gen_block_kv(wl, 1)
        ref = oracle.attention(K, V, 1, 2, 8, P, T, q, kb, vb)
        cache = das.DepthKVCache(dev_bf16(K), dev_bf16(V))
        cases.append((wl, cache, dev_i32(P), dev_i32(T), dev_bf16(q), dev_bf16(kb), dev_bf16(vb), ref))
    need = max(das.das_workspace_size(c[1], c[0].q_heads, c[0].max_block) for c in cases)
    ws = torch.zeros(need, dtype=torch.uint8, device="cuda")
    for rnd in range(2):
        for wl, cache, pl, bl, q, kb, vb, (ro, rl) in cases:
            n = das.das_workspace_size(cache, wl.q_heads, wl.max_block)
            out, lse = das.das_mature_v_attention(cache, 1, 2, 8, pl, bl, q, kb, vb, ws[:n])
            torch.cuda.synchronize()
            assert_close(out.float().cpu().numpy(), ro, lse.cpu().numpy(), rl,
                         where=f"[shared workspace, round {rnd}, B {wl.batch} Hkv {wl.kv_heads}]")
            assert das.workspace_status(ws) == 0


@pytest.mark.parametrize("q_heads", [8, 2])
def test_sharp_softmax_scale(q_heads):
    """scale = 1 makes the softmax peaked (the default 1/sqrt(D) is nearly flat
    here), so the reference max moves often; 32 and 8 rows per kv head."""
    run_small(small(q_heads=q_heads, kv_heads=2, prefix=(500, 500), block=(8,)), scale=1.0)


@pytest.mark.parametrize("kap,nu", [(2, 8), (2, 2), (8, 2), (8, 8), (5, 3)])
def test_read_policies(kap, nu):
    """Eq. 4: Mature-V (r,R), Aligned (r,r), Deep K (R,r), Deep K/V (R,R), any pair."""
    run_small(small(q_heads=4, kv_heads=2, prefix=(150, 150), block=(8,)), key_depth=kap,
              value_depth=nu)


@pytest.mark.parametrize("q_heads", [8, 2])
def test_verify_attention(q_heads):
    """Full-depth verify over 16 candidates: 64 and 16 rows per kv head."""
    run_small(small(q_heads=q_heads, kv_heads=2, prefix=(400, 400), block=(16,), key_depth=8),
              key_depth=8, value_depth=8, verify=True)


def test_positions_past_the_prefix_are_never_read():
    """NaN beyond prefix_len / block_len (cache, block K/V, queries) leaves the result exact."""
    wl = small(batch=3, q_heads=8, kv_heads=2, block=(16,), prefix=(0, 300))
    run_small(wl, prefix=[70, 300, 5], block=[5, 16, 9], poison_tail=True)


def test_rows_past_block_are_zero_and_status_clean():
    import paper_2609_34538_gb300 as das
    wl = small(batch=2, q_heads=4, kv_heads=2, block=(16,), prefix=(0, 200))
    out, lse, ws = run_small(wl, prefix=[200, 10], block=[3, 7])
    o = out.float().cpu().numpy()
    l = lse.cpu().numpy()
    assert np.all(o[0, 3:] == 0) and np.all(o[1, 7:] == 0)
    assert np.all(np.isneginf(l[0, :, 3:])) and np.all(np.isneginf(l[1, :, 7:]))
    assert das.workspace_status(ws) == 0


def test_out_of_range_lengths_are_clamped_and_flagged():
    import paper_2609_34538_gb300 as das
    wl = small(prefix=(50, 50), block=(4,))
    cap = wl.capacity
    from tests.gpu_util import dev_bf16 as up
    K, V = wl_mod.gen_cache(wl, depths=[2, 8])
    cache = das.DepthKVCache(up(K), up(V))
    ws = das.new_workspace(cache, 2, 4)
    q = up(wl_mod.gen_q(wl, 0))
    kb, vb = map(up, wl_mod.gen_block_kv(wl, 0))
    out1, l1 = das.das_mature_v_attention(cache, 0, 2, 8, dev_i32([cap + 100]), dev_i32([9]), q, kb,
                                          vb, ws)
    ws2 = das.new_workspace(cache, 2, 4)
    out2, l2 = das.das_mature_v_attention(cache, 0, 2, 8, dev_i32([cap]), dev_i32([4]), q, kb, vb,
                                          ws2)
    torch.cuda.synchronize()
    assert das.workspace_status(ws) == 2 and das.workspace_status(ws2) == 0
    assert torch.equal(out1, out2) and torch.equal(l1, l2)
    # a prefix that fills the whole capacity, against the oracle
    ro, rl = oracle.attention(K, V, 0, 2, 8, np.array([cap], np.int32), np.array([4], np.int32),
                              wl_mod.gen_q(wl, 0), *wl_mod.gen_block_kv(wl, 0))
    assert_close(out2.float().cpu().numpy(), ro, l2.cpu().numpy(), rl, where="[P = capacity]")


def test_deterministic_and_graph_capturable():
    import paper_2609_34538_gb300 as das
    wl = small(batch=2, q_heads=8, kv_heads=2, prefix=(3000, 3000), block=(8,))
    K, V = wl_mod.gen_cache(wl, depths=[2, 8])
    cache = das.DepthKVCache(dev_bf16(K), dev_bf16(V))
    ws = das.new_workspace(cache, 8, 8)
    q = dev_bf16(wl_mod.gen_q(wl, 0))
    kb, vb = map(dev_bf16, wl_mod.gen_block_kv(wl, 0))
    pl, bl = dev_i32(wl.prefix_lens()), dev_i32(wl.block_lens())
    o1, l1 = das.das_mature_v_attention(cache, 0, 2, 8, pl, bl, q, kb, vb, ws)
    o2, l2 = das.das_mature_v_attention(cache, 0, 2, 8, pl, bl, q, kb, vb, ws)
    torch.cuda.synchronize()
    assert torch.equal(o1, o2) and torch.equal(l1, l2)
    o3, l3 = torch.zeros_like(o1), torch.zeros_like(l1)
    s = torch.cuda.Stream()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        das.das_mature_v_attention(cache, 0, 2, 8, pl, bl, q, kb, vb, ws, out=o3, lse=l3)
    g.replay()
    torch.cuda.synchronize()
    assert torch.equal(o1, o3) and torch.equal(l1, l3)


def test_workspace_reused_by_back_to_back_calls():
    """Calls enqueued back to back on one workspace (each kernel a programmatic
    dependent of the one before): every result matches the oracle."""
    import oracle
    import paper_2609_34538_gb300 as das
    wl = small(batch=2, q_heads=8, kv_heads=2, prefix=(3000, 3000), block=(8,))
    K, V = wl_mod.gen_cache(wl, depths=[2, 8])
    cache = das.DepthKVCache(dev_bf16(K), dev_bf16(V))
    ws = das.new_workspace(cache, 8, 8)
    cases = [(0, [3000, 2900], [8, 5]), (1, [64, 0], [8, 8]), (0, [1, 2999], [3, 8]),
             (1, [3000, 3000], [8, 8]), (1, [0, 0], [1, 8])]
    results = []
    for layer, pl, bl in cases:
        q = wl_mod.gen_q(wl, layer)
        kb, vb = wl_mod.gen_block_kv(wl, layer)
        out, lse = das.das_mature_v_attention(cache, layer, 2, 8, dev_i32(pl), dev_i32(bl),
                                              dev_bf16(q), dev_bf16(kb), dev_bf16(vb), ws)
        results.append((layer, pl, bl, q, kb, vb, out, lse))
    torch.cuda.synchronize()
    for layer, pl, bl, q, kb, vb, out, lse in results:
        ref_o, ref_l = oracle.attention(K, V, layer, 2, 8, np.asarray(pl, np.int32),
                                        np.asarray(bl, np.int32), q, kb, vb)
        assert_close(out.float().cpu().numpy(), ref_o, lse.cpu().numpy(), ref_l,
                     where=f"[layer {layer} prefix {pl} block {bl}]")
    assert das.workspace_status(ws) == 0


def test_attention_call_object_matches_functional_api():
    """AttentionCall (arguments checked once) gives the functional calls' bits."""
    import paper_2609_34538_gb300 as das
    wl = small(batch=2, q_heads=8, kv_heads=2, prefix=(700, 700), block=(8,))
    K, V = wl_mod.gen_cache(wl, depths=[2, 8])
    cache = das.DepthKVCache(dev_bf16(K), dev_bf16(V))
    ws = das.new_workspace(cache, 8, 8)
    q = dev_bf16(wl_mod.gen_q(wl, 1))
    kb, vb = map(dev_bf16, wl_mod.gen_block_kv(wl, 1))
    pl, bl = dev_i32([700, 650]), dev_i32([8, 3])
    call = das.AttentionCall(cache, pl, bl, q, kb, vb, ws)
    o1, l1 = das.das_mature_v_attention(cache, 1, 2, 8, pl, bl, q, kb, vb, ws)
    o2, l2 = call.mature_v(1, 2, 8)
    o1, l1, o2, l2 = o1.clone(), l1.clone(), o2.clone(), l2.clone()
    o3, l3 = das.das_verify_attention(cache, 1, 8, pl, bl, q, kb, vb, ws)
    o3, l3 = o3.clone(), l3.clone()
    o4, l4 = call.verify(1, 8)
    torch.cuda.synchronize()
    assert torch.equal(o1, o2) and torch.equal(l1, l2)
    assert torch.equal(o3, o4) and torch.equal(l3, l4)
    with pytest.raises(TypeError):
        das.AttentionCall(cache, pl, bl, q.float(), kb, vb, ws)


def test_host_errors_raise():
    import paper_2609_34538_gb300 as das
    wl = small()
    cache = das.DepthKVCache.empty(8, 2, 1, wl.capacity, 2, 128)
    ws = das.new_workspace(cache, 2, 4)
    q = torch.zeros((1, 4, 2, 128), dtype=torch.bfloat16, device="cuda")
    kb = torch.zeros((1, 4, 2, 128), dtype=torch.bfloat16, device="cuda")
    pl, bl = dev_i32([10]), dev_i32([4])
    with pytest.raises(das.DasError) as e:
        das.das_mature_v_attention(cache, 0, 9, 8, pl, bl, q, kb, kb, ws)
    assert e.value.code == das.DAS_ERR_INVALID_ARG
    with pytest.raises(das.DasError) as e:
        das.das_mature_v_attention(cache, 0, 2, 8, pl, bl, q, kb, kb, ws[:100])
    assert e.value.code == das.DAS_ERR_WORKSPACE
