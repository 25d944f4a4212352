"""DAS-Wave carried parallel refinement (Sec. 3.3): the shifted readout of
Eq. 6 is bit-exact against the oracle, and the refinement driver runs every
round at the width of Eq. 5 with Deep K/V prefix reads; its attention calls
and its token guesses are checked against the oracle."""
import numpy as np
import pytest
import torch

import oracle
from synth import workloads as wl_mod
from tests.gpu_util import assert_close, dev_bf16, dev_i32

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("B,W,V", [(1, 1, 7), (3, 25, 32000), (2, 32, 1001), (1, 1024, 64),
                                   (4, 2, 131072)])
def test_wave_readout_bit_exact(B, W, V):
    import paper_2609_34538_gb300 as das
    rng = np.random.default_rng(B * 1000 + W)
    logits = rng.normal(0, 2, (B, W, V)).astype(np.float32)
    logits[0, 0, [V // 3, V - 1]] = 40.0              # a tie: the smaller index wins
    if W > 1:
        logits[-1, 1, :] = -np.inf                     # reads out 0
    tokens = rng.integers(0, V, (B, W + 3)).astype(np.int32)
    dt = torch.from_numpy(tokens).cuda()
    das.das_wave_readout(torch.from_numpy(logits).cuda(), dt)
    torch.cuda.synchronize()
    assert np.array_equal(dt.cpu().numpy(), oracle.wave_readout(logits, tokens))


def test_refinement_driver_rounds():
    """gamma 6, W_init 2, J 7, k 2 over 2 layers: every attention call reads
    the prefix at depth R for keys and values with block length W_j, and the
    token guesses after the last round are the oracle's readouts."""
    import paper_2609_34538_gb300 as das
    gamma, w_init, J, k = 6, 2, 7, 2
    wl = wl_mod.Workload(name="wave", batch=2, layers=2, q_heads=4, kv_heads=4, head_dim=64,
                         depths=4, key_depth=4, value_depth=4, prefix=(300, 300),
                         block=(gamma,))
    R, B, V = wl.depths, wl.batch, 97
    K, Vc = wl_mod.gen_cache(wl, depths=[R])
    cache = das.DepthKVCache(dev_bf16(K), dev_bf16(Vc))
    pl_host = np.array([300, 123], np.int32)
    pl = dev_i32(pl_host)
    ws = das.new_workspace(cache, wl.q_heads, gamma)
    drv = das.WaveRefinement(cache, pl, ws, wl.q_heads, gamma=gamma, w_init=w_init, rounds=J,
                             k_steps=k)
    assert drv.widths == [oracle.wave_width(gamma, w_init, j) for j in range(J)]
    rng = np.random.default_rng(5)
    calls, round_logits = [], []

    def step(j, s, layer):
        sub = wl.replace(seed=1000 * j + 10 * s + layer)
        q = wl_mod.gen_q(sub, layer)
        kb, vb = wl_mod.gen_block_kv(sub, layer)
        out = torch.empty((B, gamma, wl.q_heads, wl.head_dim), dtype=torch.bfloat16, device="cuda")
        lse = torch.empty((B, wl.q_heads, gamma), dtype=torch.float32, device="cuda")
        calls.append((j, layer, q, kb, vb, out, lse))
        return dev_bf16(q), dev_bf16(kb), dev_bf16(vb), out, lse

    def logits(j):
        lg = rng.normal(0, 1, (B, drv.widths[j], V)).astype(np.float32)
        round_logits.append(lg)
        return torch.from_numpy(lg).cuda()

    anchor = dev_i32([9, 4])
    tokens = drv.run(anchor, step, logits).cpu().numpy()
    assert len(calls) == J * k * wl.layers
    for j, layer, q, kb, vb, out, lse in calls[::5]:
        W = drv.widths[j]
        ref_o, ref_l = oracle.attention(K, Vc, layer, R, R, pl_host, np.full(B, W, np.int32), q,
                                        kb, vb)
        assert_close(out.float().cpu().numpy(), ref_o, lse.cpu().numpy(), ref_l,
                     where=f"[round {j} layer {layer}]")
    exp = np.repeat(np.array([[9], [4]], np.int32), gamma + 1, axis=1)
    for lg in round_logits:
        exp = oracle.wave_readout(lg, exp)
    assert np.array_equal(tokens, exp)
    assert das.workspace_status(ws) == 0
