"""The sequential Mature-Spec / Mature-V drafting loop (Sec. 3.2, Eq. 4;
App. A.2): one draft token at a time, each attention call with a block that
holds the tokens drafted so far, recurrence steps s = 1..d reading prefix
keys at depth s (Mature-V) or R (Deep K/V) and prefix values at depth R.
Every call is compared with the fp64 oracle."""
import numpy as np
import pytest
import torch

import oracle
from synth import workloads as wl_mod
from tests.gpu_util import assert_close, dev_bf16, dev_i32, run_small

pytestmark = pytest.mark.gpu


def seq_wl(**kw):
    base = dict(name="sequential", batch=1, layers=2, q_heads=8, kv_heads=8, head_dim=128,
                depths=8, key_depth=4, value_depth=8, prefix=(1500, 1500), block=(8,))
    base.update(kw)
    return wl_mod.Workload(**base)


@pytest.mark.parametrize("G", [1, 4, 8])
@pytest.mark.parametrize("P", [1, 700, 4096])
def test_single_query_row(G, P):
    """T = 1: the decode shape of a sequential draft step (one new token)."""
    run_small(seq_wl(q_heads=8 * G, prefix=(P, P), block=(1,)))


def test_recurrence_steps_and_growing_block():
    """Token i = 1..4 of a block, recurrence steps s = 1..4: key depth s,
    value depth R (Mature-V), then key depth R (Deep K/V, Mature-Spec).  All
    calls of one token go back to back on one workspace, like a captured
    draft step, and each is checked against the oracle."""
    import paper_2609_34538_gb300 as das
    wl = seq_wl(depths=8, layers=2, prefix=(900, 900), block=(4,))
    R = wl.depths
    K, V = wl_mod.gen_cache(wl, depths=list(range(1, R + 1)))
    cache = das.DepthKVCache(dev_bf16(K), dev_bf16(V))
    ws = das.new_workspace(cache, wl.q_heads, wl.max_block)
    pl = dev_i32(wl.prefix_lens())
    for i in range(1, 5):
        bl = dev_i32([i])
        results = []
        for kap in list(range(1, 5)) + [R]:
            for layer in range(wl.layers):
                q = wl_mod.gen_q(wl, layer)
                kb, vb = wl_mod.gen_block_kv(wl, layer)
                out, lse = das.das_mature_v_attention(cache, layer, kap, R, pl, bl, dev_bf16(q),
                                                      dev_bf16(kb), dev_bf16(vb), ws)
                results.append((kap, layer, q, kb, vb, out, lse))
        torch.cuda.synchronize()
        for kap, layer, q, kb, vb, out, lse in results:
            ref_o, ref_l = oracle.attention(K, V, layer, kap, R, wl.prefix_lens(),
                                            np.array([i], np.int32), q, kb, vb)
            assert_close(out.float().cpu().numpy(), ref_o, lse.cpu().numpy(), ref_l,
                         where=f"[token {i} kappa {kap} layer {layer}]")
        assert das.workspace_status(ws) == 0
