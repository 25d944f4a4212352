"""Greedy target preservation (App. B proposition), exactly, on the oracle:
a toy looped target decoded autoregressively and speculatively (any
proposals: right, corrupted or random) emits the same tokens.  A verify row
sees the same keys in the same order as the autoregressive step of its
position, so in the oracle's fp64 arithmetic every conditional is identical;
this pins the acceptance and commit logic end to end."""
import numpy as np
import pytest

from tests.toy_looped import ToyLoopedCPU, Weights, ar, spec


@pytest.mark.parametrize("w,corrupt", [(4, 0.0), (4, 0.3), (6, 0.6), (3, 1.0)])
def test_speculative_equals_autoregressive(w, corrupt):
    W = Weights(seed=1)
    prompt, n = [3, 17, 5, 40, 9], 20
    ref = ar(ToyLoopedCPU(W, 64), prompt, n + 8)
    rng = np.random.default_rng(int(w * 10 + corrupt * 100))

    def propose(emitted, k):
        base = len(emitted)
        ys = [ref[base + i] if base + i < len(ref) else 0 for i in range(k)]
        return [int(rng.integers(0, W.V)) if rng.random() < corrupt else y for y in ys]

    out, accs = spec(ToyLoopedCPU(W, 64), prompt, n, propose, w)
    assert out == ref[:n]
    if corrupt == 0.0:
        assert all(a == w for a in accs[:-1])   # right proposals are all accepted
    if corrupt == 1.0:
        assert sum(accs) < len(accs)            # random proposals are mostly rejected
