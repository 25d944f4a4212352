"""Verify -> accept -> commit on the GPU with a toy looped target (App. B
proposition, Sec. 3.4): das_verify_attention at every recurrent depth over a
block [anchor, y_1 .. y_{w-1}], das_greedy_accept, das_kv_append, decoding
speculatively with right, corrupted and random proposals, emits the tokens
of autoregressive decoding computed by the oracle (the same toy model in
fp64 with the oracle's attention, acceptance and commit).

The proposition holds in exact arithmetic (test_oracle_pipeline checks it
exactly on the oracle).  The library returns attention outputs rounded to
bf16, so the GPU model's logits differ from the oracle's in the last bits;
the tokens must agree up to the first oracle step whose two largest logits
are closer than TIE (a near-tie), where either of the tied tokens is a
correct greedy choice and the continuations may part.  Any divergence must
sit at such a step of the oracle's own stream."""
import numpy as np
import pytest

from tests.toy_looped import ToyLoopedCPU, ToyLoopedGPU, Weights, ar, spec

pytestmark = pytest.mark.gpu

TIE = 0.1  # oracle logit gap below which bf16 rounding may reorder the two largest


@pytest.mark.parametrize("w,corrupt", [(4, 0.0), (8, 0.3), (6, 0.6), (3, 1.0)])
def test_gpu_speculative_equals_oracle_autoregressive(w, corrupt):
    W = Weights(seed=1)
    prompt, n = [3, 17, 5, 40, 9], 24
    margins = []
    ref = ar(ToyLoopedCPU(W, 96), prompt, n + 8, margins)
    assert len(set(ref)) > 4  # a varied continuation
    rng = np.random.default_rng(int(w * 10 + corrupt * 100))

    def propose(emitted, k):
        base = len(emitted)
        ys = [ref[base + i] if base + i < len(ref) else 0 for i in range(k)]
        return [int(rng.integers(0, W.V)) if rng.random() < corrupt else y for y in ys]

    out, accs = spec(ToyLoopedGPU(W, 96), prompt, n, propose, w)
    first_tie = next((i for i in range(n) if margins[i] < TIE), n)
    print(f"w {w} corrupt {corrupt}: oracle margins min {min(margins[:n]):.3f}, "
          f"first near-tie at {first_tie} of {n}, acceptances {accs}")
    assert out[:first_tie] == ref[:first_tie]
    diverge = next((i for i in range(n) if out[i] != ref[i]), None)
    assert diverge is None or margins[diverge] < TIE
    if corrupt == 0.0 and first_tie == n:
        assert all(a == w for a in accs[:-1])
