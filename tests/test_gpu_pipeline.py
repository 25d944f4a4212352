"""Verify -> accept -> commit on the GPU with a toy looped target (App. B
proposition, Sec. 3.4): das_verify_attention at every recurrent depth over a
block [anchor, y_1 .. y_{w-1}], das_greedy_accept, das_kv_append, decoding
speculatively with right, corrupted and random proposals, emits the tokens
of autoregressive decoding computed by the oracle (the same toy model in
fp64 with the oracle's attention, acceptance and commit).

The proposition holds in exact arithmetic (test_oracle_pipeline checks it
exactly on the oracle).  The library returns attention outputs in bf16, so
the GPU model's logits differ from the oracle's.  How much is measured on
the CPU: the oracle model with its attention outputs rounded to bf16 (what
storing them in the library's output type alone does) moves the logits of
the oracle's autoregressive steps by at most delta.  The GPU's outputs are
within about one bf16 rounding of the exact ones, so a near-tie is an oracle
step whose two largest logits are closer than TIE = 4 delta; there either of
the tied tokens is a correct greedy choice and the continuations may part.
The tokens must agree up to the first near-tie, and any divergence must sit
at a near-tie of the oracle's own stream.  The toy model's scales are chosen
so that near-ties are rare (qk 0.7, v 0.5: delta is a few hundredths of a
logit against margins of tenths and more) while the continuation stays
varied."""
import numpy as np
import pytest

from tests.toy_looped import ToyLoopedCPU, ToyLoopedGPU, Weights, ar, spec

pytestmark = pytest.mark.gpu

PROMPT, N = [3, 17, 5, 40, 9], 24


@pytest.fixture(scope="module")
def oracle_stream():
    W = Weights(seed=21, qk=0.7, v=0.5)
    margins, exact, rounded = [], [], []
    ref = ar(ToyLoopedCPU(W, 96), PROMPT, N + 8, margins, exact)
    rref = ar(ToyLoopedCPU(W, 96, bf16_outputs=True), PROMPT, N + 8, None, rounded)
    agree = next((i for i in range(N + 8) if ref[i] != rref[i]), N + 8)
    delta = max(np.abs(exact[i] - rounded[i]).max() for i in range(agree))
    return W, ref, np.array(margins), 4.0 * delta


def test_bf16_rounding_moves_the_toy_logits_little(oracle_stream):
    W, ref, margins, tie = oracle_stream
    print(f"TIE {tie:.4f}; oracle margins {np.round(margins[:N], 3)}")
    assert len(set(ref[:N])) > 8      # a varied continuation
    assert tie < 0.5                   # a few hundredths of a logit per rounding
    assert (margins[:N] < tie).sum() <= 2


@pytest.mark.parametrize("w,corrupt", [(4, 0.0), (8, 0.3), (6, 0.6), (3, 1.0)])
def test_gpu_speculative_equals_oracle_autoregressive(oracle_stream, w, corrupt):
    W, ref, margins, tie = oracle_stream
    rng = np.random.default_rng(int(w * 10 + corrupt * 100))

    def propose(emitted, k):
        base = len(emitted)
        ys = [ref[base + i] if base + i < len(ref) else 0 for i in range(k)]
        return [int(rng.integers(0, W.V)) if rng.random() < corrupt else y for y in ys]

    out, accs = spec(ToyLoopedGPU(W, 96), PROMPT, N, propose, w)
    first_tie = next((i for i in range(N) if margins[i] < tie), N)
    print(f"w {w} corrupt {corrupt}: TIE {tie:.4f}, first near-tie at {first_tie} of {N}, "
          f"acceptances {accs}")
    assert out[:first_tie] == ref[:first_tie]
    diverge = next((i for i in range(N) if out[i] != ref[i]), None)
    assert diverge is None or margins[diverge] < tie
    if corrupt == 0.0 and first_tie == N:
        assert all(a == w for a in accs[:-1])
