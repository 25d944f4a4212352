"""The parity tolerance's bf16 rounding term, checked against torch's bf16
type: half_ulp_bf16(x) is half the distance from a bf16 value to the next
one up, so the extra room above 1e-2 is exactly the rounding of |o| >= 4."""
import numpy as np
import torch

from tests.gpu_util import OUT_ABS, abs_bound, half_ulp_bf16


def test_half_ulp_matches_bf16_spacing():
    rng = np.random.default_rng(0)
    x = np.concatenate([rng.uniform(-64, 64, 4000), [1.0, 2.0, 3.99, 4.0, 7.99, 8.0, -4.0]])
    xb = torch.tensor(x, dtype=torch.float32).to(torch.bfloat16)
    bits = xb.view(torch.int16).numpy().astype(np.int32)
    up = torch.from_numpy(((bits + 1) & 0xFFFF).astype(np.uint16)
                          .view(np.int16)).view(torch.bfloat16)
    spacing = (up.double() - xb.double()).abs().numpy()
    np.testing.assert_array_equal(half_ulp_bf16(xb.double().numpy()), spacing / 2)


def test_abs_bound_is_raw_below_four():
    o = np.array([0.0, 0.5, 1.9, 3.999, 4.0, 5.0, -6.0, 9.0])
    b = abs_bound(o)
    assert np.all(b[:4] == OUT_ABS)
    np.testing.assert_allclose(b[4:], OUT_ABS + np.array([2 ** -6, 2 ** -6, 2 ** -6, 2 ** -5]))
