"""Stored factors read back from the device, bit for bit (GPU).

lstm_approx_set_factors rounds sigma to fp32 and u, v to the handle's dtype
(fp64 -> fp32 -> bf16, round-to-nearest-even).  The oracle of the parity
tests receives workloads.rounded_factors, whose bf16 rounding is pinned
against torch in test_bf16_rounding.py; this test closes the loop by
reading the library's stored values back (lstm_approx_get_term) and
requiring them to equal rounded_factors exactly, including the pruned
columns (zero) and the mask read back by get_mask.
"""
import numpy as np
import pytest

from workloads import draw_factor_set, rounded_factors

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
def test_stored_terms_equal_the_rounding_rule(cuda_device, dtype):
    from paper_1905_00689_gb300 import LSTMApprox
    D, H, K, nz = 37, 44, 9, 30
    gates = [draw_factor_set(H, D + H, K, nz, 7700 + g) for g in range(4)]
    # values that exercise the rounding: ties of both parities and tiny magnitudes
    gates[1]["u"][0, :4] = [1.0 + 2.0 ** -8, 1.0 + 3 * 2.0 ** -8, -(1.0 + 2.0 ** -8), 3e-39]
    gates[2]["val"][0, :3] = [1.0 + 2.0 ** -8 + 2.0 ** -40, 1e-45, -2.5]
    m = LSTMApprox(1, [D], H, K, 1, dtype)
    m.set_layer(0, gates)
    want = rounded_factors(gates, dtype)
    for g in range(4):
        for k in range(K):
            sigma, u, v = m.get_term(0, g, k)
            assert np.float32(want[g]["sigma"][k]) == np.float32(sigma), (g, k)
            assert np.array_equal(u.view(np.uint32), want[g]["u"][k].astype(np.float32).view(np.uint32)), (g, k)
            dense = np.zeros(D + H, dtype=np.float32)
            dense[want[g]["idx"][k]] = want[g]["val"][k].astype(np.float32)
            assert np.array_equal(v.view(np.uint32), dense.view(np.uint32)), (g, k)
            assert np.array_equal(m.get_mask(0, g, k), want[g]["idx"][k])
    m.close()
