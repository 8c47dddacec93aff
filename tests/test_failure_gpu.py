"""Failure detection on the GPU without faulting it.

The persistent kernel's waits are bounded in wall time.  The test hook
makes the first wait expect 16 bytes that no CTA ever sends (a signal that
nothing delivers); the kernel must give up after the short limit, report
ETIMEOUT through lstm_approx_sync, and leave the context usable.  Invalid
calls must be rejected before any launch and leave the handle unchanged.
"""
import numpy as np
import pytest

from parity_util import FP32_TOL, assert_parity, oracle_run, run_gpu
from paper_1905_00689_gb300 import (LSTMApproxError, OPT_TEST_STALL, OPT_WAIT_LIMIT, PATH_PERSISTENT, Q_LAUNCHES,
                                    Q_PERSISTENT_VARIANT)
from workloads import draw_factor_set, draw_inputs

pytestmark = pytest.mark.gpu


def _small():
    D, H, T, K = 32, 32, 4, 8
    gates = [draw_factor_set(H, D + H, K, 20, 4000 + g) for g in range(4)]
    x = draw_inputs(T, 1, D, "uniform", 4)
    return [gates], x, K


@pytest.mark.parametrize("variant", [1, 2])
def test_bounded_wait_reports_timeout_and_context_survives(cuda_device, variant):
    import torch
    layers, x, K = _small()
    got, m = run_gpu(layers, x, K, force_path=PATH_PERSISTENT, variant=variant)
    assert m.query(Q_PERSISTENT_VARIANT) == variant
    m.set_option(OPT_WAIT_LIMIT, 50_000)        # 50 ms
    m.set_option(OPT_TEST_STALL, 1)
    xt = torch.from_numpy(x.astype(np.float32)).cuda()
    out = torch.zeros((x.shape[0], 1, 32), device="cuda")
    m.run(xt, K, out)
    with pytest.raises(LSTMApproxError) as ei:
        m.sync()
    assert ei.value.code == 4                    # LSTM_APPROX_ETIMEOUT
    # the status word is cleared and the next run is correct
    m.run(xt, K, out)
    m.sync()
    ref = oracle_run(layers, x, K)
    assert_parity({"h": out.double().cpu().numpy()}, ref, FP32_TOL, keys=("h",))


def test_invalid_calls_launch_nothing(cuda_device):
    import torch
    layers, x, K = _small()
    _, m = run_gpu(layers, x, K)
    n0 = m.query(Q_LAUNCHES)
    xt = torch.from_numpy(x.astype(np.float32)).cuda()
    out = torch.zeros((x.shape[0], 1, 32), device="cuda")
    for kw, code in [(dict(K=K + 1), 1), (dict(K=0), 1), (dict(K=K, checkpoints=[3, 3]), 1),
                     (dict(K=K, checkpoints=[K + 1]), 1), (dict(K=K, checkpoints=list(range(1, 10))), 1)]:
        with pytest.raises(LSTMApproxError) as ei:
            m.run(xt, kw.pop("K"), out, **kw)
        assert ei.value.code == code
    assert m.query(Q_LAUNCHES) == n0
    # a gate whose factors are shallower than the requested depth
    with pytest.raises(LSTMApproxError) as ei:
        m.set_factors(0, 2, np.ones(2), np.ones((2, 32)), np.array([[0, 1], [1, 5]]), np.ones((2, 2)))
        m.run(xt, 4, out)
    assert ei.value.code == 5                    # LSTM_APPROX_ESTATE
    with pytest.raises(LSTMApproxError):
        m.set_factors(0, 0, np.ones(1), np.ones((1, 32)), np.array([[3, 2]]), np.ones((1, 2)))
    with pytest.raises(LSTMApproxError):
        m.set_factors(0, 0, np.ones(1), np.ones((1, 32)), np.array([[0, 64]]), np.ones((1, 2)))
    assert m.query(Q_LAUNCHES) == n0
