"""The dense LSTM comparator kernel against the oracle's dense LSTM (GPU).

lstm_approx_dense_run computes the LSTM of Sec. II with the full gate
matrices (the baseline the approximation is compared with, Sec. VI-B).  It
is held to the fp32 bound, 1e-4 elementwise, against oracle.qor.dense_lstm
(pinned against torch.nn.LSTM on the CPU) on the same fp32-rounded W and x,
at every compiled layout (h quads per lane 1, 2, 4; 16 or 32 units per CTA;
clusters of 4, 8, 16), ragged sizes, several streams, bias and initial
state; sizes it cannot take are refused before any launch.
"""
import numpy as np
import pytest

from oracle import qor
from parity_util import FP32_TOL, assert_parity
from workloads import draw_inputs, draw_weight

pytestmark = pytest.mark.gpu


def _case(D, H, T, B, seed, extras):
    W = [draw_weight(H, D + H, seed + g).astype(np.float32).astype(np.float64) for g in range(4)]
    x = draw_inputs(T, B, D, "relu", seed + 9).astype(np.float32).astype(np.float64)
    rng = np.random.default_rng(seed)
    bias = (0.2 * rng.standard_normal((4, H))).astype(np.float32).astype(np.float64) if extras else None
    h0 = (0.3 * rng.standard_normal((B, H))).astype(np.float32).astype(np.float64) if extras else None
    c0 = (0.3 * rng.standard_normal((B, H))).astype(np.float32).astype(np.float64) if extras else None
    return W, x, bias, h0, c0


@pytest.mark.parametrize("D,H,T,B,extras", [
    (1024, 512, 20, 1, False),   # the batch-1 benchmark shape: 32 units per CTA, 16 CTAs, 4 h quads per lane
    (64, 64, 8, 1, False),       # 16 units per CTA, 4 CTAs, 1 quad
    (40, 100, 5, 3, True),       # ragged: 8 CTAs of 16 units (28 padding units), 1 quad
    (24, 200, 4, 2, True),       # 16 CTAs of 16 units, 2 quads
    (36, 300, 3, 2, True),       # 16 CTAs of 32 units, 4 quads; D not a multiple of 8 (tiled projection)
    (16, 256, 6, 5, False),
])
def test_dense_kernel_matches_oracle(cuda_device, D, H, T, B, extras):
    import torch
    from paper_1905_00689_gb300 import dense_run
    W, x, bias, h0, c0 = _case(D, H, T, B, 9000 + H, extras)
    ref_h, ref_c = qor.dense_lstm(W, x, bias=bias, h0=h0, c0=c0, return_c=True)
    dev = torch.device("cuda:0")
    f32 = lambda a: None if a is None else torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(dev)
    Wx = f32(np.concatenate([w[:, :D] for w in W]))
    Wh = f32(np.concatenate([w[:, D:] for w in W]))
    out_h = torch.full((T, B, H), float("nan"), device=dev)
    out_c = torch.full((B, H), float("nan"), device=dev)
    from paper_1905_00689_gb300 import dense_set_launch_order
    # twice in each launch order (one stream: recurrence first by default, then
    # projection first): the workspace, its flags and the kernel's barriers
    # start from scratch each call
    try:
        for order in (0, 0, 1, 1, 0):
            dense_set_launch_order(order)
            out_h.fill_(float("nan"))
            dense_run(Wx, Wh, f32(bias), f32(x), out_h, h0=f32(h0), c0=f32(c0), out_c=out_c)
            got = {"h": out_h.double().cpu().numpy(), "c_last": out_c.double().cpu().numpy()}
            assert_parity(got, {"h": ref_h, "c_last": ref_c}, FP32_TOL)
    finally:
        dense_set_launch_order(0)


def test_dense_kernel_refuses_what_it_cannot_take(cuda_device):
    import torch
    from paper_1905_00689_gb300 import LSTMApproxError, dense_run, dense_workspace_bytes
    dev = torch.device("cuda:0")
    D, H, T, B = 8, 516, 2, 1
    x = torch.zeros((T, B, D), device=dev)
    with pytest.raises(LSTMApproxError) as e:
        dense_run(torch.zeros((4 * H, D), device=dev), torch.zeros((4 * H, H), device=dev), None, x,
                  torch.zeros((T, B, H), device=dev))
    assert e.value.code == 1 and "H <= 512" in str(e.value)
    H = 64
    small = torch.empty(dense_workspace_bytes(H, T, B) - 4, dtype=torch.uint8, device=dev)
    with pytest.raises(LSTMApproxError) as e:
        dense_run(torch.zeros((4 * H, D), device=dev), torch.zeros((4 * H, H), device=dev), None, x,
                  torch.zeros((T, B, H), device=dev), workspace=small)
    assert e.value.code == 1 and "workspace" in str(e.value)
