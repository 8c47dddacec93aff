"""The allocation-free entry point agrees with the handle-based one.

lstm_approx_run_static serves callers that must not allocate device memory
while running (real-time control loops, plug-ins inside a framework that
owns all device memory).  It keeps its scratch in a fixed device array
inside the library.  This test packs one layer's fp32 factors itself,
calls the entry point through the C-ABI twice in a row (the second call
reuses the scratch the first one left behind), and checks both outputs
against lstm_approx_run on the same factors.  The file is named so that
pytest collects it last.
"""
import numpy as np
import pytest

from parity_util import FP32_TOL, max_rel_err, run_gpu
from paper_1905_00689_gb300 import LSTMApproxError, run_static
from workloads import draw_factor_set, draw_inputs

pytestmark = pytest.mark.gpu


def _pack(gates, D, H, K):
    """Masked-dense fp32 packing of one layer: Vx [4][K][D], Vh [4][K][H], U [4][H][K], sigma [4][K]."""
    Vx = np.zeros((4, K, D), np.float32)
    Vh = np.zeros((4, K, H), np.float32)
    U = np.zeros((4, H, K), np.float32)
    S = np.zeros((4, K), np.float32)
    for g, f in enumerate(gates):
        for k in range(K):
            for c, v in zip(f["idx"][k], f["val"][k]):
                if c < D:
                    Vx[g, k, c] = v
                else:
                    Vh[g, k, c - D] = v
        U[g] = f["u"][:K].T
        S[g] = f["sigma"][:K]
    return Vx, Vh, U, S


@pytest.mark.parametrize("D,H,T,B,K,nz,cps", [(1024, 512, 20, 1, 64, 384, [16, 64]),
                                              (40, 32, 6, 3, 12, 30, [5])])
def test_static_entry_point_matches_run(cuda_device, D, H, T, B, K, nz, cps):
    import torch
    gates = [draw_factor_set(H, D + H, K, nz, 6100 + 7 * D + g) for g in range(4)]
    x = draw_inputs(T, B, D, "relu", 61).astype(np.float32)
    ref, _ = run_gpu([gates], x, K, checkpoints=cps)

    dev = torch.device("cuda:0")
    Vx, Vh, U, S = (torch.from_numpy(a).to(dev) for a in _pack(gates, D, H, K))
    xt = torch.from_numpy(x).to(dev)
    for call in range(2):
        out_h = torch.full((T, B, H), float("nan"), device=dev)
        out_c = torch.full((1, B, H), float("nan"), device=dev)
        ck_h = torch.full((len(cps), T, B, H), float("nan"), device=dev)
        run_static(Vx, Vh, U, S, None, xt, K, out_h, out_c=out_c, checkpoints=cps, ckpt_h=ck_h)
        got = {"h": out_h.double().cpu().numpy(), "c_last": out_c.double().cpu().numpy(),
               "ckpt_h": ck_h.double().cpu().numpy()}
        for key in got:
            assert np.all(np.isfinite(got[key])), (call, key)
            err = max_rel_err(got[key], ref[key])
            assert err <= FP32_TOL, (call, key, err)


def test_static_entry_point_rejects_oversized_scratch(cuda_device):
    import torch
    D, H, K, T, B = 64, 64, 64, 2048, 2      # T*B*4K = 1,048,576 floats: above the fixed area
    dev = torch.device("cuda:0")
    Vx = torch.zeros((4, K, D), device=dev)
    Vh = torch.zeros((4, K, H), device=dev)
    U = torch.zeros((4, H, K), device=dev)
    S = torch.zeros((4, K), device=dev)
    x = torch.zeros((T, B, D), device=dev)
    out_h = torch.zeros((T, B, H), device=dev)
    with pytest.raises(LSTMApproxError) as ei:
        run_static(Vx, Vh, U, S, None, x, K, out_h)
    assert ei.value.code == 1 and "static scratch" in str(ei.value)
