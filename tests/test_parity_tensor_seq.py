"""GPU parity of the tensor-core path's one-launch kernel: all T timesteps
of a layer in one launch per tile of streams (bf16 factors, K <= 32,
H = 256, 512 or 1024; k_tensor_seq.cu).

Each case is checked against the oracle on the factors as the library
stores them, and against the two-launches-per-step kernels on the same
inputs (the same arithmetic except the order in which the partial tau'
sums of the cluster's CTAs are added).
"""
import numpy as np
import pytest

from parity_util import BF16_TOL, WORKLOADS, assert_parity, oracle_run, run_gpu, synthetic_layer, workload_inputs
from paper_1905_00689_gb300 import (LSTMApproxError, OPT_TEST_STALL, OPT_WAIT_LIMIT, PATH_TENSOR, Q_LAST_PATH,
                                    Q_TENSOR_SEQ, plan, BF16)
from workloads import draw_factor_set, draw_inputs

pytestmark = pytest.mark.gpu


def _gates(H, C, K, nz, seed):
    gates = [draw_factor_set(H, C, K, nz, seed + g) for g in range(4)]
    rng = np.random.default_rng(seed)
    for g in gates:
        g["bias"] = 0.2 * rng.standard_normal(H)
    return gates


def _sample(got, streams):
    out = {"h": got["h"][:, streams]}
    if "c_last" in got:
        out["c_last"] = got["c_last"][:, streams]
    for k in ("ckpt_h", "ckpt_c"):
        if k in got:
            out[k] = got[k][:, :, streams]
    return out


@pytest.mark.parametrize("D,H,T,B,K,nz,cps", [
    (64, 256, 3, 32, 16, 90, []),            # two tiles of 2 CTAs x 8 streams
    (48, 256, 4, 37, 8, 60, [8]),            # ragged third tile; K = 8 (8 packed rows per gate), depth = K
    (96, 512, 3, 100, 32, 150, [16, 32]),    # 4 CTAs x 4 streams (half an 8-stream group), ragged tile, depths
    (40, 512, 2, 5, 17, 70, [16, 17]),       # 32 packed rows per gate, K and a depth off the slices
    (64, 1024, 3, 70, 32, 200, [16]),        # 4 CTAs x 256 units x 4 streams, ragged fifth tile
    (72, 1024, 2, 64, 1, 30, []),            # one term
    (56, 1024, 2, 40, 8, 50, [8]),           # 256 units per CTA with 8 packed rows per gate
])
def test_seq_kernel_small_shapes(cuda_device, D, H, T, B, K, nz, cps):
    gates = _gates(H, D + H, K, nz, 7100 + H + K)
    rng = np.random.default_rng(B)
    x = draw_inputs(T, B, D, "uniform", 70 + B)
    h0 = 0.3 * rng.standard_normal((1, B, H))
    c0 = 0.3 * rng.standard_normal((1, B, H))
    got, m = run_gpu([gates], x, K, dtype="bf16", h0=h0, c0=c0, checkpoints=cps)
    assert m.query(Q_LAST_PATH) == PATH_TENSOR and m.query(Q_TENSOR_SEQ) == 1
    ref = oracle_run([gates], x, K, dtype="bf16", h0=h0, c0=c0, checkpoints=cps)
    assert_parity(got, ref, BF16_TOL)
    step, m2 = run_gpu([gates], x, K, dtype="bf16", h0=h0, c0=c0, checkpoints=cps, tensor_seq=1)
    assert m2.query(Q_TENSOR_SEQ) == 0
    assert_parity(got, step, BF16_TOL)


@pytest.mark.parametrize("H,B,cs,ns", [(512, 700, 4, 32), (512, 1300, 4, 64), (1024, 700, 4, 32),
                                        (1024, 1200, 8, 64)])
def test_seq_kernel_wide_tiles(cuda_device, H, B, cs, ns):
    """More streams than one wave of narrower tiles holds: 32 streams per
    tile (8 per CTA), then 64 (H = 512: 16 per CTA of 128 units; H = 1024:
    8 per CTA, on clusters of 8 CTAs of 128 units instead of 4 of 256);
    sampled streams."""
    D, T, K = 32, 2, 32
    p = plan(BF16, H, T, B, K)
    assert (p["tau_tile_streams"], p["cluster"]) == (ns, cs)
    gates = _gates(H, D + H, K, 100, 7300)
    x = draw_inputs(T, B, D, "uniform", 73)
    got, m = run_gpu([gates], x, K, dtype="bf16", checkpoints=[16])
    assert m.query(Q_TENSOR_SEQ) == 1
    streams = [0, 15, 16, B // 2 + 3, B - 1]
    ref = oracle_run([gates], x[:, streams], K, dtype="bf16", checkpoints=[16])
    assert_parity(_sample(got, streams), ref, BF16_TOL)


def test_seq_kernel_two_layers(cuda_device):
    """Layer 0 hands its h sequence to layer 1 as the bf16 pair."""
    D, H, T, B, K = 80, 512, 3, 40, 32
    layers = [_gates(H, D + H, K, 120, 7400), _gates(H, 2 * H, K, 200, 7500)]
    x = draw_inputs(T, B, D, "relu", 74)
    got, m = run_gpu(layers, x, K, dtype="bf16", checkpoints=[16, 32])
    assert m.query(Q_TENSOR_SEQ) == 1
    ref = oracle_run(layers, x, K, dtype="bf16", checkpoints=[16, 32])
    assert_parity(got, ref, BF16_TOL)
    step, _ = run_gpu(layers, x, K, dtype="bf16", checkpoints=[16, 32], tensor_seq=1)
    assert_parity(got, step, BF16_TOL)


@pytest.mark.parametrize("K,cps", [(8, []), (24, [16]), (32, [16, 32])])
def test_seq_kernel_prefix_of_stored_terms(cuda_device, K, cps):
    """Runs below the stored rank: terms past K must contribute nothing."""
    D, H, T, B, KS = 64, 256, 3, 24, 96
    gates = _gates(H, D + H, KS, 60, 7600)
    x = draw_inputs(T, B, D, "uniform", 76)
    got, m = run_gpu([gates], x, K, dtype="bf16", checkpoints=cps, max_rank=KS)
    assert m.query(Q_TENSOR_SEQ) == 1
    ref = oracle_run([gates], x, K, dtype="bf16", checkpoints=cps)
    assert_parity(got, ref, BF16_TOL)


@pytest.mark.parametrize("wname,K,keep", [("c4", 8, 0.5), ("c4", 32, 0.1), ("c3", 32, 0.5)])
def test_seq_kernel_full_size(cuda_device, wname, K, keep):
    """The workloads' small depths at full size (D=2048 H=1024 B=1024 T=64;
    D=1024 H=512 B=256 T=20), with depths, on sampled streams."""
    w = WORKLOADS[wname]
    layers = [list(synthetic_layer(wname, 0, 512, keep))]
    x = workload_inputs(w)
    cps = [16, K] if K > 16 else [K]
    got, m = run_gpu(layers, x, K, dtype="bf16", max_rank=512, checkpoints=cps)
    assert m.query(Q_TENSOR_SEQ) == 1
    streams = [0, 63, 64, w.B - 1]
    ref = oracle_run(layers, x[:, streams], K, dtype="bf16", checkpoints=cps)
    assert_parity(_sample(got, streams), ref, BF16_TOL)


def test_seq_kernel_bounded_wait_reports_timeout(cuda_device):
    """The test hook makes CTA 0 of the first tile withhold its first partial
    tau': the owners' waits run out after the short limit, the run reports
    ETIMEOUT, and the next run on the handle is correct."""
    import torch
    D, H, T, B, K = 32, 256, 3, 32, 16
    gates = _gates(H, D + H, K, 40, 7700)
    x = draw_inputs(T, B, D, "uniform", 77)
    _, m = run_gpu([gates], x, K, dtype="bf16")
    assert m.query(Q_TENSOR_SEQ) == 1
    m.set_option(OPT_WAIT_LIMIT, 50_000)  # 50 ms
    m.set_option(OPT_TEST_STALL, 1)
    xt = torch.from_numpy(x.astype(np.float32)).cuda()
    out = torch.zeros((T, B, H), device="cuda")
    m.run(xt, K, out)
    with pytest.raises(LSTMApproxError) as ei:
        m.sync()
    assert ei.value.code == 4  # LSTM_APPROX_ETIMEOUT
    m.run(xt, K, out)
    m.sync()
    ref = oracle_run([gates], x, K, dtype="bf16")
    assert_parity({"h": out.double().cpu().numpy()}, ref, BF16_TOL, keys=("h",))
