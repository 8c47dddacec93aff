"""GPU parity of the tensor-core path (bf16 factors, fp32 accumulate).

The oracle receives the factors as the library stores them (sigma fp32,
u and v bf16); the activations x, h and tau' enter the MMAs as bf16 pairs
(hi + lo), so the elementwise bound 2e-2 holds with a wide margin (the
errors are a few 1e-4).  Full-size workloads are checked on sampled streams
(streams are independent, so the oracle runs on those streams alone).
"""
import numpy as np
import pytest

from parity_util import (BF16_TOL, WORKLOADS, assert_parity, decomposed_layer, oracle_run, run_gpu,
                         synthetic_layer, workload_inputs)
from paper_1905_00689_gb300 import BF16, PATH_SIMT, PATH_TENSOR, Q_LAST_PATH, plan
from workloads import draw_factor_set, draw_inputs

pytestmark = pytest.mark.gpu


def _sample(got, streams, T=None):
    out = {"h": got["h"][:, streams]}
    if "c_last" in got:
        out["c_last"] = got["c_last"][:, streams]
    for k in ("ckpt_h", "ckpt_c"):
        if k in got:
            out[k] = got[k][:, :, streams]
    return out


@pytest.mark.parametrize("D,H,T,B,K,nz,cps", [
    (64, 128, 3, 16, 64, 96, []),            # one tile of everything
    (40, 200, 4, 3, 80, 70, [16, 48, 80]),    # ragged H, B, K; depths inside and at the end of chunks
    (300, 136, 2, 130, 128, 150, [64]),       # two stream tiles, ragged tail
    # one output tile: the gate GEMM's terms split 4 and 8 ways, depths on
    # split boundaries, inside splits and at K
    (48, 128, 3, 8, 256, 100, [64, 96, 128, 192, 256]),
    (32, 128, 2, 4, 512, 60, [16, 320, 512]),
    # depths off the 16-term slices: below the first slice, inside a slice,
    # at the start of a split's range (no MMA issued before the cut), and
    # at K when K is not a multiple of 16
    (40, 200, 4, 3, 80, 70, [5, 21, 79]),
    (48, 128, 3, 8, 256, 100, [5, 67, 130, 200, 256]),
    (64, 136, 2, 40, 45, 80, [1, 17, 45]),
    # tau' with its reduction axis (H >= 1024) split over clusters of 4 CTAs:
    # ragged H (the last split shorter), K off the 128-row tiles, two tiles
    # of 64 streams with a ragged tail
    (64, 1000, 3, 70, 200, 300, [16, 200]),
    (32, 1024, 2, 9, 130, 400, [64, 129]),
])
def test_tensor_path_small_shapes(cuda_device, D, H, T, B, K, nz, cps):
    gates = [draw_factor_set(H, D + H, K, nz, 5100 + 7 * D + g) for g in range(4)]
    rng = np.random.default_rng(H)
    for g in gates:
        g["bias"] = 0.2 * rng.standard_normal(H)
    x = draw_inputs(T, B, D, "uniform", 66)
    h0 = 0.3 * rng.standard_normal((1, B, H))
    c0 = 0.3 * rng.standard_normal((1, B, H))
    got, m = run_gpu([gates], x, K, dtype="bf16", h0=h0, c0=c0, checkpoints=cps, force_path=PATH_TENSOR)
    assert m.query(Q_LAST_PATH) == PATH_TENSOR
    if H >= 1000:  # the cases above meant to split tau'
        assert plan(BF16, H, T, B, K, cps, PATH_TENSOR)["tau_splits"] == 4
    ref = oracle_run([gates], x, K, dtype="bf16", h0=h0, c0=c0, checkpoints=cps)
    assert_parity(got, ref, BF16_TOL)


def test_tensor_path_matches_cuda_core_path(cuda_device):
    """Same factors through both bf16 paths: agreement well inside the bound."""
    D, H, T, B, K = 96, 256, 5, 40, 96
    gates = [draw_factor_set(H, D + H, K, 120, 5300 + g) for g in range(4)]
    x = draw_inputs(T, B, D, "relu", 2)
    a, _ = run_gpu([gates], x, K, dtype="bf16", checkpoints=[32], force_path=PATH_TENSOR)
    b, _ = run_gpu([gates], x, K, dtype="bf16", checkpoints=[32], force_path=PATH_SIMT)
    assert_parity(a, b, BF16_TOL)


@pytest.mark.parametrize("K", [32, 128, 512])
@pytest.mark.parametrize("with_depths", [False, True])
def test_throughput_workload_full_size(cuda_device, K, with_depths):
    """D=1024, H=512, T=20, B=256, keep 50%, at each K of the workload, with
    and without intermediate depths (one off the 16-term slices): checked on
    sampled streams."""
    w = WORKLOADS["c3"]
    layers = [list(synthetic_layer("c3", 0, 512, 0.5))]
    x = workload_inputs(w)
    cps = [16, K // 2 + 3, K] if with_depths else []
    got, m = run_gpu(layers, x, K, dtype="bf16", max_rank=512, checkpoints=cps)
    assert m.query(Q_LAST_PATH) == PATH_TENSOR
    streams = [0, 77, 255]
    ref = oracle_run(layers, x[:, streams], K, dtype="bf16", checkpoints=cps)
    assert_parity(_sample(got, streams), ref, BF16_TOL)


@pytest.mark.parametrize("K,cps", [(8, []), (24, [16]), (40, [16, 32]), (40, [3, 33, 40])])
def test_prefix_of_stored_terms(cuda_device, K, cps):
    """Runs at K below the stored rank, with K not a multiple of the MMA's 16
    terms: the terms past K in the last slice must contribute nothing."""
    D, H, T, B, KS = 72, 128, 3, 24, 96
    gates = [draw_factor_set(H, D + H, KS, 60, 6100 + g) for g in range(4)]
    x = draw_inputs(T, B, D, "uniform", 8)
    got, m = run_gpu([gates], x, K, dtype="bf16", checkpoints=cps, force_path=PATH_TENSOR, max_rank=KS)
    assert m.query(Q_LAST_PATH) == PATH_TENSOR
    ref = oracle_run([gates], x, K, dtype="bf16", checkpoints=cps)
    assert_parity(got, ref, BF16_TOL)


def test_widest_stream_tile(cuda_device):
    """Enough gate tiles that the gate GEMM takes 128 streams per tile
    (10 unit tiles x 16 tiles of 64 streams would exceed one wave); ragged
    last tile, checked on sampled streams."""
    D, H, T, B, K = 64, 1280, 2, 1000, 48
    gates = [draw_factor_set(H, D + H, K, 200, 6300 + g) for g in range(4)]
    x = draw_inputs(T, B, D, "uniform", 31)
    got, m = run_gpu([gates], x, K, dtype="bf16", checkpoints=[16, 32], force_path=PATH_TENSOR)
    assert m.query(Q_LAST_PATH) == PATH_TENSOR
    streams = [0, 517, 895, 999]
    ref = oracle_run([gates], x[:, streams], K, dtype="bf16", checkpoints=[16, 32])
    assert_parity(_sample(got, streams), ref, BF16_TOL)


def test_throughput_workload_decomposed_factors(cuda_device):
    w = WORKLOADS["c3"]
    layers = [list(decomposed_layer("c3", 0, 32, 0.5))]
    x = workload_inputs(w, T=4, B=64)
    got, _ = run_gpu(layers, x, 32, dtype="bf16", checkpoints=[16, 32])
    ref = oracle_run(layers, x, 32, dtype="bf16", checkpoints=[16, 32])
    assert_parity(got, ref, BF16_TOL)


@pytest.mark.parametrize("keep", [0.5, 0.1])
@pytest.mark.parametrize("K", [8, 32, 128, 512])
def test_large_batch_workload_full_size(cuda_device, keep, K):
    """D=2048, H=1024, T=64, B=1024 at every K and keep level of the
    workload (prefixes of one 512-term factor set): checked on sampled
    streams."""
    w = WORKLOADS["c4"]
    layers = [list(synthetic_layer("c4", 0, 512, keep))]
    x = workload_inputs(w)
    got, _ = run_gpu(layers, x, K, dtype="bf16", max_rank=512)
    streams = [0, 513, 1023]
    ref = oracle_run(layers, x[:, streams], K, dtype="bf16")
    assert_parity(_sample(got, streams), ref, BF16_TOL)


def test_two_layer_progressive_workload_full_size(cuda_device):
    """2 layers, D=4096, H=2048, T=16, B=64, K=1024, outputs at 16/64/256/1024."""
    w = WORKLOADS["c5"]
    layers = [list(synthetic_layer("c5", l, 1024, 0.3)) for l in range(2)]
    x = workload_inputs(w)
    cps = list(w.checkpoints)
    got, _ = run_gpu(layers, x, 1024, dtype="bf16", checkpoints=cps, max_rank=1024)
    streams = [5, 63]
    ref = oracle_run(layers, x[:, streams], 1024, dtype="bf16", checkpoints=cps)
    assert_parity(_sample(got, streams), ref, BF16_TOL)


def test_two_layer_unaligned_depths_automatic_path(cuda_device):
    """Two bf16 layers, no forced path, a depth off the 16-term slices: every
    layer takes the tensor path (the sequence between layers stays in the
    tensor path's bf16 pair planes)."""
    from paper_1905_00689_gb300 import BF16, plan
    D, H, T, B, K = 72, 96, 4, 12, 48
    layers = [[draw_factor_set(H, (D if l == 0 else H) + H, K, int(0.4 * ((D if l == 0 else H) + H)),
                               6600 + 10 * l + g) for g in range(4)] for l in range(2)]
    x = draw_inputs(T, B, D, "uniform", 9)
    cps = [5, K]
    got, m = run_gpu(layers, x, K, dtype="bf16", checkpoints=cps)
    assert m.query(Q_LAST_PATH) == PATH_TENSOR == plan(BF16, H, T, B, K, cps)["path"]
    ref = oracle_run(layers, x, K, dtype="bf16", checkpoints=cps)
    assert_parity(got, ref, BF16_TOL)


def test_two_layer_simt_forced_unaligned_depths(cuda_device):
    """The same stack forced onto the CUDA-core kernels for every layer."""
    D, H, T, B, K = 72, 96, 4, 12, 48
    layers = [[draw_factor_set(H, (D if l == 0 else H) + H, K, int(0.4 * ((D if l == 0 else H) + H)),
                               6600 + 10 * l + g) for g in range(4)] for l in range(2)]
    x = draw_inputs(T, B, D, "uniform", 9)
    got, m = run_gpu(layers, x, K, dtype="bf16", checkpoints=[5, K], force_path=PATH_SIMT)
    assert m.query(Q_LAST_PATH) == PATH_SIMT
    ref = oracle_run(layers, x, K, dtype="bf16", checkpoints=[5, K])
    assert_parity(got, ref, BF16_TOL)


def test_large_batch_workload_decomposed_factors(cuda_device):
    """D=2048, H=1024, T=64, B=1024, keep 50%, with the oracle's own residual
    decomposition of the workload's Gaussian gate matrices (K = 16, the top
    triplets by the Lanczos iteration) and depths 5 and 16: sampled streams."""
    w = WORKLOADS["c4"]
    layers = [list(decomposed_layer("c4", 0, 16, 0.5))]
    x = workload_inputs(w)
    cps = [5, 16]
    got, m = run_gpu(layers, x, 16, dtype="bf16", checkpoints=cps)
    assert m.query(Q_LAST_PATH) == PATH_TENSOR
    streams = [0, 700, 1023]
    ref = oracle_run(layers, x[:, streams], 16, dtype="bf16", checkpoints=cps)
    assert_parity(_sample(got, streams), ref, BF16_TOL)


def test_two_layer_workload_decomposed_factors(cuda_device):
    """The two-layer D=4096, H=2048, T=16, B=64 workload (keep 30%) with the
    oracle's decomposition of both layers' gate matrices (K = 8) and depths
    3 and 8: sampled streams."""
    w = WORKLOADS["c5"]
    layers = [list(decomposed_layer("c5", l, 8, 0.3)) for l in range(2)]
    x = workload_inputs(w)
    cps = [3, 8]
    got, _ = run_gpu(layers, x, 8, dtype="bf16", checkpoints=cps)
    streams = [2, 41]
    ref = oracle_run(layers, x[:, streams], 8, dtype="bf16", checkpoints=cps)
    assert_parity(_sample(got, streams), ref, BF16_TOL)


@pytest.mark.parametrize("D,H,T,B,K,nz,cps", [
    (40, 200, 4, 3, 80, 70, [5, 21, 79]),      # ragged H, B, K; depths off the slices
    (64, 136, 2, 40, 45, 80, [17, 45]),        # two stream tiles, ragged tail
    (48, 128, 3, 8, 256, 100, [64, 130]),      # many rows, term split of the gate GEMM
    (32, 96, 3, 5, 8, 20, []),                 # packed gates (K <= 32)
])
def test_compressed_tau_layout(cuda_device, D, H, T, B, K, nz, cps):
    """The compressed layout of v's h part (kept entries per row, CUDA cores)
    for the recurrent projection, against the oracle."""
    gates = [draw_factor_set(H, D + H, K, nz, 5400 + 7 * D + g) for g in range(4)]
    x = draw_inputs(T, B, D, "uniform", 67)
    got, m = run_gpu([gates], x, K, dtype="bf16", checkpoints=cps, tau_layout=1)
    assert m.query(Q_LAST_PATH) == PATH_TENSOR
    ref = oracle_run([gates], x, K, dtype="bf16", checkpoints=cps)
    assert_parity(got, ref, BF16_TOL)


@pytest.mark.parametrize("keep,K", [(0.1, 128), (0.5, 512)])
def test_compressed_tau_layout_large_batch_full_size(cuda_device, keep, K):
    """D=2048, H=1024, T=64, B=1024 with the compressed tau' layout: sampled streams."""
    w = WORKLOADS["c4"]
    layers = [list(synthetic_layer("c4", 0, 512, keep))]
    x = workload_inputs(w)
    got, _ = run_gpu(layers, x, K, dtype="bf16", max_rank=512, tau_layout=1)
    streams = [0, 513, 1023]
    ref = oracle_run(layers, x[:, streams], K, dtype="bf16")
    assert_parity(_sample(got, streams), ref, BF16_TOL)


def test_compressed_tau_layout_refused_where_it_does_not_apply(cuda_device):
    from paper_1905_00689_gb300 import LSTMApprox, LSTMApproxError, OPT_TAU_LAYOUT
    m = LSTMApprox(1, [8], 16, 4, 1, "fp32")
    with pytest.raises(LSTMApproxError):
        m.set_option(OPT_TAU_LAYOUT, 1)
    m.close()
    m = LSTMApprox(1, [8], 2048, 4, 1, "bf16")
    with pytest.raises(LSTMApproxError):
        m.set_option(OPT_TAU_LAYOUT, 1)
    m.close()


@pytest.mark.parametrize("K", [16, 200])
@pytest.mark.parametrize("D,offset", [(64, 0), (42, 0), (64, 1)])
def test_projection_input_forms(cuda_device, D, offset, K):
    """Up to K = 32 at layer 0 the projection reads x in fp32 and forms its
    bf16 pair itself when D is a multiple of 4 and x is 16-byte aligned;
    otherwise (and at K = 200, two 128-row tiles per gate) x goes through
    the separate conversion pass.  All agree with the oracle (offset = 1: x
    starts one float into its buffer)."""
    import torch
    from paper_1905_00689_gb300 import LSTMApprox
    H, T, B = 256, 3, 20
    gates = [draw_factor_set(H, D + H, K, 70, 6600 + D + K + g) for g in range(4)]
    x = draw_inputs(T, B, D, "uniform", 9)
    m = LSTMApprox(1, [D], H, K, B, "bf16")
    m.set_layer(0, gates)
    buf = torch.zeros(T * B * D + 4, device="cuda")
    xt = buf[offset:offset + T * B * D].view(T, B, D)
    xt.copy_(torch.from_numpy(x.astype(np.float32)))
    out = torch.empty((T, B, H), device="cuda")
    m.run(xt, K, out)
    m.sync()
    ref = oracle_run([gates], x, K, dtype="bf16")
    assert_parity({"h": out.double().cpu().numpy()}, ref, BF16_TOL, keys=("h",))
