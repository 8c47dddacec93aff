"""GPU parity of the fp32 path against the fp64 oracle (max relative error <= 1e-4).

Covers the persistent cluster kernel and the per-timestep CUDA-core kernels
on the two batch-1 workloads (D=64/H=64/T=8 and D=1024/H=512/T=20), with the
oracle's own residual decomposition where it is affordable and seeded
random factor sets of the same structure elsewhere, plus ragged and
degenerate shapes.
"""
import numpy as np
import pytest

from parity_util import (FP32_TOL, WORKLOADS, assert_parity, decomposed_layer, oracle_run, run_gpu,
                         synthetic_layer, workload_inputs)
from paper_1905_00689_gb300 import PATH_PERSISTENT, PATH_SIMT, Q_LAST_PATH
from workloads import draw_factor_set, draw_inputs

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("K", [1, 4, 16, 64])
@pytest.mark.parametrize("path", [PATH_PERSISTENT, PATH_SIMT])
def test_small_workload_decomposed_factors(cuda_device, K, path):
    w = WORKLOADS["c1"]
    layers = [list(decomposed_layer("c1", 0, 64, 0.5))]
    x = workload_inputs(w)
    got, m = run_gpu(layers, x, K, force_path=path)
    assert m.query(Q_LAST_PATH) == path
    ref = oracle_run(layers, x, K)
    assert_parity(got, ref, FP32_TOL)


@pytest.mark.parametrize("path", [PATH_PERSISTENT, PATH_SIMT])
def test_small_workload_checkpoints(cuda_device, path):
    w = WORKLOADS["c1"]
    layers = [list(decomposed_layer("c1", 0, 64, 0.5))]
    x = workload_inputs(w)
    cps = [1, 4, 16, 64]
    got, _ = run_gpu(layers, x, 64, checkpoints=cps, force_path=path)
    ref = oracle_run(layers, x, 64, checkpoints=cps)
    assert_parity(got, ref, FP32_TOL)
    assert np.array_equal(got["ckpt_h"][-1], got["h"])


@pytest.mark.parametrize("K", [16, 64, 256])
def test_latency_workload_full_size(cuda_device, K):
    """D=1024, H=512, T=20, B=1, keep 25%: the benchmark's launch configuration."""
    w = WORKLOADS["c2"]
    layers = [list(synthetic_layer("c2", 0, 256, 0.25))]
    x = workload_inputs(w)
    got, m = run_gpu(layers, x, K, max_rank=256)
    assert m.query(Q_LAST_PATH) == PATH_PERSISTENT
    ref = oracle_run(layers, x, K)
    assert_parity(got, ref, FP32_TOL)


def test_latency_workload_decomposed_factors(cuda_device):
    w = WORKLOADS["c2"]
    layers = [list(decomposed_layer("c2", 0, 16, 0.25))]
    x = workload_inputs(w, T=6)
    cps = [4, 8, 16]
    got, _ = run_gpu(layers, x, 16, checkpoints=cps)
    ref = oracle_run(layers, x, 16, checkpoints=cps)
    assert_parity(got, ref, FP32_TOL)


def test_latency_workload_progressive_outputs_in_one_run(cuda_device):
    w = WORKLOADS["c2"]
    layers = [list(synthetic_layer("c2", 0, 256, 0.25))]
    x = workload_inputs(w)
    cps = [16, 64, 256]
    got, _ = run_gpu(layers, x, 256, checkpoints=cps)
    ref = oracle_run(layers, x, 256, checkpoints=cps)
    assert_parity(got, ref, FP32_TOL)


@pytest.mark.parametrize("keep", WORKLOADS["f1"].keeps)
@pytest.mark.parametrize("K", [4, 16])
def test_paper_case_study_shape(cuda_device, keep, K):
    """The paper's case-study LSTM (Sec. VI): H = R = 64, C = 8320, fp32, NZ =
    4160 / 130 / 32, oracle-decomposed factors, three steps of one stream."""
    w = WORKLOADS["f1"]
    layers = [list(decomposed_layer("f1", 0, 16, keep))]
    x = draw_inputs(3, 1, w.D, w.x_dist, 8320 + K)
    cps = [5, 8] if K == 16 else [2]
    got, m = run_gpu(layers, x, K, checkpoints=cps, max_rank=16)
    assert m.query(Q_LAST_PATH) == PATH_PERSISTENT
    ref = oracle_run(layers, x, K, checkpoints=cps)
    assert_parity(got, ref, FP32_TOL)


@pytest.mark.parametrize("residual,nz_u", [(True, 16), (False, 0), (False, 24)])
def test_scheme_variants(cuda_device, residual, nz_u):
    """Factors of the scheme's variants (pruned u, non-residual truncated SVD)
    go through the same path: the kernels take any factor set."""
    import oracle
    from workloads import draw_weights, nz_from_keep
    w = WORKLOADS["c1"]
    K, nz = 32, nz_from_keep(0.5, w.C())
    gates = [oracle.decompose_gate_variant(W, K, nz, residual=residual, nz_u=nz_u) for W in draw_weights(w, 0)]
    x = workload_inputs(w)
    got, _ = run_gpu([gates], x, K, checkpoints=[8, 20])
    ref = oracle_run([gates], x, K, checkpoints=[8, 20])
    assert_parity(got, ref, FP32_TOL)


@pytest.mark.parametrize("cs", [1, 2, 4, 8, 16])
def test_every_cluster_size_agrees(cuda_device, cs):
    D, H, T, K = 96, 64, 5, 64
    layers = [[draw_factor_set(H, D + H, K, 40, 900 + g) for g in range(4)]]
    x = draw_inputs(T, 1, D, "relu", 21)
    got, m = run_gpu(layers, x, K, cluster=cs, force_path=PATH_PERSISTENT, checkpoints=[8, 33])
    ref = oracle_run(layers, x, K, checkpoints=[8, 33])
    assert_parity(got, ref, FP32_TOL)


@pytest.mark.parametrize("D,H,T,B,K,nz,cps", [
    (5, 12, 3, 3, 7, 9, [1, 3, 5]),        # ragged sizes, unaligned depths, several streams
    (24, 36, 4, 2, 1, 60, [1]),            # K = 1, nothing pruned (nz = C)
    (40, 100, 2, 1, 50, 1, [25, 49]),      # one kept entry per term
    (3, 4, 1, 1, 3, 2, []),                # T = 1
    (64, 44, 6, 5, 33, 17, [2, 32, 33]),
])
@pytest.mark.parametrize("path", [PATH_PERSISTENT, PATH_SIMT])
def test_ragged_and_degenerate_shapes(cuda_device, D, H, T, B, K, nz, cps, path):
    C = D + H
    gates = [draw_factor_set(H, C, K, nz, 7000 + 13 * D + g) for g in range(4)]
    rng = np.random.default_rng(D * H)
    for g in gates:
        g["bias"] = 0.3 * rng.standard_normal(H)
    x = draw_inputs(T, B, D, "uniform", 55 + D)
    h0 = 0.5 * rng.standard_normal((1, B, H))
    c0 = 0.5 * rng.standard_normal((1, B, H))
    if path == PATH_PERSISTENT and H % 4:
        pytest.skip("persistent kernel needs H % 4 == 0")
    got, m = run_gpu([gates], x, K, h0=h0, c0=c0, checkpoints=cps, force_path=path)
    ref = oracle_run([gates], x, K, h0=h0, c0=c0, checkpoints=cps)
    assert_parity(got, ref, FP32_TOL)


def test_two_layer_stack_fp32(cuda_device):
    D, H, T, B, K = 48, 32, 5, 2, 12
    layers = [[draw_factor_set(H, (D if l == 0 else H) + H, K, 20, 800 + 10 * l + g) for g in range(4)]
              for l in range(2)]
    x = draw_inputs(T, B, D, "uniform", 3)
    for path in (PATH_PERSISTENT, PATH_SIMT):
        got, _ = run_gpu(layers, x, K, checkpoints=[3, 12], force_path=path)
        ref = oracle_run(layers, x, K, checkpoints=[3, 12])
        assert_parity(got, ref, FP32_TOL)


def test_masks_read_back_bit_exact(cuda_device):
    layers = [list(decomposed_layer("c1", 0, 64, 0.5))]
    x = workload_inputs(WORKLOADS["c1"])
    _, m = run_gpu(layers, x, 4)
    for g, f in enumerate(layers[0]):
        for k in range(64):
            assert np.array_equal(m.get_mask(0, g, k), f["idx"][k])
    syn = list(synthetic_layer("c2", 0, 256, 0.25))
    _, m2 = run_gpu([syn], workload_inputs(WORKLOADS["c2"], T=1), 16, max_rank=256)
    for g, f in enumerate(syn):
        for k in (0, 1, 100, 255):
            assert np.array_equal(m2.get_mask(0, g, k), f["idx"][k])


def test_host_buffer_entry_point_matches_device_run(cuda_device):
    w = WORKLOADS["c2"]
    layers = [list(synthetic_layer("c2", 0, 64, 0.25))]
    x = workload_inputs(w).astype(np.float32)
    got, m = run_gpu(layers, x, 64, checkpoints=[16])
    out_h = np.zeros((w.T, 1, w.H), np.float32)
    out_c = np.zeros((1, 1, w.H), np.float32)
    ck_h = np.zeros((1, w.T, 1, w.H), np.float32)
    m.run_host(np.ascontiguousarray(x), 64, out_h, out_c=out_c, checkpoints=[16], ckpt_h=ck_h)
    assert np.array_equal(out_h.astype(np.float64), got["h"])
    assert np.array_equal(out_c.astype(np.float64), got["c_last"])
    assert np.array_equal(ck_h.astype(np.float64), got["ckpt_h"])


@pytest.mark.parametrize("xproj", [1, 2])
@pytest.mark.parametrize("wl,keep,K,cps", [("c2", 0.25, 256, [16, 64]), ("c1", 0.5, 64, [4, 16]),
                                           ("f1", 130 / 8320, 16, [5])])
def test_both_input_projections(cuda_device, xproj, wl, keep, K, cps):
    """The masked-dense and the compressed projection kernels, each forced, on
    the batch-1 workloads (the automatic choice runs only one per shape)."""
    w = WORKLOADS[wl]
    layers = [list(synthetic_layer(wl, 0, K, keep))]
    x = workload_inputs(w, T=min(w.T, 6))
    got, m = run_gpu(layers, x, K, checkpoints=cps, max_rank=K, xproj=xproj)
    ref = oracle_run(layers, x, K, checkpoints=cps)
    assert_parity(got, ref, FP32_TOL)


@pytest.mark.parametrize("pinned", [False, True])
def test_host_entry_pinned_and_pageable_buffers(cuda_device, pinned):
    """lstm_approx_run_host writes out_h and the checkpoints in place when
    they are page-locked, and stages them otherwise: both give the device
    run's outputs bit for bit (with initial states and the final c, which
    are always staged)."""
    import torch
    w = WORKLOADS["c2"]
    layers = [list(synthetic_layer("c2", 0, 64, 0.25))]
    x = workload_inputs(w, T=7).astype(np.float32)
    rng = np.random.default_rng(5)
    h0 = (0.3 * rng.standard_normal((1, 1, w.H))).astype(np.float32)
    c0 = (0.3 * rng.standard_normal((1, 1, w.H))).astype(np.float32)
    got, m = run_gpu(layers, x, 64, h0=h0, c0=c0, checkpoints=[16, 40])

    def buf(shape, src=None):
        t = torch.zeros(shape, dtype=torch.float32)
        if pinned:
            t = t.pin_memory()
        if src is not None:
            t.copy_(torch.from_numpy(src))
        return t
    xt, oh, oc = buf(x.shape, x), buf((7, 1, w.H)), buf((1, 1, w.H))
    kh, kc = buf((2, 7, 1, w.H)), buf((2, 7, 1, w.H))
    assert xt.is_pinned() == pinned
    m.run_host(xt.numpy(), 64, oh.numpy(), h0=buf(h0.shape, h0).numpy(), c0=buf(c0.shape, c0).numpy(),
               out_c=oc.numpy(), checkpoints=[16, 40], ckpt_h=kh.numpy(), ckpt_c=kc.numpy())
    assert np.array_equal(oh.numpy().astype(np.float64), got["h"])
    assert np.array_equal(oc.numpy().astype(np.float64), got["c_last"])
    assert np.array_equal(kh.numpy().astype(np.float64), got["ckpt_h"])
    assert np.array_equal(kc.numpy().astype(np.float64), got["ckpt_c"])


@pytest.mark.parametrize("dtype,B", [("fp32", 1), ("fp32", 3), ("bf16", 5)])
def test_input_view_not_16_byte_aligned(cuda_device, dtype, B):
    """x passed as a view 4 bytes into its allocation: the kernels that copy
    x in 16-byte pieces are not taken (the result equals the oracle's)."""
    import torch
    from paper_1905_00689_gb300 import LSTMApprox
    D, H, T, K = 64, 64, 5, 16
    gates = [draw_factor_set(H, D + H, K, 60, 6800 + g) for g in range(4)]
    x = draw_inputs(T, B, D, "uniform", 12).astype(np.float32)
    dev = torch.device("cuda:0")
    buf = torch.zeros(T * B * D + 4, device=dev)
    xv = buf[1:1 + T * B * D].view(T, B, D)
    assert xv.data_ptr() % 16 == 4
    xv.copy_(torch.from_numpy(x))
    m = LSTMApprox(1, [D], H, K, B, dtype)
    m.set_layer(0, gates)
    out = torch.full((T, B, H), float("nan"), device=dev)
    m.run(xv, K, out)
    m.sync()
    ref = oracle_run([gates], x, K, dtype=dtype)
    assert_parity({"h": out.double().cpu().numpy()}, ref, FP32_TOL if dtype == "fp32" else 2e-2, keys=("h",))
    m.close()
