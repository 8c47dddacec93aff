"""GPU parity of the bf16-factor path against the oracle (max relative error <= 2e-2).

The oracle is fed the factors exactly as the library stores them (sigma in
fp32, u and v rounded to bf16), so the tolerance measures the kernels'
error (bf16 operands, fp32 accumulation), not the storage rounding.
"""
import numpy as np
import pytest

from parity_util import BF16_TOL, WORKLOADS, assert_parity, oracle_run, run_gpu, synthetic_layer, workload_inputs
from paper_1905_00689_gb300 import PATH_SIMT
from workloads import draw_factor_set, draw_inputs

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("K", [32, 128])
def test_throughput_workload_shape_simt(cuda_device, K):
    w = WORKLOADS["c3"]
    layers = [list(synthetic_layer("c3", 0, 512, 0.5))]
    x = workload_inputs(w, T=6, B=16)
    got, _ = run_gpu(layers, x, K, dtype="bf16", force_path=PATH_SIMT, max_rank=512)
    ref = oracle_run(layers, x, K, dtype="bf16")
    assert_parity(got, ref, BF16_TOL)


def test_two_layer_progressive_simt(cuda_device):
    D, H, T, B, K = 96, 64, 4, 8, 64
    layers = [[draw_factor_set(H, (D if l == 0 else H) + H, K, int(0.3 * ((D if l == 0 else H) + H)),
                               1200 + 10 * l + g) for g in range(4)] for l in range(2)]
    x = draw_inputs(T, B, D, "uniform", 8)
    cps = [16, 32, 64]
    got, _ = run_gpu(layers, x, K, dtype="bf16", checkpoints=cps, force_path=PATH_SIMT)
    ref = oracle_run(layers, x, K, dtype="bf16", checkpoints=cps)
    assert_parity(got, ref, BF16_TOL)
