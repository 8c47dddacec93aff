"""Both persistent kernels against the fp64 oracle (fp32, max relative error <= 1e-4).

Variant 1 splits the hidden units over the cluster and exchanges tau' and
h every timestep; variant 2 gives each CTA a range of one gate's terms and
exchanges partial gate sums once per timestep, with every CTA running all
cells.  The cases below pin each variant explicitly (the automatic choice
only ever runs one of them for a shape): the two batch-1 workloads, every
cluster size of variant 2, intermediate depths on and inside the term
ranges (several inside one range, one at K), and ragged shapes.
"""
import numpy as np
import pytest

from parity_util import (FP32_TOL, WORKLOADS, assert_parity, decomposed_layer, oracle_run,
                         persistent_layout_cases, run_gpu, synthetic_layer, workload_inputs)
from paper_1905_00689_gb300 import (FP32, OPT_LAUNCH_ORDER, OPT_TIMING, PATH_PERSISTENT, Q_CLUSTER, Q_LAST_PATH,
                                    Q_LAUNCHES, Q_PERSISTENT_VARIANT, plan)
from workloads import draw_factor_set, draw_inputs

pytestmark = pytest.mark.gpu


def _check(layers, x, K, variant, cluster=0, **kw):
    got, m = run_gpu(layers, x, K, force_path=PATH_PERSISTENT, variant=variant, cluster=cluster, **kw)
    assert m.query(Q_LAST_PATH) == PATH_PERSISTENT
    assert m.query(Q_PERSISTENT_VARIANT) == variant
    if cluster:
        assert m.query(Q_CLUSTER) == cluster
    # the host-side plan of the same shape names the kernel that ran
    T, B = x.shape[:2]
    p = plan(FP32, layers[0][0]["u"].shape[1], T, B, K, kw.get("checkpoints", ()), PATH_PERSISTENT, cluster, variant)
    assert (m.query(Q_CLUSTER), m.query(Q_PERSISTENT_VARIANT)) == (p["cluster"], p["persistent_variant"])
    ref = oracle_run(layers, x, K, **{k: v for k, v in kw.items() if k in ("h0", "c0", "checkpoints")})
    assert_parity(got, ref, FP32_TOL)
    return got


@pytest.mark.parametrize("variant", [1, 2])
@pytest.mark.parametrize("K", [1, 4, 16, 64])
def test_small_workload(cuda_device, variant, K):
    layers = [list(decomposed_layer("c1", 0, 64, 0.5))]
    x = workload_inputs(WORKLOADS["c1"])
    cps = [c for c in (1, 4, 16, 64) if c <= K]
    got = _check(layers, x, K, variant, checkpoints=cps)
    assert np.array_equal(got["ckpt_h"][-1], got["h"])


@pytest.mark.parametrize("variant", [1, 2])
@pytest.mark.parametrize("K,cps", [(256, [16, 64]), (256, [16, 64, 100, 255]), (64, [3, 17, 40]), (16, [4, 8])])
def test_latency_workload_full_size(cuda_device, variant, K, cps):
    """D=1024, H=512, T=20, B=1, keep 25%: the benchmark's launch configuration."""
    layers = [list(synthetic_layer("c2", 0, 256, 0.25))]
    x = workload_inputs(WORKLOADS["c2"])
    _check(layers, x, K, variant, checkpoints=cps, max_rank=256)


@pytest.mark.parametrize("cs", [4, 8, 16])
@pytest.mark.parametrize("cps", [[8, 33], [1, 2, 3, 61, 64], [16, 32, 48]])
def test_one_exchange_every_cluster_size(cuda_device, cs, cps):
    """Cuts on range boundaries, inside ranges, several inside one range, at K."""
    D, H, T, K = 96, 64, 5, 64
    layers = [[draw_factor_set(H, D + H, K, 40, 900 + g) for g in range(4)]]
    x = draw_inputs(T, 1, D, "relu", 21)
    _check(layers, x, K, 2, cluster=cs, checkpoints=cps)


@pytest.mark.parametrize("D,H,T,B,K,nz,cps", [
    (5, 12, 3, 3, 7, 9, [1, 3, 5]),        # ragged sizes, unaligned depths, several streams
    (24, 36, 4, 2, 1, 60, [1]),            # K = 1, nothing pruned (nz = C)
    (40, 100, 2, 1, 50, 1, [25, 49]),      # one kept entry per term
    (3, 4, 1, 1, 3, 2, []),                # T = 1
    (64, 44, 6, 5, 33, 17, [2, 32, 33]),
    (16, 508, 3, 2, 255, 30, [1, 100, 254]),  # H and K just under the one-exchange limits
])
@pytest.mark.parametrize("variant", [1, 2])
def test_ragged_shapes(cuda_device, D, H, T, B, K, nz, cps, variant):
    C = D + H
    gates = [draw_factor_set(H, C, K, nz, 7000 + 13 * D + g) for g in range(4)]
    rng = np.random.default_rng(D * H)
    for g in gates:
        g["bias"] = 0.3 * rng.standard_normal(H)
    x = draw_inputs(T, B, D, "uniform", 55 + D)
    h0 = 0.5 * rng.standard_normal((1, B, H))
    c0 = 0.5 * rng.standard_normal((1, B, H))
    _check([gates], x, K, variant, h0=h0, c0=c0, checkpoints=cps)


def test_variants_agree_on_two_layers(cuda_device):
    D, H, T, B, K = 48, 32, 5, 2, 12
    layers = [[draw_factor_set(H, (D if l == 0 else H) + H, K, 20, 800 + 10 * l + g) for g in range(4)]
              for l in range(2)]
    x = draw_inputs(T, B, D, "uniform", 3)
    for variant in (1, 2):
        _check(layers, x, K, variant, checkpoints=[3, 12])


def test_one_exchange_rejects_what_it_cannot_hold(cuda_device):
    """H above 512 or K above 256: forcing variant 2 is an error, the automatic
    choice falls back to variant 1."""
    from paper_1905_00689_gb300 import LSTMApproxError
    D, H, T, K = 16, 520, 2, 8
    layers = [[draw_factor_set(H, D + H, K, 30, 50 + g) for g in range(4)]]
    x = draw_inputs(T, 1, D, "uniform", 5)
    with pytest.raises(LSTMApproxError):
        run_gpu(layers, x, K, force_path=PATH_PERSISTENT, variant=2)
    got, m = run_gpu(layers, x, K, force_path=PATH_PERSISTENT)
    assert m.query(Q_PERSISTENT_VARIANT) == 1
    assert_parity(got, oracle_run(layers, x, K), FP32_TOL)


@pytest.mark.parametrize("D,H,T,B,K", [(64, 64, 4, 16, 64), (96, 512, 3, 12, 64), (40, 128, 2, 40, 16)])
def test_many_streams_take_the_persistent_path(cuda_device, D, H, T, B, K):
    """fp32 runs with more streams than one wave of clusters holds still take
    a persistent kernel (the later clusters run in the next wave)."""
    gates = [draw_factor_set(H, D + H, K, (D + H) // 3, 60 + D + g) for g in range(4)]
    x = draw_inputs(T, B, D, "uniform", 7 + B)
    got, m = run_gpu([gates], x, K, checkpoints=[8])
    assert m.query(Q_LAST_PATH) == PATH_PERSISTENT
    ref = oracle_run([gates], x, K, checkpoints=[8])
    assert_parity(got, ref, FP32_TOL)


@pytest.mark.parametrize("D,H,T,K,nz,cps,cs,variant", [
    (256, 1024, 3, 128, 380, [16, 100], 0, 1),  # V_h in tensor memory, 32 h values per lane
    (200, 768, 4, 40, 290, [7, 40], 0, 1),      # the same with lanes past H reading zeros
    (128, 384, 3, 256, 150, [64, 130], 0, 1),   # V_h and U in tensor memory, 8 units per warp
    (128, 384, 3, 100, 150, [33], 8, 1),        # 16 units per warp
    (128, 384, 3, 100, 150, [33, 64], 0, 2),    # one-exchange kernel, four h quarters per thread
])
def test_wider_hidden_sizes(cuda_device, D, H, T, K, nz, cps, cs, variant):
    """Hidden sizes other than the workloads': each selects another
    instantiation of the kernel's on-chip layout."""
    layers = [[draw_factor_set(H, D + H, K, nz, 4400 + H + g) for g in range(4)]]
    x = draw_inputs(T, 1, D, "relu", H)
    rng = np.random.default_rng(H)
    h0 = 0.5 * rng.standard_normal((1, 1, H))
    c0 = 0.5 * rng.standard_normal((1, 1, H))
    _check(layers, x, K, variant, cluster=cs, checkpoints=cps, h0=h0, c0=c0)


# One case per compiled layout of the per-unit-block kernel (see
# parity_util.persistent_layout_cases), ragged hidden sizes, two depths.
@pytest.mark.parametrize("H,K,cs", persistent_layout_cases())
def test_per_unit_block_kernel_every_layout(cuda_device, H, K, cs):
    D, T = 40, 3
    layers = [[draw_factor_set(H, D + H, K, 30, 5100 + H + K + g) for g in range(4)]]
    x = draw_inputs(T, 1, D, "uniform", H + K)
    _check(layers, x, K, 1, cluster=cs, checkpoints=[K // 3, K - 7])


# The one-exchange kernel: each thread keeps HQ quarters of h (1 up to H = 128,
# 2 up to 256, 4 up to 512), at each cluster size.
@pytest.mark.parametrize("H", [100, 200, 340])
@pytest.mark.parametrize("cs,K", [(4, 60), (8, 120), (16, 250)])
def test_one_exchange_kernel_every_layout(cuda_device, H, cs, K):
    D, T = 40, 3
    layers = [[draw_factor_set(H, D + H, K, 30, 5300 + H + K + g) for g in range(4)]]
    x = draw_inputs(T, 1, D, "relu", H + K)
    _check(layers, x, K, 2, cluster=cs, checkpoints=[K // 3, K - 7])


def _run_again(m, x, K, H, checkpoints):
    import torch
    T, B, _ = x.shape
    xt = torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32)).cuda()
    out = torch.full((T, B, H), float("nan"), device="cuda")
    ck = torch.full((len(checkpoints), T, B, H), float("nan"), device="cuda")
    m.run(xt, K, out, checkpoints=list(checkpoints), ckpt_h=ck)
    m.sync()
    return {"h": out.double().cpu().numpy(), "ckpt_h": ck.double().cpu().numpy()}


def test_launch_orders_agree(cuda_device):
    """Batch 1, per-unit-block kernel: by default the recurrence is launched
    before its input projection and waits for the projection's per-CTA flags;
    with phase timing on, the projection comes first.  Both orders, several
    calls in a row (each call raises its flags with a new value), on the
    benchmark workload, against the oracle."""
    K, cps = 256, [16, 64]
    layers = [list(synthetic_layer("c2", 0, 256, 0.25))]
    x = workload_inputs(WORKLOADS["c2"])
    ref = oracle_run(layers, x, K, checkpoints=cps)
    got, m = run_gpu(layers, x, K, force_path=PATH_PERSISTENT, variant=1, checkpoints=cps, max_rank=256)
    assert_parity(got, ref, FP32_TOL)
    n0 = m.query(Q_LAUNCHES)
    for timing, order in ((0, 0), (1, 0), (0, 0), (0, 1), (0, 0)):
        m.set_option(OPT_TIMING, timing)
        m.set_option(OPT_LAUNCH_ORDER, order)
        again = _run_again(m, x, K, 512, cps)
        assert_parity(again, ref, FP32_TOL, keys=("h", "ckpt_h"))
    assert m.query(Q_LAUNCHES) - n0 == 5 * 2  # projection and recurrence in either order


def test_launch_orders_two_layer_stack(cuda_device):
    """Two fp32 layers of one stream: the second layer's recurrence (launched
    first) and projection read the first layer's outputs."""
    D, H, T, K = 64, 128, 6, 32
    layers = [[draw_factor_set(H, (D if l == 0 else H) + H, K, 60, 1700 + 10 * l + g) for g in range(4)]
              for l in range(2)]
    x = draw_inputs(T, 1, D, "uniform", 17)
    ref = oracle_run(layers, x, K, checkpoints=[8, 32])
    for timing in (0, 1):
        got, m = run_gpu(layers, x, K, force_path=PATH_PERSISTENT, variant=1, checkpoints=[8, 32])
        if timing:
            m.set_option(OPT_TIMING, 1)
            got = _run_again(m, x, K, H, [8, 32])
        assert m.query(Q_PERSISTENT_VARIANT) == 1
        assert_parity(got, ref, FP32_TOL, keys=("h", "ckpt_h"))


def test_blocking_launches_take_the_projection_first(cuda_device):
    """With CUDA_LAUNCH_BLOCKING=1 no two kernels run side by side: a handle
    created then starts with the projection first, and the batch-1 run of
    the per-unit-block kernel completes and matches the oracle."""
    import os
    import subprocess
    import sys
    here = os.path.dirname(os.path.abspath(__file__))
    code = (
        "import sys; sys.path[:0] = [%r, %r]\n"
        "import numpy as np\n"
        "from parity_util import FP32_TOL, assert_parity, decomposed_layer, oracle_run, run_gpu, WORKLOADS, "
        "workload_inputs\n"
        "from paper_1905_00689_gb300 import PATH_PERSISTENT\n"
        "layers = [list(decomposed_layer('c1', 0, 16, 0.5))]\n"
        "x = workload_inputs(WORKLOADS['c1'])\n"
        "got, m = run_gpu(layers, x, 16, force_path=PATH_PERSISTENT, variant=1, checkpoints=[4])\n"
        "assert_parity(got, oracle_run(layers, x, 16, checkpoints=[4]), FP32_TOL, keys=('h', 'ckpt_h'))\n"
        "print('ok')\n") % (here, os.path.dirname(here))
    env = dict(os.environ, CUDA_LAUNCH_BLOCKING="1")
    r = subprocess.run([sys.executable, "-c", code], env=env, capture_output=True, text=True, timeout=300)
    assert r.returncode == 0 and r.stdout.strip().endswith("ok"), r.stdout[-2000:] + r.stderr[-2000:]


def test_graph_replays_with_new_inputs(cuda_device):
    """A batch-1 run of the per-unit-block kernel captured into a CUDA graph
    (where the projection comes first) and replayed after the input changed
    in place matches the oracle on the new input each time."""
    import torch
    from paper_1905_00689_gb300 import LSTMApprox
    D, H, T, K = 96, 256, 5, 48
    layers = [[draw_factor_set(H, D + H, K, 120, 1800 + g) for g in range(4)]]
    xs = [draw_inputs(T, 1, D, "uniform", 30 + i) for i in range(3)]
    stream = torch.cuda.Stream()
    m = LSTMApprox(1, [D], H, K, 1, "fp32", stream=stream)
    m.set_layer(0, layers[0])
    from paper_1905_00689_gb300 import OPT_FORCE_PATH, OPT_PERSISTENT_VARIANT
    m.set_option(OPT_FORCE_PATH, PATH_PERSISTENT)
    m.set_option(OPT_PERSISTENT_VARIANT, 1)
    x = torch.from_numpy(xs[0].astype(np.float32)).cuda()
    out = torch.zeros((T, 1, H), device="cuda")
    ck = torch.zeros((1, T, 1, H), device="cuda")
    torch.cuda.synchronize()
    with torch.cuda.stream(stream):
        m.run(x, K, out, checkpoints=[8], ckpt_h=ck)  # eager, recurrence first
    m.sync()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        m.run(x, K, out, checkpoints=[8], ckpt_h=ck)
    for xi in xs[1:] + xs[:1]:
        with torch.cuda.stream(stream):
            x.copy_(torch.from_numpy(xi.astype(np.float32)))
            g.replay()
        stream.synchronize()
        ref = oracle_run(layers, xi, K, checkpoints=[8])
        assert_parity({"h": out.double().cpu().numpy(), "ckpt_h": ck.double().cpu().numpy()}, ref, FP32_TOL,
                      keys=("h", "ckpt_h"))
    assert m.query(Q_PERSISTENT_VARIANT) == 1
