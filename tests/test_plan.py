"""The library's kernel planning on the host (no GPU): lstm_approx_plan.

The run and lstm_approx_plan take their decisions from the same functions;
these tests pin those decisions to the rules stated for them (which path,
which persistent kernel, how a CTA's share is laid out, how the tensor-core
GEMMs are tiled and split) and check that every plan covers its shape and
fits the SM (shared memory, tensor memory).
"""
import pytest

from parity_util import persistent_layout_cases
from paper_1905_00689_gb300 import (BF16, FP32, PATH_PERSISTENT, PATH_SIMT, PATH_TENSOR, LSTMApproxError, plan)


@pytest.fixture(scope="module", autouse=True)
def built_lib():
    from paper_1905_00689_gb300 import build as b
    b.build()


def _pow2_at_least(n):
    p = 1
    while p < n:
        p *= 2
    return p


def _round4(n):
    return (n + 3) & ~3


# ---- the workloads -----------------------------------------------------------

def test_batch_one_workloads():
    # D=1024, H=512, T=20, K=256 with depths 16 and 64: per-unit-block kernel
    # on 16 CTAs (one-exchange share 512 x 64 terms is above 16384)
    p = plan(FP32, 512, 20, 1, 256, [16, 64])
    assert (p["path"], p["persistent_variant"], p["cluster"]) == (PATH_PERSISTENT, 1, 16)
    assert (p["terms_per_cta"], p["units_per_warp"], p["terms_per_lane"], p["vh_layout"]) == (64, 8, 8, 1)
    # the same at K = 16: one-exchange kernel on 4 CTAs
    p = plan(FP32, 512, 20, 1, 16)
    assert (p["persistent_variant"], p["cluster"], p["terms_per_cta"], p["h_quads"]) == (2, 4, 16, 4)
    # D = H = 64, T = 8, K = 64
    p = plan(FP32, 64, 8, 1, 64)
    assert (p["persistent_variant"], p["cluster"], p["terms_per_cta"], p["h_quads"]) == (2, 4, 64, 1)


def test_large_batch_workloads():
    # D=1024, H=512, B=256, K=512: 4 unit tiles x 8 tiles of 32 streams, the
    # terms split 4 ways to fill the GPU
    p = plan(BF16, 512, 20, 256, 512)
    assert (p["path"], p["gate_tile_streams"], p["gate_splits"], p["tau_tile_streams"], p["tau_splits"]) == \
        (PATH_TENSOR, 32, 4, 32, 1)
    # D=2048, H=1024, B=1024, K=512: 8 x 16 tiles of 64 streams, no split;
    # the tau' GEMM's 16 row tiles take 128 streams per tile
    p = plan(BF16, 1024, 64, 1024, 512)
    assert (p["gate_tile_streams"], p["gate_splits"], p["tau_tile_streams"], p["tau_splits"]) == (64, 1, 128, 1)
    # the same at K = 128: 4 row tiles x 32 tiles of 32 streams
    p = plan(BF16, 1024, 64, 1024, 128)
    assert (p["tau_tile_streams"], p["tau_splits"]) == (32, 1)
    # second layer of D=4096, H=2048, B=64, K=1024 with four depths (tau':
    # 32 row tiles of 64 streams, H split over clusters of 4)
    p = plan(BF16, 2048, 16, 64, 1024, [16, 64, 256, 1024])
    assert (p["path"], p["gate_tile_streams"], p["gate_splits"], p["tau_tile_streams"], p["tau_splits"]) == \
        (PATH_TENSOR, 32, 4, 64, 4)


# ---- the rules -----------------------------------------------------------------

@pytest.mark.parametrize("H,K,cs", persistent_layout_cases())
def test_per_unit_block_layout_rule(H, K, cs):
    """Units per warp: the smallest power of two with 4 UW >= the CTA's
    units (ceil(H / CS) rounded up to 4); terms per lane: the smallest power
    of two with 32 KT >= K; V_h in shared memory up to H = 256, in tensor
    memory with U up to 512, at 32 values per lane above."""
    p = plan(FP32, H, 3, 1, K, [K // 3, K - 7], PATH_PERSISTENT, cs, 1)
    assert p["cluster"] == cs and p["persistent_variant"] == 1
    assert p["units_per_warp"] == _pow2_at_least(_round4(-(-H // cs)) // 4)
    assert p["terms_per_lane"] == _pow2_at_least(-(-K // 32))
    assert p["vh_layout"] == (0 if H <= 256 else 1 if H <= 512 else 2)


def test_layout_cases_cover_every_compiled_layout():
    """The GPU parity cases of the per-unit-block kernel reach each compiled
    combination once: units per warp 1..16 and terms per lane 1..8 with V_h
    in shared memory (16 units per warp up to 4 terms per lane), and the
    tensor-memory layouts."""
    got = set()
    for H, K, cs in persistent_layout_cases():
        p = plan(FP32, H, 3, 1, K, [K // 3, K - 7], PATH_PERSISTENT, cs, 1)
        got.add((p["units_per_warp"], p["terms_per_lane"], p["vh_layout"]))
    want = {(uw, kt, 0) for uw in (1, 2, 4, 8) for kt in (1, 2, 4, 8)} | {(16, kt, 0) for kt in (1, 2, 4)}
    want |= {(8, kt, 1) for kt in (1, 2, 4, 8)} | {(16, kt, 1) for kt in (1, 2, 4)} | {(16, kt, 2) for kt in (1, 2, 4)}
    assert got == want


@pytest.mark.parametrize("H", [4, 36, 64, 100, 128, 200, 256, 300, 384, 512])
@pytest.mark.parametrize("K", [1, 7, 16, 33, 64, 100, 128, 200, 256])
def test_automatic_choice_of_the_persistent_kernel(H, K):
    """The one-exchange kernel where it fits and H x its terms per CTA is at
    most 16384, else the per-unit-block kernel."""
    auto = plan(FP32, H, 4, 1, K)
    assert auto["path"] == PATH_PERSISTENT
    try:
        ag = plan(FP32, H, 4, 1, K, (), PATH_PERSISTENT, 0, 2)
    except LSTMApproxError:
        ag = None
    if ag is not None and H * ag["terms_per_cta"] <= 16384:
        assert auto == ag
    else:
        assert auto == plan(FP32, H, 4, 1, K, (), PATH_PERSISTENT, 0, 1)


@pytest.mark.parametrize("H", [4, 52, 64, 100, 256, 300, 512, 516, 772, 1024])
@pytest.mark.parametrize("K", [1, 9, 32, 65, 128, 200, 256])
@pytest.mark.parametrize("cs", [0, 1, 2, 4, 8, 16])
@pytest.mark.parametrize("variant", [1, 2])
def test_every_plan_covers_its_shape_and_fits(H, K, cs, variant):
    cps = [max(1, K // 2)] if K > 2 else []
    try:
        p = plan(FP32, H, 2, 1, K, cps, PATH_PERSISTENT, cs, variant)
    except LSTMApproxError:
        return  # the shape is rejected (the run rejects it too)
    CS = p["cluster"]
    assert CS in (1, 2, 4, 8, 16) and (cs == 0 or CS == cs)
    assert 116 * 1024 <= p["smem_bytes"] <= 227 * 1024  # alone on its SM
    assert p["tmem_columns"] in (0, 32, 64, 128, 256, 512)
    if variant == 1:
        assert H <= 1024 and K <= 256
        assert p["terms_per_cta"] % 4 == 0 and CS * p["terms_per_cta"] >= 4 * K  # all rows owned
        assert 4 * p["units_per_warp"] * CS >= H                                # all units owned
        assert 32 * p["terms_per_lane"] >= K and p["units_per_warp"] * p["terms_per_lane"] <= 64
    else:
        assert H <= 512 and CS in (4, 8, 16)
        assert p["terms_per_cta"] <= 64 and (CS // 4) * p["terms_per_cta"] >= K  # each gate's terms owned
        assert p["h_quads"] == (1 if H <= 128 else 2 if H <= 256 else 4)


@pytest.mark.parametrize("H,B", [(128, 1), (512, 16), (512, 256), (1024, 1024), (1280, 1000), (2048, 64),
                                 (2048, 2048), (136, 130)])
@pytest.mark.parametrize("K", [8, 64, 256, 1024])
def test_tensor_tiles(H, B, K):
    """Stream tiles: the narrowest of 32/64/128 (gates) that keeps the grid
    within one wave of 148 CTAs, else the widest; tau' takes 32 streams up to
    K = 32 (one tile of all four gates' rows), else the narrowest of 32/64
    that keeps one wave, else 128, except where few tiles of 64 streams
    over H >= 1024 split its reduction axis over clusters of 4 CTAs; the gate GEMM's
    terms split over min(148 // tiles, 8, chunks of 64) CTAs."""
    p = plan(BF16, H, 2, B, K)
    if K <= 32 and H in (256, 512, 1024):  # one launch for all timesteps (test_tensor_seq_plan)
        assert p["tensor_seq"] == 1
        return
    assert p["tensor_seq"] == 0
    units = -(-H // 128)
    nt = next((n for n in (32, 64, 128) if units * -(-B // n) <= 148), 128)
    assert p["gate_tile_streams"] == nt
    rows = 4 * -(-K // 128)
    bn = 32 if K <= 32 else next((n for n in (32, 64) if rows * -(-B // n) <= 148), 128)
    # few tiles of 64 streams over H >= 1024: the reduction axis over clusters of 4
    tiles64, hchunks = rows * -(-B // 64), -(-H // 64)
    sk = 1 if K <= 32 else 4 if tiles64 * 4 <= 148 and hchunks >= 16 else 1
    if sk > 1:
        bn, per = 64, -(-hchunks // sk)
        sk = -(-hchunks // per)
    assert (p["tau_tile_streams"], p["tau_splits"]) == (bn, sk)
    tiles = units * -(-B // nt)
    chunks = -(-K // 64)
    ks = min(148 // tiles, 8, chunks)
    if ks < 2:
        assert p["gate_splits"] == 1
    else:
        per = -(-chunks // ks)
        assert p["gate_splits"] == -(-chunks // per)  # no empty split


@pytest.mark.parametrize("H,B", [(256, 1), (256, 3000), (512, 256), (512, 700), (512, 1300), (1024, 1024), (1024, 5),
                                 (1024, 600)])
@pytest.mark.parametrize("K", [1, 8, 16, 17, 32])
def test_tensor_seq_plan(H, B, K):
    """One launch per tile of streams for all timesteps: the narrowest tiles
    (16, then 32 streams) whose clusters fit in one wave (36 clusters of 4
    CTAs, 72 of 2), else 64 streams.  H = 256: clusters of 2 CTAs of 128
    units; H = 512: 4 of 128; H = 1024: 4 of 256 with 16 or 32 streams, or 8
    of 128 with 64.  Each CTA owns 4, 8 or 16 streams of a tile."""
    p = plan(BF16, H, 2, B, K)
    t16, t32 = -(-B // 16), -(-B // 32)
    if H == 256:
        cs, ns = 2, (16 if t16 <= 72 else 32)
    elif H == 512:
        cs, ns = 4, (16 if t16 <= 36 else 32 if t32 <= 36 else 64)
    else:
        cs, ns = (4, 16) if t16 <= 36 else (4, 32) if t32 <= 36 else (8, 64)
    assert (p["tensor_seq"], p["cluster"], p["tau_tile_streams"], p["gate_tile_streams"], p["gate_splits"]) == \
        (1, cs, ns, ns, 1)
    assert ns // cs in (4, 8, 16)


@pytest.mark.parametrize("H,K,ck,seq", [
    (512, 32, [16], 1), (512, 32, [16, 32], 1), (512, 20, [16, 20], 1),  # depths on the slices, or = K
    (512, 32, [10], 0), (512, 32, [8, 16], 0),                            # a depth off the 16-term slices
    (512, 33, [], 0), (2048, 16, [], 0), (384, 16, [], 0), (128, 16, [], 0), (96, 8, [], 0),
])
def test_tensor_seq_rejections(H, K, ck, seq):
    """Shapes outside the one-launch kernel take two launches per timestep."""
    assert plan(BF16, H, 2, 64, K, ck)["tensor_seq"] == seq


def test_paths():
    assert plan(BF16, 64, 2, 4, 32, [16])["path"] == PATH_TENSOR
    assert plan(BF16, 64, 2, 4, 32, [10])["path"] == PATH_TENSOR     # a depth off the 16-term slices
    assert plan(BF16, 64, 2, 4, 32, [10], PATH_SIMT)["path"] == PATH_SIMT
    assert plan(FP32, 2048, 2, 1, 32)["path"] == PATH_SIMT           # no persistent kernel for H > 1024
    assert plan(FP32, 64, 2, 1, 300)["path"] == PATH_SIMT            # nor for K > 256
    assert plan(FP32, 64, 2, 4096, 32)["path"] == PATH_PERSISTENT    # at any batch
    simt = plan(FP32, 64, 2, 1, 32, (), PATH_SIMT)
    assert simt["path"] == PATH_SIMT and all(v == 0 for k, v in simt.items() if k != "path")


@pytest.mark.parametrize("args,text", [
    ((BF16, 64, 2, 1, 32, (), PATH_PERSISTENT), "fp32 factors only"),
    ((FP32, 64, 2, 1, 32, (), PATH_TENSOR), "bf16"),
    ((FP32, 64, 2, 1, 300, (), PATH_PERSISTENT), "persistent path unavailable"),
    ((FP32, 600, 2, 1, 32, (), PATH_PERSISTENT, 0, 2), "persistent path unavailable"),
    ((FP32, 64, 2, 1, 32, (), 0, 3), "cluster"),
    ((FP32, 64, 2, 1, 32, (), 0, 0, 3), "variant"),
    ((FP32, 64, 2, 1, 32, (), 4), "path"),
    ((FP32, 64, 2, 1, 32, [5, 5]), "increasing"),
    ((FP32, 64, 2, 1, 32, [33]), "outside"),
    ((FP32, 64, 0, 1, 32), ">= 1"),
    ((2, 64, 2, 1, 32), "dtype"),
])
def test_rejections(args, text):
    with pytest.raises(LSTMApproxError) as e:
        plan(*args)
    assert e.value.code == 1 and text in str(e.value)
