"""Helpers shared by the GPU parity tests (test infrastructure)."""
from __future__ import annotations

import functools

import numpy as np

import oracle
from workloads import (WORKLOADS, draw_weights, nz_from_keep, rounded_factors, synthetic_layer_factors,
                       workload_inputs)

FP32_TOL = 1e-4   # max relative error, fp32 factors
BF16_TOL = 2e-2   # max relative error, bf16 factors / fp32 accumulate


def max_rel_err_vec(got, ref) -> float:
    """Normwise relative error of every output vector (last axis: the H units):
    max over vectors of max_j |got_j - ref_j| / max_j |ref_j|.  Reported
    beside the elementwise error; no bound is asserted on it."""
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert got.shape == ref.shape, (got.shape, ref.shape)
    if ref.size == 0:
        return 0.0
    num = np.abs(got - ref).max(axis=-1)
    den = np.maximum(np.abs(ref).max(axis=-1), 1e-30)
    return float((num / den).max())


def max_rel_err(got, ref) -> float:
    """max_i |got_i - ref_i| / max(|ref_i|, 1e-2 * max_j |ref_j|)."""
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert got.shape == ref.shape, (got.shape, ref.shape)
    if ref.size == 0:
        return 0.0
    floor = 1e-2 * max(np.abs(ref).max(), 1e-30)
    return float((np.abs(got - ref) / np.maximum(np.abs(ref), floor)).max())


@functools.lru_cache(maxsize=None)
def decomposed_layer(wname: str, layer: int, K: int, keep: float):
    """Oracle residual decomposition of the workload's seeded gate matrices."""
    w = WORKLOADS[wname]
    nz = nz_from_keep(keep, w.C(layer))
    return tuple(oracle.decompose_layer(draw_weights(w, layer), K, nz))


@functools.lru_cache(maxsize=None)
def synthetic_layer(wname: str, layer: int, K: int, keep: float):
    return tuple(synthetic_layer_factors(WORKLOADS[wname], layer, K, keep))


def run_gpu(layers, x, K, dtype="fp32", h0=None, c0=None, checkpoints=(), force_path=0, cluster=0,
            max_rank=None, max_batch=None, want_c=True, variant=0, xproj=0, tau_layout=0, tensor_seq=0):
    """Set factors, run through the C-ABI, return numpy outputs and the handle."""
    import torch
    from paper_1905_00689_gb300 import (LSTMApprox, OPT_CLUSTER, OPT_FORCE_PATH, OPT_PERSISTENT_VARIANT,
                                        OPT_TAU_LAYOUT, OPT_TENSOR_SEQ, OPT_XPROJ)
    dev = torch.device("cuda:0")
    T, B, D = x.shape
    L = len(layers)
    H = layers[0][0]["u"].shape[1]
    mr = max_rank or max(len(g["sigma"]) for lay in layers for g in lay)
    m = LSTMApprox(L, [D] + [H] * (L - 1), H, mr, max_batch or B, dtype)
    for l, gates in enumerate(layers):
        m.set_layer(l, gates)
    if force_path:
        m.set_option(OPT_FORCE_PATH, force_path)
    if cluster:
        m.set_option(OPT_CLUSTER, cluster)
    if variant:
        m.set_option(OPT_PERSISTENT_VARIANT, variant)
    if xproj:
        m.set_option(OPT_XPROJ, xproj)
    if tau_layout:
        m.set_option(OPT_TAU_LAYOUT, tau_layout)
    if tensor_seq:
        m.set_option(OPT_TENSOR_SEQ, tensor_seq)
    xt = torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32)).to(dev)
    out_h = torch.full((T, B, H), float("nan"), device=dev)
    out_c = torch.full((L, B, H), float("nan"), device=dev) if want_c else None
    J = len(checkpoints)
    ck_h = torch.full((J, T, B, H), float("nan"), device=dev) if J else None
    ck_c = torch.full((J, T, B, H), float("nan"), device=dev) if J else None
    th0 = None if h0 is None else torch.from_numpy(np.ascontiguousarray(h0, dtype=np.float32)).to(dev)
    tc0 = None if c0 is None else torch.from_numpy(np.ascontiguousarray(c0, dtype=np.float32)).to(dev)
    m.run(xt, K, out_h, h0=th0, c0=tc0, out_c=out_c, checkpoints=list(checkpoints), ckpt_h=ck_h, ckpt_c=ck_c)
    m.sync()
    res = {"h": out_h.double().cpu().numpy()}
    if want_c:
        res["c_last"] = out_c.double().cpu().numpy()
    if J:
        res["ckpt_h"] = ck_h.double().cpu().numpy()
        res["ckpt_c"] = ck_c.double().cpu().numpy()
    return res, m


def oracle_run(layers, x, K, dtype="fp32", **kw):
    """Oracle on the factors as the library stores them (rounded to dtype)."""
    rl = [rounded_factors(g, dtype) for g in layers]
    xr = np.asarray(x, dtype=np.float32).astype(np.float64)
    return oracle.run_lstm(rl, xr, K, **kw)


# (test id, bound, {output: (elementwise, normwise)}) of every parity check of
# the session, printed by the terminal-summary hook in conftest.py
REPORT = []
CURRENT_TEST = [""]
NOTES = []  # lines a test asks to print in the session summary (tables measured on the GPU)


def assert_parity(got, ref, tol, keys=("h", "c_last", "ckpt_h", "ckpt_c")):
    """Every output within `tol` under the elementwise metric (max_rel_err),
    for both factor types.  Returns {key: (elementwise, normwise)} errors;
    the normwise figure is a report only."""
    errs = {}
    for k in keys:
        if k in got and k in ref:
            assert np.all(np.isfinite(got[k])), f"{k}: non-finite output"
            errs[k] = (max_rel_err(got[k], ref[k]), max_rel_err_vec(got[k], ref[k]))
    REPORT.append((CURRENT_TEST[0], tol, errs))
    bad = {k: v for k, v in errs.items() if v[0] > tol}
    assert not bad, f"max relative error (elementwise, normwise) above {tol}: {errs}"
    return errs


__all__ = ["FP32_TOL", "BF16_TOL", "max_rel_err", "max_rel_err_vec", "decomposed_layer", "synthetic_layer", "run_gpu",
           "oracle_run", "assert_parity", "workload_inputs", "WORKLOADS", "persistent_layout_cases"]


# The per-unit-block kernel is compiled for each combination of units per
# warp (the smallest power of two with 4 * UW >= the CTA's units, about
# H / CS), terms per lane (the smallest power of two with 32 * KT >= K) and
# where V_h lives (shared memory up to H = 256, tensor memory with U up to
# 512, tensor memory with 32 h values per lane up to 1024).
# persistent_layout_cases() gives one (H, K, cluster size) for each compiled
# combination, with ragged hidden sizes.
UB_LAYOUTS = [  # (H, cluster size) for UW = 1, 2, 4, 8, 16 with V_h in shared memory
    (36, 16), (100, 16), (196, 16), (196, 8), (196, 4)]
LAYOUT_K = {1: 23, 2: 50, 4: 100, 8: 200}  # a K for each number of terms per lane


def persistent_layout_cases():
    cases = []
    for i, (H, cs) in enumerate(UB_LAYOUTS):
        for kt in (1, 2, 4, 8) if i < 4 else (1, 2, 4):
            cases.append((H, LAYOUT_K[kt], cs))
    for kt in (1, 2, 4, 8):
        cases.append((388, LAYOUT_K[kt], 16))  # UW = 8, V_h and U in tensor memory
    for kt in (1, 2, 4):
        cases.append((388, LAYOUT_K[kt], 8))   # UW = 16, V_h and U in tensor memory
        cases.append((772, LAYOUT_K[kt], 16))  # UW = 16, V_h in tensor memory, 32 values per lane
    return cases
