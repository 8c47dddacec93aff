"""Seeded synthetic workloads for the approximate-LSTM recurrence.

This module only draws random numbers with the shapes and distributions of
the workloads; it contains none of the method's arithmetic (no SVD, no
pruning, no recurrence).  It is the one module shared by the fp64 oracle,
the tests and the benchmark.

The five workloads stand in for the paper's case-study inputs (FCN features
of BDDV driving video feeding the driving model's LSTM, Sec. VI "Experimental
Setup"), which are not available: every weight and input is drawn from a
seeded PCG64 generator.

Seeds: weights of (workload w, layer l, gate g) use ``1905_00689 + 100*w +
10*l + g``; the input sequence of workload w uses that base + 7.  Gates are
ordered (i, f, g, o).
"""
from __future__ import annotations

import dataclasses
import math
from typing import List, Optional, Sequence, Tuple

import numpy as np

SEED_BASE = 190500689
GATES = ("i", "f", "g", "o")


@dataclasses.dataclass(frozen=True)
class Workload:
    """One LSTM workload: sizes, factor dtype, approximation levels."""

    index: int            # 1..6, used in the seeds
    name: str
    D: int                # input size of layer 0
    H: int                # hidden size (R in the paper)
    T: int                # timesteps
    B: int                # independent streams
    L: int                # stacked layers
    dtype: str            # "fp32" or "bf16" factor/operand type
    keeps: Tuple[float, ...]
    Ks: Tuple[int, ...]
    checkpoints: Tuple[int, ...]
    x_dist: str           # "uniform" = U(-1,1), "relu" = max(0, N(0,1))

    def C(self, layer: int = 0) -> int:
        """Augmented width C = D_l + H of layer `layer` (Sec. III)."""
        return (self.D if layer == 0 else self.H) + self.H

    def input_dim(self, layer: int) -> int:
        return self.D if layer == 0 else self.H


WORKLOADS = {
    "c1": Workload(1, "lstm-d64-h64-t8-b1-fp32", 64, 64, 8, 1, 1, "fp32",
                   (0.5,), (1, 4, 16, 64), (), "uniform"),
    "c2": Workload(2, "lstm-d1024-h512-t20-b1-fp32", 1024, 512, 20, 1, 1, "fp32",
                   (0.25,), (16, 64, 256), (), "relu"),
    "c3": Workload(3, "lstm-d1024-h512-t20-b256-bf16", 1024, 512, 20, 256, 1, "bf16",
                   (0.5,), (32, 128, 512), (), "relu"),
    "c4": Workload(4, "lstm-d2048-h1024-t64-b1024-bf16", 2048, 1024, 64, 1024, 1, "bf16",
                   (0.5, 0.1), (8, 32, 128, 512), (), "uniform"),
    "c5": Workload(5, "lstm2-d4096-h2048-t16-b64-bf16", 4096, 2048, 16, 64, 2, "bf16",
                   (0.3,), (1024,), (16, 64, 256, 1024), "uniform"),
    # the paper's case-study LSTM (Sec. VI): R = 64 hidden units, C = 8320
    # columns per gate, one timestep of one stream, fp32; NZ = 4160 (no
    # pruning of half the columns), 130 and 32 kept entries per v
    "f1": Workload(6, "lstm-d8256-h64-t1-b1-fp32", 8256, 64, 1, 1, 1, "fp32",
                   (0.5, 130 / 8320, 32 / 8320), (1, 4, 16, 64), (), "relu"),
}


def nz_from_keep(keep: float, C: int) -> int:
    """Number of kept entries per pruned vector: max(1, floor(keep*C + 1/2))."""
    return max(1, int(math.floor(keep * C + 0.5)))


def weight_seed(w: Workload, layer: int, gate: int) -> int:
    return SEED_BASE + 100 * w.index + 10 * layer + gate


def input_seed(w: Workload) -> int:
    return SEED_BASE + 100 * w.index + 7


def draw_weight(H: int, C: int, seed: int) -> np.ndarray:
    """Augmented gate matrix W = [Wx Wh] (H x C), entries N(0, std=1/sqrt(C))."""
    rng = np.random.Generator(np.random.PCG64(seed))
    return rng.standard_normal((H, C)) / math.sqrt(C)


def draw_weights(w: Workload, layer: int) -> List[np.ndarray]:
    """The four augmented gate matrices of one layer, gate order (i, f, g, o)."""
    C = w.C(layer)
    return [draw_weight(w.H, C, weight_seed(w, layer, g)) for g in range(4)]


def draw_inputs(T: int, B: int, D: int, dist: str, seed: int) -> np.ndarray:
    """Input sequence x[T][B][D] (float64)."""
    rng = np.random.Generator(np.random.PCG64(seed))
    if dist == "uniform":
        return rng.uniform(-1.0, 1.0, size=(T, B, D))
    if dist == "relu":
        return np.maximum(0.0, rng.standard_normal((T, B, D)))
    raise ValueError(f"unknown input distribution {dist!r}")


def workload_inputs(w: Workload, T: Optional[int] = None, B: Optional[int] = None) -> np.ndarray:
    """The workload's seeded input sequence, optionally cut to T steps / B streams."""
    x = draw_inputs(w.T, w.B, w.D, w.x_dist, input_seed(w))
    return x[: (T or w.T), : (B or w.B)]


def draw_factor_set(H: int, C: int, K: int, nz: int, seed: int) -> dict:
    """Random factor set with the structure of a pruned residual expansion.

    Used where the decomposition itself is too slow to run (large shapes) and
    for timing, whose cost does not depend on the factor values.  The draw
    mimics the statistics of the residual rank-1 expansion of a Gaussian W
    with std 1/sqrt(C): sigma_k decreasing inside the Marchenko-Pastur edge
    [1 - sqrt(H/C), 1 + sqrt(H/C)], u_k a Haar-random unit vector, and v'_k a
    random unit vector supported on `nz` distinct random columns.
    Returns sigma[K], u[K][H], idx[K][nz] (int32, ascending), val[K][nz].
    """
    rng = np.random.Generator(np.random.PCG64(seed))
    r = math.sqrt(H / C)
    sigma = np.sort(rng.uniform(max(1.0 - r, 0.05), 1.0 + r, size=K))[::-1].copy()
    u = rng.standard_normal((K, H))
    u /= np.linalg.norm(u, axis=1, keepdims=True)
    idx = np.empty((K, nz), dtype=np.int32)
    val = rng.standard_normal((K, nz))
    val /= np.linalg.norm(val, axis=1, keepdims=True)
    for k in range(K):
        idx[k] = np.sort(rng.choice(C, size=nz, replace=False))
    return {"sigma": sigma, "u": u, "idx": idx, "val": val}


def synthetic_layer_factors(w: Workload, layer: int, K: int, keep: float) -> List[dict]:
    """Per-gate random factor sets (see draw_factor_set) for one layer of `w`."""
    C = w.C(layer)
    nz = nz_from_keep(keep, C)
    return [draw_factor_set(w.H, C, K, nz, weight_seed(w, layer, g) + 50_000) for g in range(4)]


def bf16_bits(a: np.ndarray) -> np.ndarray:
    """bfloat16 bit patterns of `a` rounded through float32 (both steps
    round-to-nearest-even, ties to the even pattern).

    Written from the formats' definitions: bfloat16 is the upper half of an
    IEEE binary32, so rounding adds 0x7FFF plus the lowest kept bit and
    drops the low 16 bits; a carry out of the mantissa moves to the next
    binade (and past the largest finite value, to infinity).  Infinities
    keep their sign; every NaN becomes the quiet NaN 0x7FC0.
    """
    f = np.ascontiguousarray(np.asarray(a, dtype=np.float64).astype(np.float32))
    bits = f.view(np.uint32).astype(np.uint64)
    lsb = (bits >> 16) & 1
    rounded = (bits + 0x7FFF + lsb) >> 16
    nan = (bits & 0x7FFFFFFF) > 0x7F800000
    inf = (bits & 0x7FFFFFFF) == 0x7F800000
    out = np.where(inf, bits >> 16, rounded)
    out = np.where(nan, 0x7FC0, out)
    return out.astype(np.uint16)


def round_bf16(a: np.ndarray) -> np.ndarray:
    """Round to bfloat16 (through float32, both steps round-to-nearest-even).

    Returns float64 values that are exactly representable in bfloat16: the
    storage rounding of the bf16 factor path, so that the oracle can be fed
    the values the library stores.
    """
    bits = bf16_bits(a).astype(np.uint32) << 16
    return bits.view(np.float32).astype(np.float64)


def round_fp32(a: np.ndarray) -> np.ndarray:
    """Round to float32 (round-to-nearest-even), returned as float64."""
    return np.asarray(a, dtype=np.float64).astype(np.float32).astype(np.float64)


def rounded_factors(factors: Sequence[dict], dtype: str) -> List[dict]:
    """Factors as the library stores them: sigma in fp32; u and v in `dtype`."""
    rnd = round_bf16 if dtype == "bf16" else round_fp32
    out = []
    for f in factors:
        g = dict(f)
        g["sigma"] = round_fp32(f["sigma"])
        g["u"] = rnd(f["u"])
        g["val"] = rnd(f["val"])
        if f.get("bias") is not None:
            g["bias"] = round_fp32(f["bias"])
        out.append(g)
    return out
