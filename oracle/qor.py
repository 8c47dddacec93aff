"""Quality of result of the approximation against the dense LSTM (oracle side).

TEST AND ANALYSIS INFRASTRUCTURE ONLY, like the rest of this package.

The paper measures the quality of an approximation as the KL divergence of
the driving model's output distribution from the dense model's (Sec. VI),
which needs the trained model and its data.  This module measures the same
kind of curve on the seeded synthetic workloads: the LSTM is run once with
its dense gate matrices W (Sec. II) and once with the K-term refinement of
Eq. 1 at each pruning level, and for every (NZ, K) it reports

* the relative error of the hidden states, ||h~ - h|| / ||h|| over all t;
* the KL divergence KL(p || p~) of softmax(A h_t), averaged over t, for a
  seeded random linear head A (classes x H, N(0, 1/sqrt(H))) standing in
  for the model's output layer;
* the operations per timestep of Sec. III, 4 gates x K (2R + 2NZ + 1),
  against the dense 4 x 2RC;
* the relative Frobenius error of the gate matrices themselves,
  ||W - W~^(K)|| / ||W|| over the four gates.

Two schemes are compared: the residual refinement of Eq. 1, where each
term is the top triplet of what the pruned terms before it left over, and
the non-residual scheme Sec. III contrasts it with, where the terms are the
first K singular triplets of W itself, each pruned afterwards.  Without
pruning the two coincide (deflation by exact triplets leaves the remaining
ones).

``python -m oracle.qor`` prints the tables for the small workload and the
paper's case-study shape.
"""
from __future__ import annotations

import sys
from typing import Dict, List, Sequence

import numpy as np

from .factors import decompose_gate, decompose_gate_variant
from .recurrence import lstm_cell, op_count, run_lstm


def dense_lstm(weights: Sequence[np.ndarray], x: np.ndarray, bias=None, h0=None, c0=None,
               return_c: bool = False):
    """h_t of the dense LSTM of Sec. II: y_g = W_g [x_t; h_{t-1}] (+ b_g).

    bias: None or [4][H]; h0, c0: None (zeros) or [B][H].  Returns h [T][B][H],
    and the final c [B][H] as well when return_c."""
    T, B, _ = x.shape
    H = weights[0].shape[0]
    h = np.zeros((B, H)) if h0 is None else np.asarray(h0, dtype=np.float64)
    c = np.zeros((B, H)) if c0 is None else np.asarray(c0, dtype=np.float64)
    out = np.zeros((T, B, H))
    for t in range(T):
        xt = np.concatenate([x[t], h], axis=1)          # [B][C]
        y = [xt @ W.T for W in weights]                 # four [B][H]
        h, c = lstm_cell(y, c, bias)
        out[t] = h
    return (out, c) if return_c else out


def softmax(z: np.ndarray) -> np.ndarray:
    z = z - z.max(axis=-1, keepdims=True)
    e = np.exp(z)
    return e / e.sum(axis=-1, keepdims=True)


def head_matrix(H: int, classes: int = 10, seed: int = 1905) -> np.ndarray:
    """The seeded random linear head A (classes x H, entries N(0, 1/sqrt(H)))
    that stands in for the driving model's output layer."""
    return np.random.Generator(np.random.PCG64(seed)).normal(0.0, 1.0 / np.sqrt(H), (classes, H))


def curve_point(h: np.ndarray, h_ref: np.ndarray, A: np.ndarray) -> Dict:
    """Quality of approximate hidden states h against the dense ones h_ref
    (same shape, last axis H): the relative error ||h - h_ref|| / ||h_ref||
    over all entries, and KL(p_ref || p) of the head's softmax averaged over
    every output vector."""
    p_ref = softmax(h_ref @ A.T)
    p = softmax(h @ A.T)
    kl = float(np.mean(np.sum(p_ref * (np.log(p_ref) - np.log(p)), axis=-1)))
    return {"rel_h_error": float(np.linalg.norm(h - h_ref) / np.linalg.norm(h_ref)), "head_kl": kl}


def reconstruct(f: dict, K: int, C: int) -> np.ndarray:
    """W~^(K) = sum_{n<K} sigma_n u_n prune(v_n)^T of one gate's factors."""
    V = np.zeros((K, C))
    for n in range(K):
        V[n, f["idx"][n]] = f["val"][n]
    return (f["u"][:K].T * f["sigma"][:K]) @ V


def qor_table(weights: Sequence[np.ndarray], x: np.ndarray, nzs: Sequence[int], Ks: Sequence[int],
              classes: int = 10, seed: int = 1905, scheme: str = "residual") -> List[Dict]:
    """One row per (NZ, K): relative h error, head KL, ops per timestep,
    relative gate-matrix error.  scheme: "residual" (Eq. 1) or "truncated"
    (the first K triplets of W, each pruned)."""
    if scheme not in ("residual", "truncated"):
        raise ValueError(scheme)
    H, C = weights[0].shape
    h_ref = dense_lstm(weights, x)
    A = head_matrix(H, classes, seed)
    w_norm = np.sqrt(sum(float(np.sum(W * W)) for W in weights))
    rows = []
    for nz in nzs:
        if scheme == "residual":
            layer = [decompose_gate(W, max(Ks), nz) for W in weights]
        else:
            layer = [decompose_gate_variant(W, max(Ks), nz, residual=False) for W in weights]
        for K in Ks:
            h = run_lstm([layer], x, K)["h"]
            pt = curve_point(h, h_ref, A)
            w_err = np.sqrt(sum(float(np.sum((W - reconstruct(f, K, C)) ** 2)) for W, f in zip(weights, layer)))
            rows.append({"NZ": nz, "K": K, "scheme": scheme,
                         "rel_h_error": pt["rel_h_error"],
                         "head_kl": pt["head_kl"],
                         "rel_w_error": w_err / w_norm,
                         "ops": 4 * op_count(H, nz, K), "dense_ops": 4 * 2 * H * C})
    return rows


def pareto(rows: List[Dict], cost: str = "ops", err: str = "rel_h_error") -> List[Dict]:
    """The candidate designs (NZ, K) of Sec. III that no other candidate
    beats: a row stays unless another has cost <= and error <= with one of
    them strictly lower.  Sorted by cost."""
    keep = []
    for r in rows:
        dominated = any(o[cost] <= r[cost] and o[err] <= r[err] and (o[cost] < r[cost] or o[err] < r[err])
                        for o in rows)
        if not dominated:
            keep.append(r)
    return sorted(keep, key=lambda r: (r[cost], r[err]))


def best_within(rows: List[Dict], budget: float, cost: str = "ops", err: str = "rel_h_error"):
    """The candidate with the lowest error among those whose cost fits the
    budget (the cheaper one on a tie), or None if none fits."""
    fit = [r for r in rows if r[cost] <= budget]
    return min(fit, key=lambda r: (r[err], r[cost])) if fit else None


def markdown(rows: List[Dict]) -> str:
    lines = ["| NZ | K | rel. h error | head KL | rel. W error | ops / step | fraction of dense ops |",
             "|---|---|---|---|---|---|---|"]
    for r in rows:
        lines.append(f"| {r['NZ']} | {r['K']} | {r['rel_h_error']:.3g} | {r['head_kl']:.3g} | "
                     f"{r['rel_w_error']:.3g} | {r['ops']} | {r['ops'] / r['dense_ops']:.3g} |")
    return "\n".join(lines)


def markdown_schemes(res: List[Dict], trunc: List[Dict]) -> str:
    """The two schemes side by side, row for row."""
    lines = ["| NZ | K | rel. W error, residual | rel. W error, truncated | rel. h error, residual | "
             "rel. h error, truncated |", "|---|---|---|---|---|---|"]
    for a, b in zip(res, trunc):
        lines.append(f"| {a['NZ']} | {a['K']} | {a['rel_w_error']:.3g} | {b['rel_w_error']:.3g} | "
                     f"{a['rel_h_error']:.3g} | {b['rel_h_error']:.3g} |")
    return "\n".join(lines)


def main(argv: Sequence[str]) -> None:
    from workloads import WORKLOADS, draw_inputs, draw_weights, nz_from_keep
    for name, T in (("c1", 8), ("f1", 4)):
        w = WORKLOADS[name]
        weights = draw_weights(w, 0)
        x = draw_inputs(T, 1, w.D, w.x_dist, 4242)
        nzs = [nz_from_keep(k, w.C()) for k in w.keeps] if name == "f1" else [w.C(), nz_from_keep(0.5, w.C()),
                                                                              nz_from_keep(0.125, w.C())]
        print(f"## {w.name} (H={w.H}, C={w.C()}, T={T})\n")
        res = qor_table(weights, x, nzs, w.Ks)
        print(markdown(res))
        print()
        pruned = [nz for nz in nzs if nz < w.C()]
        res_p = [r for r in res if r["NZ"] in pruned]
        print(f"### residual refinement against truncated SVD then pruning ({w.name})\n")
        print(markdown_schemes(res_p, qor_table(weights, x, pruned, w.Ks, scheme="truncated")))
        print()
        print(f"### candidate designs (NZ, K) no other beats on ops and h error ({w.name})\n")
        print(markdown(pareto(res)))
        print()


if __name__ == "__main__":
    main(sys.argv[1:])
