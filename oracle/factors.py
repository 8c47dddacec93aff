"""Offline factor generation: hybrid SVD + pruning with residual refinement.

TEST INFRASTRUCTURE ONLY (see the package docstring).

Follows Sec. III of the paper:

* "Information-maximising approximation": the gate's two matrices are
  concatenated into W = [Wx Wh] (R x C) and approximated by the top singular
  triplet sigma_1 u_1 v_1^T.
* "Pruning by means of network sparsification": keep the NZ entries of
  largest absolute value.  Eq. 1 applies prune() to v only, so every row of
  sigma u prune(v)^T keeps the same NZ columns and no output element is
  zeroed.
* "Hybrid compression and pruning", Eq. 1 and the paragraph after it: step n
  takes the top singular triplet of the residual R^(n) = W - W~^(n-1), prunes
  its v, and adds sigma u prune(v)^T to the running approximation W~.

Readings where the paper is silent:
* ties in the magnitude ranking go to the lower column index; the kept index
  list is stored in ascending order;
* the triplet's sign is fixed so that v's largest-magnitude entry (lowest
  index among ties) is positive -- sigma u v^T and the mask do not depend on
  it;
* the top triplet is taken from LAPACK's full SVD (numpy.linalg.svd, fp64)
  when min(R, C) <= 512, and from ARPACK's implicitly restarted Lanczos
  iteration for the largest singular value (scipy.sparse.linalg.svds,
  k = 1, tolerance 1e-13) above that, where a full SVD per refinement step
  takes minutes; both give the same sigma u v^T up to the accuracy of the
  iteration (pinned against each other in the tests).
"""
from __future__ import annotations

from typing import List

import numpy as np


def prune(v: np.ndarray, nz: int):
    """prune(v, NZ) of Eq. 1: indices and values of the nz largest |v_c|.

    Ranking is by |v| descending, then by index ascending.  Returns
    (idx, val) with idx ascending (int32).
    """
    v = np.asarray(v, dtype=np.float64)
    C = v.shape[0]
    if not 1 <= nz <= C:
        raise ValueError(f"nz={nz} outside [1, {C}]")
    order = np.lexsort((np.arange(C), -np.abs(v)))  # last key is primary
    kept = np.sort(order[:nz])
    return kept.astype(np.int32), v[kept].copy()


LANCZOS_ABOVE = 512  # min(R, C) above which the top triplet comes from the Lanczos iteration


def top_triplet(R: np.ndarray, method: str = "auto"):
    """Top singular triplet (sigma, u, v) of R, with ||u|| = ||v|| = 1.

    method: "svd" (LAPACK, full SVD), "lanczos" (ARPACK, largest singular
    value only) or "auto" (Lanczos when min(R.shape) > LANCZOS_ABOVE)."""
    if method == "auto":
        method = "lanczos" if min(R.shape) > LANCZOS_ABOVE else "svd"
    if method == "svd":
        U, s, Vt = np.linalg.svd(R, full_matrices=False)
        sigma, u, v = float(s[0]), U[:, 0].copy(), Vt[0].copy()
    elif method == "lanczos":
        from scipy.sparse.linalg import svds
        # a fixed start vector keeps the result reproducible run to run
        v0 = np.ones(min(R.shape)) / np.sqrt(min(R.shape))
        U, s, Vt = svds(R, k=1, tol=1e-13, v0=v0, solver="arpack")
        sigma, u, v = float(s[0]), U[:, 0].copy(), Vt[0].copy()
        nu, nv = np.linalg.norm(u), np.linalg.norm(v)
        u, v = u / nu, v / nv
    else:
        raise ValueError(method)
    a = np.abs(v)
    lead = int(np.flatnonzero(a == a.max())[0])
    if v[lead] < 0:
        u, v = -u, -v
    return sigma, u, v


def decompose_gate(W: np.ndarray, K: int, nz: int, return_residual_norms: bool = False,
                   method: str = "auto") -> dict:
    """K residual refinement steps of Eq. 1 for one gate matrix W (R x C).

    Returns {"sigma": [K], "u": [K][R], "idx": [K][nz], "val": [K][nz]} and,
    if asked, "resid_fro2": ||R^(n)||_F^2 for n = 1..K+1.  method selects the
    top-triplet routine (see top_triplet).
    """
    W = np.asarray(W, dtype=np.float64)
    R_rows, C = W.shape
    sigma = np.empty(K)
    u = np.empty((K, R_rows))
    idx = np.empty((K, nz), dtype=np.int32)
    val = np.empty((K, nz))
    W_tilde = np.zeros_like(W)          # W~^(0) = 0
    fro2 = []
    for n in range(K):
        residual = W - W_tilde          # R^(n) = W - W~^(n-1)
        fro2.append(float(np.sum(residual * residual)))
        s_n, u_n, v_n = top_triplet(residual, method)
        i_n, p_n = prune(v_n, nz)       # prune(v^(n), NZ); u is not pruned
        v_pruned = np.zeros(C)
        v_pruned[i_n] = p_n
        W_tilde = W_tilde + s_n * np.outer(u_n, v_pruned)
        sigma[n], u[n], idx[n], val[n] = s_n, u_n, i_n, p_n
    out = {"sigma": sigma, "u": u, "idx": idx, "val": val}
    if return_residual_norms:
        residual = W - W_tilde
        fro2.append(float(np.sum(residual * residual)))
        out["resid_fro2"] = np.array(fro2)
    return out


def prune_dense(a: np.ndarray, n: int) -> np.ndarray:
    """a with all but its n largest-magnitude entries set to zero (same
    ranking as prune)."""
    i, p = prune(a, n)
    out = np.zeros_like(np.asarray(a, dtype=np.float64))
    out[i] = p
    return out


def decompose_gate_variant(W: np.ndarray, K: int, nz: int, residual: bool = True, nz_u: int = 0) -> dict:
    """Variants of the scheme around Eq. 1, in the same output format.

    residual=False: the non-residual scheme Sec. III contrasts with Eq. 1 --
    the first K singular triplets of W itself (truncated SVD), each v pruned
    to nz.  nz_u > 0 additionally keeps only the nz_u largest-magnitude
    entries of each u (stored dense, zeros elsewhere); in the residual scheme
    the pruned u enters the running approximation W~.  residual=True,
    nz_u=0 is decompose_gate.
    """
    W = np.asarray(W, dtype=np.float64)
    R_rows, C = W.shape
    sigma = np.empty(K)
    u = np.empty((K, R_rows))
    idx = np.empty((K, nz), dtype=np.int32)
    val = np.empty((K, nz))
    if not residual:
        U_all, s_all, Vt_all = np.linalg.svd(W, full_matrices=False)
        if K > s_all.shape[0]:
            raise ValueError(f"K={K} above the rank bound {s_all.shape[0]}")
    W_tilde = np.zeros_like(W)
    for n in range(K):
        if residual:
            s_n, u_n, v_n = top_triplet(W - W_tilde)
        else:  # n-th triplet of W, with the sign convention of top_triplet
            s_n, u_n, v_n = float(s_all[n]), U_all[:, n].copy(), Vt_all[n].copy()
            a = np.abs(v_n)
            if v_n[int(np.flatnonzero(a == a.max())[0])] < 0:
                u_n, v_n = -u_n, -v_n
        if nz_u > 0:
            u_n = prune_dense(u_n, nz_u)
        i_n, p_n = prune(v_n, nz)
        v_pruned = np.zeros(C)
        v_pruned[i_n] = p_n
        W_tilde = W_tilde + s_n * np.outer(u_n, v_pruned)
        sigma[n], u[n], idx[n], val[n] = s_n, u_n, i_n, p_n
    return {"sigma": sigma, "u": u, "idx": idx, "val": val}


def decompose_layer(weights, K: int, nz: int) -> List[dict]:
    """decompose_gate for the four gate matrices (i, f, g, o) of one layer."""
    return [decompose_gate(W, K, nz) for W in weights]


def reconstruct(f: dict, k: int, C: int) -> np.ndarray:
    """W~^(k) = sum_{n<=k} sigma^(n) u^(n) prune(v^(n))^T as a dense R x C matrix."""
    R_rows = f["u"].shape[1]
    Wt = np.zeros((R_rows, C))
    for n in range(k):
        v_pruned = np.zeros(C)
        v_pruned[f["idx"][n]] = f["val"][n]
        Wt += f["sigma"][n] * np.outer(f["u"][n], v_pruned)
    return Wt
