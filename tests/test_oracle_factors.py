"""Pins of the factor generator (Sec. III, Eq. 1) against mathematics and LAPACK.

Each test fixes a property that a plausible mistake would break:
* prune(): brute-force ranking and the tie rule (wrong key, wrong order);
* keep = 1 (no pruning): the residual scheme is Eckart-Young deflation, so
  sigma_n equal the singular values of W and K = R steps rebuild W exactly
  (a residual formed with the wrong sign or never updated fails);
* any keep: ||R^(n+1)||_F^2 = ||R^(n)||_F^2 - sigma_n^2 ||v'_n||^2 exactly,
  because u^T R = sigma v^T; pruning u, or subtracting the unpruned term,
  or a transposed residual, breaks the identity.
"""
import numpy as np
import pytest

import oracle
from oracle import factors as F
from workloads import draw_weight, nz_from_keep


def _brute_prune(v, nz):
    pairs = sorted(((-abs(float(x)), i) for i, x in enumerate(v)))
    kept = sorted(i for _, i in pairs[:nz])
    return kept


@pytest.mark.parametrize("C,nz", [(7, 1), (7, 3), (7, 7), (128, 64), (300, 31)])
def test_prune_matches_brute_force(C, nz):
    rng = np.random.default_rng(C * 131 + nz)
    for _ in range(5):
        v = rng.standard_normal(C)
        idx, val = F.prune(v, nz)
        assert list(idx) == _brute_prune(v, nz)
        assert np.array_equal(val, v[idx])
        assert idx.dtype == np.int32 and np.all(np.diff(idx) > 0)
        dropped = np.setdiff1d(np.arange(C), idx)
        if dropped.size:
            assert np.abs(v[idx]).min() >= np.abs(v[dropped]).max()


def test_prune_ties_prefer_lower_index():
    v = np.array([0.5, -2.0, 2.0, 0.5, -0.5, 1.0])
    # |v| ranking: 2.0 (idx 1), 2.0 (idx 2), 1.0 (idx 5), 0.5 (idx 0), 0.5 (3), 0.5 (4)
    assert list(F.prune(v, 2)[0]) == [1, 2]
    assert list(F.prune(v, 4)[0]) == [0, 1, 2, 5]
    assert list(F.prune(v, 5)[0]) == [0, 1, 2, 3, 5]


def test_prune_rejects_bad_nz():
    with pytest.raises(ValueError):
        F.prune(np.ones(4), 0)
    with pytest.raises(ValueError):
        F.prune(np.ones(4), 5)


def test_nz_from_keep_values():
    # NZ = max(1, floor(keep*C + 1/2)) for the five workloads' (keep, C)
    assert nz_from_keep(0.5, 128) == 64
    assert nz_from_keep(0.25, 1536) == 384
    assert nz_from_keep(0.5, 1536) == 768
    assert nz_from_keep(0.5, 3072) == 1536
    assert nz_from_keep(0.1, 3072) == 307
    assert nz_from_keep(0.3, 6144) == 1843
    assert nz_from_keep(0.3, 4096) == 1229
    assert nz_from_keep(1e-9, 100) == 1


def test_top_triplet_sign_and_norms():
    W = draw_weight(6, 11, 5)
    s, u, v = F.top_triplet(W)
    assert abs(np.linalg.norm(u) - 1) < 1e-12 and abs(np.linalg.norm(v) - 1) < 1e-12
    assert np.isclose(s, np.linalg.svd(W, compute_uv=False)[0], rtol=1e-13)
    assert v[np.argmax(np.abs(v))] > 0
    assert np.allclose(W.T @ u, s * v, atol=1e-12)   # u^T W = sigma v^T
    assert np.allclose(W @ v, s * u, atol=1e-12)


@pytest.mark.parametrize("H,C", [(8, 16), (64, 128)])
def test_unpruned_residual_scheme_is_svd_deflation(H, C):
    W = draw_weight(H, C, 17 + H)
    f = F.decompose_gate(W, H, C)                   # keep = 1, full rank
    s_ref = np.linalg.svd(W, compute_uv=False)
    assert np.allclose(f["sigma"], s_ref, rtol=1e-10, atol=1e-12)
    assert np.abs(F.reconstruct(f, H, C) - W).max() < 1e-12
    # each rank-1 term is the LAPACK SVD term of the same index (up to sign)
    U, _, Vt = np.linalg.svd(W, full_matrices=False)
    for n in range(0, H, max(1, H // 8)):
        v_full = np.zeros(C)
        v_full[f["idx"][n]] = f["val"][n]
        assert np.allclose(np.outer(f["u"][n], v_full), np.outer(U[:, n], Vt[n]), atol=1e-8)


@pytest.mark.parametrize("keep", [0.5, 0.25, 0.1, 0.02])
def test_frobenius_decrease_law(keep):
    H, C = 32, 96
    W = draw_weight(H, C, 23)
    nz = nz_from_keep(keep, C)
    K = 40
    f = F.decompose_gate(W, K, nz, return_residual_norms=True)
    fro2 = f["resid_fro2"]
    assert np.isclose(fro2[0], np.sum(W * W), rtol=1e-14)
    for n in range(K):
        vn2 = float(np.sum(f["val"][n] ** 2))
        pred = fro2[n] - f["sigma"][n] ** 2 * vn2
        assert abs(fro2[n + 1] - pred) <= 1e-10 * fro2[0]
        assert fro2[n + 1] <= fro2[n] + 1e-12 * fro2[0]
        assert np.count_nonzero(f["u"][n]) == H       # u is dense: not pruned
        assert len(f["idx"][n]) == nz


def test_masks_are_top_magnitudes_of_residual_triplet():
    H, C = 16, 40
    W = draw_weight(H, C, 31)
    nz = 9
    f = F.decompose_gate(W, 6, nz)
    # recompute step n's unpruned v from the residual and check the mask
    Wt = np.zeros_like(W)
    for n in range(6):
        _, _, v = F.top_triplet(W - Wt)
        assert list(f["idx"][n]) == _brute_prune(v, nz)
        Wt = F.reconstruct(f, n + 1, C)


def test_rank1_keep1_is_top_svd_term():
    W = draw_weight(12, 30, 3)
    f = F.decompose_gate(W, 1, 30)
    U, s, Vt = np.linalg.svd(W, full_matrices=False)
    assert np.allclose(F.reconstruct(f, 1, 30), s[0] * np.outer(U[:, 0], Vt[0]), atol=1e-13)


# ---- variants of the scheme (non-residual truncated SVD, pruned u) --------

def test_variant_default_is_the_residual_scheme():
    from oracle import decompose_gate_variant
    W = np.random.default_rng(11).standard_normal((6, 14))
    a = F.decompose_gate(W, 4, 5)
    b = decompose_gate_variant(W, 4, 5)
    for key in ("sigma", "u", "idx", "val"):
        np.testing.assert_array_equal(a[key], b[key])


def test_unpruned_residual_equals_truncated_svd():
    """Without pruning, the residual of a rank-n truncation has the (n+1)-th
    singular triplet of W as its top one (Eckart-Young), so both schemes
    give the same terms."""
    from oracle import decompose_gate_variant
    W = np.random.default_rng(12).standard_normal((5, 9))
    a = decompose_gate_variant(W, 5, 9, residual=True)
    b = decompose_gate_variant(W, 5, 9, residual=False)
    np.testing.assert_allclose(a["sigma"], b["sigma"], rtol=1e-12)
    np.testing.assert_allclose(np.abs(np.einsum("ki,ki->k", a["u"], b["u"])), 1.0, rtol=1e-10)
    np.testing.assert_allclose(a["val"], b["val"], rtol=1e-9, atol=1e-12)


def test_pruned_residual_beats_pruned_truncated_svd():
    """With pruning, the residual scheme re-fits what pruning dropped, so its
    approximation error after K terms is lower than pruning the truncated
    SVD's vectors -- on average and on most draws (it is greedy, so not on
    every one)."""
    from oracle import decompose_gate_variant
    ratios = []
    for seed in range(10):
        W = np.random.default_rng(100 + seed).standard_normal((8, 24))
        a = decompose_gate_variant(W, 6, 6, residual=True)
        b = decompose_gate_variant(W, 6, 6, residual=False)
        ratios.append(np.linalg.norm(W - F.reconstruct(a, 6, 24)) / np.linalg.norm(W - F.reconstruct(b, 6, 24)))
    ratios = np.array(ratios)
    assert ratios.mean() < 0.97 and np.count_nonzero(ratios < 1.0) >= 8, ratios


def test_pruned_u_keeps_the_largest_entries():
    from oracle import decompose_gate_variant, prune_dense
    W = np.random.default_rng(13).standard_normal((10, 12))
    f = decompose_gate_variant(W, 3, 12, nz_u=4)
    for n in range(3):
        assert np.count_nonzero(f["u"][n]) == 4
    np.testing.assert_array_equal(prune_dense(np.array([0.1, -3.0, 2.0, 2.0]), 2), [0.0, -3.0, 2.0, 0.0])


# ---- the Lanczos route for large gate matrices ----------------------------

def test_lanczos_top_triplet_equals_lapack():
    """ARPACK's largest singular triplet equals LAPACK's full SVD (two
    independent library routines) on a Gaussian matrix above the size limit
    and on a residual after three pruned refinement steps."""
    from oracle.factors import LANCZOS_ABOVE, top_triplet
    rng = np.random.default_rng(31)
    R = rng.standard_normal((LANCZOS_ABOVE + 8, 3 * LANCZOS_ABOVE)) / np.sqrt(3 * LANCZOS_ABOVE)
    f = oracle.decompose_gate(R, 3, 700, method="svd")
    residual = R - oracle.reconstruct(f, 3, R.shape[1])
    for M in (R, residual):
        a = top_triplet(M, "svd")
        b = top_triplet(M, "lanczos")
        assert abs(a[0] - b[0]) <= 1e-12 * a[0]
        assert np.abs(a[0] * np.outer(a[1], a[2]) - b[0] * np.outer(b[1], b[2])).max() <= 1e-12
        # same sign convention: v's largest-magnitude entry positive
        assert np.array_equal(np.sign(a[2]), np.sign(b[2]))
        assert abs(np.linalg.norm(b[1]) - 1) < 1e-14 and abs(np.linalg.norm(b[2]) - 1) < 1e-14
    assert top_triplet(R)[0] == top_triplet(R, "lanczos")[0]  # the automatic choice above the limit


def test_lanczos_decomposition_matches_lapack_and_keeps_the_frobenius_law():
    from oracle.factors import LANCZOS_ABOVE
    rng = np.random.default_rng(32)
    H, C, K, nz = LANCZOS_ABOVE + 4, 1100, 6, 300
    W = rng.standard_normal((H, C)) / np.sqrt(C)
    a = oracle.decompose_gate(W, K, nz, method="svd")
    b = oracle.decompose_gate(W, K, nz, return_residual_norms=True)  # automatic: Lanczos
    assert np.array_equal(a["idx"], b["idx"])
    np.testing.assert_allclose(b["sigma"], a["sigma"], rtol=1e-11)
    np.testing.assert_allclose(b["u"], a["u"], atol=1e-10)
    np.testing.assert_allclose(b["val"], a["val"], atol=1e-10)
    # ||R^(n+1)||^2 = ||R^(n)||^2 - sigma_n^2 ||v'_n||^2 (exact for any accurate triplet)
    f2 = b["resid_fro2"]
    drop = b["sigma"] ** 2 * np.sum(b["val"] ** 2, axis=1)
    np.testing.assert_allclose(f2[:-1] - f2[1:], drop, rtol=1e-9)
