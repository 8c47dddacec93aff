"""The quality-of-result analysis of the oracle (approximation vs dense LSTM).

Pins: the dense reference agrees with torch.nn.LSTM built from the same W,
and at full rank without pruning the refinement reproduces the dense LSTM,
so both metrics vanish there; pruning or truncating raises them.
"""
import numpy as np
import pytest

from oracle import qor
from workloads import draw_factor_set, draw_inputs, draw_weight


def _weights(H, C, seed):
    return [draw_weight(H, C, seed + g) for g in range(4)]


def test_dense_reference_matches_torch_lstm():
    torch = pytest.importorskip("torch")
    D, H, T = 5, 4, 6
    W = _weights(H, D + H, 300)
    x = draw_inputs(T, 2, D, "uniform", 3)
    lstm = torch.nn.LSTM(D, H, bias=False).double()
    with torch.no_grad():
        lstm.weight_ih_l0.copy_(torch.from_numpy(np.concatenate([w[:, :D] for w in W])))
        lstm.weight_hh_l0.copy_(torch.from_numpy(np.concatenate([w[:, D:] for w in W])))
        ref, _ = lstm(torch.from_numpy(x))
    np.testing.assert_allclose(qor.dense_lstm(W, x), ref.numpy(), rtol=1e-12, atol=1e-13)


def test_dense_reference_with_bias_and_initial_state_matches_torch_lstm():
    torch = pytest.importorskip("torch")
    D, H, T, B = 5, 4, 6, 3
    W = _weights(H, D + H, 310)
    rng = np.random.default_rng(7)
    bias = rng.standard_normal((4, H))
    h0, c0 = rng.standard_normal((B, H)), rng.standard_normal((B, H))
    x = draw_inputs(T, B, D, "uniform", 5)
    lstm = torch.nn.LSTM(D, H).double()
    with torch.no_grad():
        lstm.weight_ih_l0.copy_(torch.from_numpy(np.concatenate([w[:, :D] for w in W])))
        lstm.weight_hh_l0.copy_(torch.from_numpy(np.concatenate([w[:, D:] for w in W])))
        lstm.bias_ih_l0.copy_(torch.from_numpy(bias.reshape(-1)))
        lstm.bias_hh_l0.zero_()
        ref, (hn, cn) = lstm(torch.from_numpy(x), (torch.from_numpy(h0)[None], torch.from_numpy(c0)[None]))
    got, c_last = qor.dense_lstm(W, x, bias=bias, h0=h0, c0=c0, return_c=True)
    np.testing.assert_allclose(got, ref.numpy(), rtol=1e-12, atol=1e-13)
    np.testing.assert_allclose(c_last, cn.numpy()[0], rtol=1e-12, atol=1e-13)


def test_full_rank_unpruned_has_zero_error_and_kl():
    D, H, T = 6, 4, 5
    C = D + H
    W = _weights(H, C, 400)
    x = draw_inputs(T, 1, D, "uniform", 4)
    rows = qor.qor_table(W, x, nzs=[C], Ks=[H])
    assert rows[0]["rel_h_error"] < 1e-12
    assert abs(rows[0]["head_kl"]) < 1e-12
    assert rows[0]["rel_w_error"] < 1e-12


def test_truncation_and_pruning_raise_the_error():
    D, H, T = 12, 8, 6
    C = D + H
    W = _weights(H, C, 500)
    x = draw_inputs(T, 1, D, "uniform", 5)
    rows = {(r["NZ"], r["K"]): r for r in qor.qor_table(W, x, nzs=[C, 4], Ks=[1, H])}
    assert rows[(C, 1)]["rel_h_error"] > 1e-3          # rank 1 of rank 8
    assert rows[(4, H)]["rel_h_error"] > 1e-3          # 4 of 20 columns kept
    assert rows[(C, H)]["rel_h_error"] < 1e-12
    for r in rows.values():
        assert r["head_kl"] >= -1e-15
        assert r["ops"] == 4 * r["K"] * (2 * H + 2 * r["NZ"] + 1)


def test_schemes_coincide_without_pruning():
    """Deflating W by exact singular triplets leaves the remaining ones, so
    without pruning the residual refinement and the truncated SVD are the
    same approximation at every K (Eckart-Young)."""
    D, H, T = 10, 6, 4
    C = D + H
    W = _weights(H, C, 600)
    x = draw_inputs(T, 1, D, "uniform", 6)
    res = qor.qor_table(W, x, nzs=[C], Ks=[1, 2, 4, 6])
    trunc = qor.qor_table(W, x, nzs=[C], Ks=[1, 2, 4, 6], scheme="truncated")
    for a, b in zip(res, trunc):
        for key in ("rel_h_error", "head_kl", "rel_w_error"):
            assert abs(a[key] - b[key]) < 1e-9, (a["K"], key, a[key], b[key])


def test_residual_matrix_error_never_increases():
    """||W - W~^(n+1)||^2 = ||W - W~^(n)||^2 - sigma_n^2 ||prune(v_n)||^2:
    with any pruning the residual scheme's error falls or stays with K, and
    the law holds term by term."""
    D, H, T = 12, 8, 3
    C = D + H
    W = _weights(H, C, 700)
    x = draw_inputs(T, 1, D, "uniform", 7)
    for nz in (3, 9):
        rows = qor.qor_table(W, x, nzs=[nz], Ks=list(range(1, 13)))
        errs = [r["rel_w_error"] for r in rows]
        assert all(b <= a + 1e-12 for a, b in zip(errs, errs[1:])), errs
    from oracle import decompose_gate
    f = decompose_gate(W[0], 6, 5)
    prev = float(np.sum(W[0] ** 2))
    for K in range(1, 7):
        cur = float(np.sum((W[0] - qor.reconstruct(f, K, C)) ** 2))
        drop = f["sigma"][K - 1] ** 2 * float(np.sum(f["val"][K - 1] ** 2))
        assert abs(prev - cur - drop) < 1e-10 * max(1.0, prev)
        prev = cur


def test_design_selection_by_definition():
    """A hand-checked set: (ops, error) pairs where b and d are beaten by a
    and c respectively, e ties a on error at a higher cost, and f is the
    most accurate."""
    rows = [{"name": n, "ops": o, "rel_h_error": e} for n, o, e in
            [("a", 10, 0.5), ("b", 12, 0.6), ("c", 20, 0.3), ("d", 20, 0.4), ("e", 15, 0.5), ("f", 40, 0.1)]]
    assert [r["name"] for r in qor.pareto(rows)] == ["a", "c", "f"]
    assert qor.best_within(rows, 9) is None
    assert qor.best_within(rows, 15)["name"] == "a"   # e has the same error at a higher cost
    assert qor.best_within(rows, 39)["name"] == "c"
    assert qor.best_within(rows, 40)["name"] == "f"


def test_every_front_design_is_the_best_at_its_own_cost():
    D, H, T = 12, 8, 3
    C = D + H
    W = _weights(H, C, 800)
    x = draw_inputs(T, 1, D, "uniform", 8)
    rows = qor.qor_table(W, x, nzs=[C, 10, 4], Ks=[1, 2, 4, 8])
    front = qor.pareto(rows)
    assert front and all(r in rows for r in front)
    for r in front:
        assert qor.best_within(rows, r["ops"]) is r
    errs = [r["rel_h_error"] for r in front]
    assert all(b < a for a, b in zip(errs, errs[1:]))   # more cost buys strictly less error along the front
