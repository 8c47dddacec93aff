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


def test_full_rank_unpruned_has_zero_error_and_kl():
    D, H, T = 6, 4, 5
    C = D + H
    W = _weights(H, C, 400)
    x = draw_inputs(T, 1, D, "uniform", 4)
    rows = qor.qor_table(W, x, nzs=[C], Ks=[H])
    assert rows[0]["rel_h_error"] < 1e-12
    assert abs(rows[0]["head_kl"]) < 1e-12


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
