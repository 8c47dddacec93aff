"""Pins of the fp64 recurrence oracle (Sec. II, Sec. III Eq. 1, progressive outputs).

* Full rank, no pruning: the expansion equals W, so the oracle must equal a
  dense LSTM computed from W by a library routine (torch.nn.LSTM in fp64,
  gate order i, f, g, o, no bias).  Catches a wrong gate nonlinearity, a
  swapped [x; h] order, a transposed factor or a wrong cell update.
* Intermediate depths: the k-prefix sums equal the truncated reconstruction
  W~^(k) applied densely (torch.nn.LSTMCell with W~^(k), driven by the
  full-depth state).
* Tiny shapes: agreement with an independently written scalar implementation.
* Special cases: all-zero input keeps h = c = 0; with h0 = 0 and T = 1 only
  the x columns matter; op count N_steps(2R + 2NZ + 1) per gate.
"""
import numpy as np
import pytest
import torch

from oracle import factors as F
from oracle import recurrence as R
from workloads import draw_inputs, draw_weight, draw_factor_set

from scalar_lstm import scalar_run


def _torch_lstm(weights_per_layer, D, H, x, bias_per_layer=None):
    L = len(weights_per_layer)
    m = torch.nn.LSTM(D, H, num_layers=L, bias=bias_per_layer is not None).double()
    with torch.no_grad():
        for l, Ws in enumerate(weights_per_layer):
            Din = D if l == 0 else H
            getattr(m, f"weight_ih_l{l}").copy_(torch.from_numpy(np.vstack([W[:, :Din] for W in Ws])))
            getattr(m, f"weight_hh_l{l}").copy_(torch.from_numpy(np.vstack([W[:, Din:] for W in Ws])))
            if bias_per_layer is not None:
                getattr(m, f"bias_ih_l{l}").copy_(torch.from_numpy(np.concatenate(bias_per_layer[l])))
                getattr(m, f"bias_hh_l{l}").zero_()
        out, (hn, cn) = m(torch.from_numpy(x))
    return out.numpy(), hn.numpy(), cn.numpy()


@pytest.mark.parametrize("L,D,H,T,B", [(1, 5, 4, 6, 3), (2, 6, 5, 4, 2), (1, 64, 64, 8, 1)])
def test_full_rank_unpruned_equals_dense_lstm(L, D, H, T, B):
    weights = [[draw_weight(H, (D if l == 0 else H) + H, 1000 + 10 * l + g) for g in range(4)]
               for l in range(L)]
    layers = []
    for l, Ws in enumerate(weights):
        C = Ws[0].shape[1]
        layers.append(F.decompose_layer(Ws, H, C))   # K = R = H (full rank), NZ = C
    x = draw_inputs(T, B, D, "uniform", 77)
    ref_out, ref_h, ref_c = _torch_lstm(weights, D, H, x)
    got = R.run_lstm(layers, x, H)
    assert np.abs(got["h"] - ref_out).max() < 1e-11
    assert np.abs(got["h_last"] - ref_h).max() < 1e-11
    assert np.abs(got["c_last"] - ref_c).max() < 1e-11


def test_bias_enters_preactivation():
    D, H, T, B = 3, 4, 5, 2
    Ws = [draw_weight(H, D + H, 400 + g) for g in range(4)]
    gates = F.decompose_layer(Ws, H, D + H)
    rng = np.random.default_rng(5)
    biases = [rng.standard_normal(H) for _ in range(4)]
    for g, b in zip(gates, biases):
        g["bias"] = b
    x = draw_inputs(T, B, D, "uniform", 8)
    ref_out, _, ref_c = _torch_lstm([Ws], D, H, x, [biases])
    got = R.run_lstm([gates], x, H)
    assert np.abs(got["h"] - ref_out).max() < 1e-11
    assert np.abs(got["c_last"] - ref_c).max() < 1e-11


@pytest.mark.parametrize("keep_nz", [3, 7, 12])
def test_prefix_sums_equal_truncated_reconstruction(keep_nz):
    D, H, T, B = 4, 8, 5, 3
    C = D + H
    Ws = [draw_weight(H, C, 900 + g) for g in range(4)]
    K = 10
    gates = F.decompose_layer(Ws, K, keep_nz)
    x = draw_inputs(T, B, D, "relu", 12)
    cps = [1, 3, 7, 10]
    got = R.run_lstm([gates], x, K, checkpoints=cps)
    h_prev = np.zeros((B, H))
    c_prev = np.zeros((B, H))
    for t in range(T):
        for j, k in enumerate(cps):
            Wk = [F.reconstruct(g, k, C) for g in gates]
            cell = torch.nn.LSTMCell(D, H, bias=False).double()
            with torch.no_grad():
                cell.weight_ih.copy_(torch.from_numpy(np.vstack([W[:, :D] for W in Wk])))
                cell.weight_hh.copy_(torch.from_numpy(np.vstack([W[:, D:] for W in Wk])))
                hk, ck = cell(torch.from_numpy(x[t]), (torch.from_numpy(h_prev), torch.from_numpy(c_prev)))
            assert np.abs(got["ckpt_h"][j, t] - hk.numpy()).max() < 1e-12
            assert np.abs(got["ckpt_c"][j, t] - ck.numpy()).max() < 1e-12
        # the carried state is the full-depth one
        assert np.array_equal(got["ckpt_h"][-1, t], got["h"][t])
        h_prev = got["h"][t]
        # recover c_t from the last checkpoint (k = K is the full depth)
        c_prev = got["ckpt_c"][-1, t]


@pytest.mark.parametrize("L,D,H,T,B,K,nz", [(1, 1, 1, 3, 1, 2, 1), (1, 2, 3, 3, 2, 4, 3),
                                            (2, 3, 2, 2, 2, 3, 4), (1, 3, 2, 3, 1, 4, 5)])
def test_tiny_shapes_match_scalar_implementation(L, D, H, T, B, K, nz):
    layers = []
    for l in range(L):
        C = (D if l == 0 else H) + H
        layers.append([draw_factor_set(H, C, K, min(nz, C), 3000 + 10 * l + g) for g in range(4)])
    x = draw_inputs(T, B, D, "uniform", 41)
    cps = [k for k in (1, 2, K) if k <= K]
    cps = sorted(set(cps))
    got = R.run_lstm(layers, x, K, checkpoints=cps)
    ref, ref_ck = scalar_run(layers, x, K, checkpoints=cps)
    assert np.abs(got["h"] - np.array(ref)).max() < 1e-13
    assert np.abs(got["ckpt_h"] - np.array(ref_ck)).max() < 1e-13


def test_zero_input_stays_zero():
    D, H, T, B, K = 6, 5, 7, 2, 4
    gates = [draw_factor_set(H, D + H, K, 5, 50 + g) for g in range(4)]
    got = R.run_lstm([gates], np.zeros((T, B, D)), K, checkpoints=[2, 4])
    assert np.all(got["h"] == 0) and np.all(got["c_last"] == 0) and np.all(got["ckpt_h"] == 0)


def test_first_step_from_zero_state_ignores_h_columns():
    D, H, B, K = 5, 4, 3, 6
    gates = [draw_factor_set(H, D + H, K, 7, 70 + g) for g in range(4)]
    x = draw_inputs(1, B, D, "uniform", 9)
    a = R.run_lstm([gates], x, K)
    for g in gates:
        g["val"] = np.where(g["idx"] >= D, 123.0, g["val"])   # change only h-column weights
    b = R.run_lstm([gates], x, K)
    assert np.array_equal(a["h"], b["h"])


def test_op_count_per_gate():
    D, H, T, B, K, nz = 6, 5, 3, 2, 4, 7
    gates = [draw_factor_set(H, D + H, K, nz, 90 + g) for g in range(4)]
    counter = [0]
    R.run_lstm([gates], draw_inputs(T, B, D, "uniform", 1), K, counter=counter)
    # 4 gates x T x B x N_steps (2R + 2NZ + 1)
    assert counter[0] == 4 * T * B * K * (2 * H + 2 * nz + 1)
    assert R.op_count(H, nz, K) == K * (2 * H + 2 * nz + 1)


def test_truncated_run_reading_a_equals_checkpoint_at_first_step():
    """At t = 1 the two progressive readings coincide (same h0)."""
    D, H, B, K = 4, 6, 2, 9
    gates = [draw_factor_set(H, D + H, K, 6, 110 + g) for g in range(4)]
    x = draw_inputs(1, B, D, "uniform", 3)
    full = R.run_lstm([gates], x, K, checkpoints=[3, 9])
    trunc = R.run_lstm([gates], x, 3)
    assert np.array_equal(full["ckpt_h"][0, 0], trunc["h"][0])


def test_checkpoint_validation():
    gates = [draw_factor_set(2, 4, 3, 2, g) for g in range(4)]
    with pytest.raises(ValueError):
        R.run_lstm([gates], np.zeros((1, 1, 2)), 3, checkpoints=[2, 2])
    with pytest.raises(ValueError):
        R.run_lstm([gates], np.zeros((1, 1, 2)), 3, checkpoints=[4])
