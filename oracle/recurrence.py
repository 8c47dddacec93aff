"""fp64 recurrence of the approximate LSTM (progressive inference).

TEST INFRASTRUCTURE ONLY (see the package docstring).

Per timestep t and stream b (Sec. II, Fig. 2; Sec. III):

1. augmented input x~ = [x_t ; h_{t-1}] (Sec. III, "Information-maximising
   approximation");
2. for each gate, the refinement sum of Eq. 1:
   y = sum_{n=1..K} sigma^(n) u^(n) (prune(v^(n))^T x~), accumulated in n
   order, with a snapshot of the partial sum after each requested depth k_j
   (progressive inference, Sec. I / Fig. 1b: the best estimate available
   when the computation is cut short, Sec. VI);
3. the gate nonlinearities and the cell/output update of Sec. II: the input,
   forget and output gates use the logistic sigmoid, the cell gate tanh;
   c_t = f * c_{t-1} + i * g,  h_t = o * tanh(c_t).

Readings: gates are ordered (i, f, g, o); the
paper writes no bias, so the optional per-gate bias defaults to zero and is
exact (not approximated); the carried state h_t, c_t always uses the full
depth K, and the output at depth k_j applies step 3 to the k_j-prefix sums
with the carried c_{t-1}; in a stack, layer l+1 consumes layer l's full-depth
h_t and only the top layer's intermediate outputs are returned.
"""
from __future__ import annotations

from typing import Optional, Sequence

import numpy as np


def sigmoid(z: np.ndarray) -> np.ndarray:
    """Logistic function 1 / (1 + exp(-z)), evaluated without overflow."""
    z = np.asarray(z, dtype=np.float64)
    out = np.empty_like(z)
    pos = z >= 0
    out[pos] = 1.0 / (1.0 + np.exp(-z[pos]))
    ez = np.exp(z[~pos])
    out[~pos] = ez / (1.0 + ez)
    return out


def lstm_cell(y, c_prev, bias=None):
    """Gate nonlinearities and cell update of Sec. II.

    y: pre-activations [4][B][H] in gate order (i, f, g, o); c_prev [B][H];
    bias: None or [4][H].  Returns (h, c).
    """
    y = np.asarray(y, dtype=np.float64)
    if bias is not None:
        y = y + np.asarray(bias, dtype=np.float64)[:, None, :]
    i = sigmoid(y[0])
    f = sigmoid(y[1])
    g = np.tanh(y[2])
    o = sigmoid(y[3])
    c = f * c_prev + i * g
    h = o * np.tanh(c)
    return h, c


def refinement_sums(gate: dict, xt: np.ndarray, K: int, depths: Sequence[int] = (), counter=None):
    """Eq. 1 for one gate over a batch of augmented inputs.

    gate: {"sigma": [>=K], "u": [>=K][H], "idx": [>=K][nz], "val": [>=K][nz]};
    xt: x~ for every stream, [B][C].  Returns (y [B][H], {k_j: partial sum}).
    Each refinement step costs 2*NZ (dot product) + 1 (sigma times the dot
    product) + 2*R (scale u, accumulate) operations, as counted in Sec. III;
    `counter` (a one-element list) accumulates them per stream.
    """
    B = xt.shape[0]
    H = gate["u"].shape[1]
    y = np.zeros((B, H))
    snaps = {}
    want = set(depths)
    for n in range(K):
        idx, val = gate["idx"][n], gate["val"][n]
        tau = xt[:, idx] @ val                  # prune(v^(n))^T x~   (2 NZ ops)
        s = gate["sigma"][n] * tau              # sigma^(n) * (...)   (1 op)
        y = y + s[:, None] * gate["u"][n][None, :]   # u^(n) * s, accumulate (2 R ops)
        if counter is not None:
            counter[0] += B * (2 * len(idx) + 1 + 2 * H)
        if (n + 1) in want:
            snaps[n + 1] = y.copy()
    return y, snaps


def run_lstm(layers, x, K: int, h0=None, c0=None, checkpoints: Sequence[int] = (),
             counter=None):
    """Run the approximate LSTM stack over a sequence.

    layers: per layer, four gate factor dicts (i, f, g, o), each optionally
    with "bias" [H].  x: [T][B][D].  h0, c0: [L][B][H] or None (zeros).
    checkpoints: increasing depths 1 <= k_j <= K for the top layer.
    Returns {"h": [T][B][H] top layer at depth K, "h_last"/"c_last": [L][B][H],
    "ckpt_h"/"ckpt_c": [J][T][B][H]}.
    """
    x = np.asarray(x, dtype=np.float64)
    T, B, _ = x.shape
    L = len(layers)
    H = layers[0][0]["u"].shape[1]
    cps = list(checkpoints)
    if any(not 1 <= k <= K for k in cps) or any(a >= b for a, b in zip(cps, cps[1:])):
        raise ValueError("checkpoints must be strictly increasing within [1, K]")
    h_last = np.zeros((L, B, H)) if h0 is None else np.array(h0, dtype=np.float64)
    c_last = np.zeros((L, B, H)) if c0 is None else np.array(c0, dtype=np.float64)
    J = len(cps)
    ckpt_h = np.zeros((J, T, B, H))
    ckpt_c = np.zeros((J, T, B, H))
    layer_in = x
    for l, gates in enumerate(layers):
        bias = None
        if any(g.get("bias") is not None for g in gates):
            bias = np.stack([np.zeros(H) if g.get("bias") is None else np.asarray(g["bias"], dtype=np.float64)
                             for g in gates])
        top = l == L - 1
        out = np.zeros((T, B, H))
        h, c = h_last[l].copy(), c_last[l].copy()
        for t in range(T):
            xt = np.concatenate([layer_in[t], h], axis=1)        # x~ = [x_t ; h_{t-1}]
            ys, snaps = [], []
            for g in gates:
                y_g, s_g = refinement_sums(g, xt, K, cps if top else (), counter)
                ys.append(y_g)
                snaps.append(s_g)
            if top:
                for j, k in enumerate(cps):
                    hj, cj = lstm_cell(np.stack([s[k] for s in snaps]), c, bias)
                    ckpt_h[j, t], ckpt_c[j, t] = hj, cj
            h, c = lstm_cell(np.stack(ys), c, bias)
            out[t] = h
        h_last[l], c_last[l] = h, c
        layer_in = out
    return {"h": layer_in, "h_last": h_last, "c_last": c_last, "ckpt_h": ckpt_h, "ckpt_c": ckpt_c}


def op_count(H: int, nz: int, K: int) -> int:
    """Operations per gate per timestep and stream: N_steps (2R + 2NZ + 1), Sec. III."""
    return K * (2 * H + 2 * nz + 1)
