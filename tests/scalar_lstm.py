"""A second, independently written scalar implementation of the recurrence.

Pure Python floats and loops, for tiny shapes only (brute-force pin of the
oracle).  It follows the same definitions -- x~ = [x_t; h_{t-1}] (Sec. III),
Eq. 1 for each gate, the cell update of Sec. II -- but keeps the pruned v as
a dense length-C list with zeros and evaluates every product element by
element, so it shares no code path with oracle.recurrence.
"""
import math


def _sig(z):
    if z >= 0:
        return 1.0 / (1.0 + math.exp(-z))
    e = math.exp(z)
    return e / (1.0 + e)


def scalar_run(layers, x, K, checkpoints=()):
    """layers[l][g] = dict(sigma, u, idx, val); x[T][B][D] nested lists/arrays.

    Returns (h_top[T][B][H], ckpt_h[J][T][B][H]) as nested lists.
    """
    T = len(x)
    B = len(x[0])
    H = len(layers[0][0]["u"][0])
    seq = [[list(map(float, x[t][b])) for b in range(B)] for t in range(T)]
    ck_out = [[[None] * B for _ in range(T)] for _ in checkpoints]
    for l, gates in enumerate(layers):
        top = l == len(layers) - 1
        C = len(seq[0][0]) + H
        dense_v = []
        for g in gates:
            rows = []
            for n in range(K):
                row = [0.0] * C
                for j, c in enumerate(g["idx"][n]):
                    row[int(c)] = float(g["val"][n][j])
                rows.append(row)
            dense_v.append(rows)
        new_seq = [[None] * B for _ in range(T)]
        for b in range(B):
            h = [0.0] * H
            c = [0.0] * H
            for t in range(T):
                xt = seq[t][b] + h
                pre = [[0.0] * H for _ in range(4)]
                snaps = {}
                for gi, g in enumerate(gates):
                    acc = [0.0] * H
                    for n in range(K):
                        d = 0.0
                        for cc in range(C):
                            d += dense_v[gi][n][cc] * xt[cc]
                        for r in range(H):
                            acc[r] += float(g["sigma"][n]) * float(g["u"][n][r]) * d
                        if (n + 1) in checkpoints:
                            snaps.setdefault(n + 1, [None] * 4)[gi] = list(acc)
                    pre[gi] = acc

                def cell(p, cprev):
                    hh, cc_ = [], []
                    for r in range(H):
                        ig = _sig(p[0][r])
                        fg = _sig(p[1][r])
                        gg = math.tanh(p[2][r])
                        og = _sig(p[3][r])
                        cn = fg * cprev[r] + ig * gg
                        cc_.append(cn)
                        hh.append(og * math.tanh(cn))
                    return hh, cc_

                if top:
                    for j, k in enumerate(checkpoints):
                        ck_out[j][t][b] = cell(snaps[k], c)[0]
                h, c = cell(pre, c)
                new_seq[t][b] = h
        seq = new_seq
    return seq, ck_out
