"""Quality-of-result curves computed from the library's own outputs (GPU).

The paper's progressive-inference curve (Sec. VI-B, Fig. 5a: output quality
against refinement depth) is measured here on the seeded small workload
(D = H = 64, T = 8, one stream) with the oracle's residual decomposition of
its Gaussian gate matrices at three pruning levels, and compared point by
point with the same curve computed by the oracle:

* reading A: one run per depth K (the model truncated at K for every t),
  against oracle.qor.qor_table;
* reading B: one run at K = 64 whose intermediate outputs at 1, 4, 16, 64
  are the progressive estimates (h_{t-1}, c_{t-1} from the full-depth
  chain), against the oracle's intermediate outputs.

Each point is the relative error of h against the dense LSTM of Sec. II and
the KL divergence of a seeded random linear head's softmax (qor.curve_point).
The fp32 path runs on the persistent kernel, the bf16 path on the tensor
cores; the bf16 curve is compared with the oracle on the bf16-stored factors.
"""
import numpy as np
import pytest

import oracle
from oracle import qor
from parity_util import NOTES, oracle_run, run_gpu
from workloads import WORKLOADS, draw_inputs, draw_weights, rounded_factors

pytestmark = pytest.mark.gpu

KS = (1, 4, 16, 64)
NZS = (128, 64, 16)  # keep 1, 1/2, 1/8 of C = 128


@pytest.fixture(scope="module")
def small_workload():
    w = WORKLOADS["c1"]
    weights = draw_weights(w, 0)
    x = draw_inputs(8, 1, w.D, w.x_dist, 4242)
    h_ref = qor.dense_lstm(weights, x)
    layers = {nz: [oracle.decompose_gate(W, max(KS), nz) for W in weights] for nz in NZS}
    return w, weights, x, h_ref, layers


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
def test_quality_curve_from_the_library(cuda_device, small_workload, dtype):
    from paper_1905_00689_gb300 import PATH_PERSISTENT, PATH_TENSOR, Q_LAST_PATH
    w, weights, x, h_ref, layers = small_workload
    A = qor.head_matrix(w.H)
    x32 = x.astype(np.float32).astype(np.float64)
    h_tol = 1e-4 if dtype == "fp32" else 2e-3
    want_path = PATH_PERSISTENT if dtype == "fp32" else PATH_TENSOR
    oracle_rows = {(r["NZ"], r["K"]): r for r in qor.qor_table(weights, x, NZS, KS)} if dtype == "fp32" else None
    lines = [f"quality against depth from the library, {w.name} ({dtype}, T=8, one stream)",
             "| NZ | K | rel. h error, per-K runs | head KL, per-K runs | rel. h error, one run's outputs at k_j "
             "| head KL, one run's outputs at k_j |", "|---|---|---|---|---|---|"]
    for nz in NZS:
        layer = layers[nz]
        # reading B: one run, intermediate outputs at every depth of the curve
        got_b, m = run_gpu([layer], x, max(KS), dtype=dtype, checkpoints=list(KS))
        assert m.query(Q_LAST_PATH) == want_path
        ref_b = oracle_run([layer], x, max(KS), dtype=dtype, checkpoints=list(KS))
        for i, K in enumerate(KS):
            # reading A: the model truncated at K
            got_a, m = run_gpu([layer], x, K, dtype=dtype, max_rank=max(KS))
            pa = qor.curve_point(got_a["h"], h_ref, A)
            if dtype == "fp32":
                wa = oracle_rows[(nz, K)]           # the oracle's own table (fp64 factors)
            else:
                wa = qor.curve_point(oracle.run_lstm([rounded_factors(layer, "bf16")], x32, K)["h"], h_ref, A)
            pb = qor.curve_point(got_b["ckpt_h"][i], h_ref, A)
            wb = qor.curve_point(ref_b["ckpt_h"][i], h_ref, A)
            for got, want in ((pa, wa), (pb, wb)):
                assert abs(got["rel_h_error"] - want["rel_h_error"]) <= h_tol, (nz, K, got, want)
                assert abs(got["head_kl"] - want["head_kl"]) <= 1e-5 + 1e-2 * abs(want["head_kl"]), (nz, K, got, want)
            lines.append(f"| {nz} | {K} | {pa['rel_h_error']:.3g} | {pa['head_kl']:.3g} | {pb['rel_h_error']:.3g} "
                         f"| {pb['head_kl']:.3g} |")
        # the progressive estimate at the full depth is the run's own output
        assert np.array_equal(got_b["ckpt_h"][-1], got_b["h"])
    NOTES.extend(lines + [""])
