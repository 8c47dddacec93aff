"""Progressive approximate-LSTM inference on GB300 (sm_103a).

The compute path is the C-ABI library ``liblstm_approx.so`` (CUDA kernels,
declared in include/lstm_approx.h); this package is its thin Python binding.
Importing the package does not load the library; constructing
:class:`LSTMApprox` (or calling :func:`load`) does, and raises if it has not
been built.
"""
from ._binding import (  # noqa: F401
    BF16, FP32, LSTMApprox, LSTMApproxError, dense_run, dense_set_launch_order, dense_workspace_bytes, load, plan,
    run_static, PLAN_KEYS,
    PATH_NONE, PATH_PERSISTENT, PATH_SIMT, PATH_TENSOR,
    OPT_CLUSTER, OPT_FORCE_PATH, OPT_LAUNCH_ORDER, OPT_PERSISTENT_VARIANT, OPT_TAU_LAYOUT, OPT_TENSOR_SEQ,
    OPT_TEST_STALL, OPT_TIMING, OPT_WAIT_LIMIT, OPT_XPROJ,
    Q_CLUSTER, Q_DEVICE_BYTES, Q_LAST_PATH, Q_LAUNCHES, Q_PERSISTENT_VARIANT, Q_TENSOR_SEQ,
)
