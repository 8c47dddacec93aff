"""ctypes binding of liblstm_approx.so (argument marshalling only).

Every entry point of include/lstm_approx.h is exposed under its own name;
:class:`LSTMApprox` wraps a handle for callers holding torch tensors (device
memory and the current stream come from PyTorch; every step of the
recurrence runs in the library's kernels).  There is no fallback: if the
library is missing or cannot run, calls raise.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Sequence

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "liblstm_approx.so")

OK, EINVAL, ENOMEM, ECUDA, ETIMEOUT, ESTATE = range(6)
FP32, BF16 = 0, 1
Q_LAUNCHES, Q_LAST_PATH, Q_CLUSTER, Q_DEVICE_BYTES, Q_PERSISTENT_VARIANT, Q_TENSOR_SEQ = range(6)
PATH_NONE, PATH_SIMT, PATH_PERSISTENT, PATH_TENSOR = range(4)
(OPT_FORCE_PATH, OPT_CLUSTER, OPT_TIMING, OPT_WAIT_LIMIT, OPT_TEST_STALL, OPT_PERSISTENT_VARIANT, OPT_XPROJ,
 OPT_TAU_LAYOUT, OPT_TENSOR_SEQ, OPT_LAUNCH_ORDER) = range(10)
(PLAN_PATH, PLAN_PERSISTENT_VARIANT, PLAN_CLUSTER, PLAN_TERMS_PER_CTA, PLAN_UNITS_PER_WARP, PLAN_TERMS_PER_LANE,
 PLAN_VH_LAYOUT, PLAN_H_QUADS, PLAN_SMEM_BYTES, PLAN_TMEM_COLUMNS, PLAN_TAU_TILE_STREAMS, PLAN_GATE_TILE_STREAMS,
 PLAN_GATE_SPLITS, PLAN_TENSOR_SEQ, PLAN_TAU_SPLITS, PLAN_ITEMS) = range(16)
PLAN_KEYS = ("path", "persistent_variant", "cluster", "terms_per_cta", "units_per_warp", "terms_per_lane",
             "vh_layout", "h_quads", "smem_bytes", "tmem_columns", "tau_tile_streams", "gate_tile_streams",
             "gate_splits", "tensor_seq", "tau_splits")
STATUS_NAMES = {OK: "OK", EINVAL: "EINVAL", ENOMEM: "ENOMEM", ECUDA: "ECUDA", ETIMEOUT: "ETIMEOUT",
                ESTATE: "ESTATE"}

EXPORTS = (
    "lstm_approx_create", "lstm_approx_set_factors", "lstm_approx_run", "lstm_approx_run_host",
    "lstm_approx_sync", "lstm_approx_get_mask", "lstm_approx_last_error", "lstm_approx_destroy",
    "lstm_approx_query", "lstm_approx_set_option", "lstm_approx_phase_times", "lstm_approx_run_static",
    "lstm_approx_plan", "lstm_approx_get_term", "lstm_approx_dense_run", "lstm_approx_dense_workspace_bytes",
    "lstm_approx_dense_set_launch_order",
)

_lib = None


class LSTMApproxError(RuntimeError):
    def __init__(self, code: int, message: str):
        super().__init__(f"{STATUS_NAMES.get(code, code)}: {message}")
        self.code = code


def load(path: str = LIB_PATH):
    """Load the library (once).  Raises if it has not been built."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError(f"{path} is missing: build it with __graft_entry__.build() "
                           "or python -m paper_1905_00689_gb300.build")
    lib = ctypes.CDLL(path)
    P, I, LL = ctypes.c_void_p, ctypes.c_int, ctypes.c_longlong
    lib.lstm_approx_create.argtypes = [ctypes.POINTER(P), I, ctypes.POINTER(I), I, I, I, I, P]
    lib.lstm_approx_set_factors.argtypes = [P, I, I, I, I, P, P, P, P, P]
    run_args = [P, P, I, I, I, P, P, P, P, P, I, P, P]
    lib.lstm_approx_run.argtypes = run_args
    lib.lstm_approx_run_host.argtypes = run_args
    lib.lstm_approx_sync.argtypes = [P]
    lib.lstm_approx_get_mask.argtypes = [P, I, I, I, P, ctypes.POINTER(I)]
    lib.lstm_approx_get_term.argtypes = [P, I, I, I, P, P, P]
    lib.lstm_approx_last_error.argtypes = [P]
    lib.lstm_approx_last_error.restype = ctypes.c_char_p
    lib.lstm_approx_destroy.argtypes = [P]
    lib.lstm_approx_destroy.restype = None
    lib.lstm_approx_query.argtypes = [P, I, ctypes.POINTER(LL)]
    lib.lstm_approx_set_option.argtypes = [P, I, LL]
    lib.lstm_approx_phase_times.argtypes = [P, ctypes.POINTER(ctypes.c_float)]
    lib.lstm_approx_run_static.argtypes = [P, P, P, P, P, I, I, I, P, I, I, P, P, P, P, P, I, P, P, P,
                                           ctypes.c_char_p, I]
    lib.lstm_approx_plan.argtypes = [I, I, I, I, I, P, I, I, I, I, P, I, ctypes.c_char_p, I]
    lib.lstm_approx_dense_run.argtypes = [P, P, P, I, I, P, I, I, P, P, P, P, P, ctypes.c_size_t, P,
                                          ctypes.c_char_p, I]
    lib.lstm_approx_dense_workspace_bytes.argtypes = [I, I, I]
    lib.lstm_approx_dense_set_launch_order.argtypes = [I]
    for name in EXPORTS:
        if name not in ("lstm_approx_last_error", "lstm_approx_destroy", "lstm_approx_dense_workspace_bytes"):
            getattr(lib, name).restype = ctypes.c_int
    lib.lstm_approx_dense_workspace_bytes.restype = ctypes.c_size_t
    _lib = lib
    return lib


def _ptr(t) -> Optional[int]:
    """Device address of a torch tensor (None passes NULL)."""
    if t is None:
        return None
    if not t.is_contiguous() or t.dtype.itemsize != 4:
        raise ValueError("tensors must be contiguous fp32")
    return t.data_ptr()


def _np_ptr(a) -> Optional[int]:
    if a is None:
        return None
    return a.ctypes.data


def run_static(Vx, Vh, U, sigma, bias, x, K, out_h, h0=None, c0=None, out_c=None, checkpoints=(),
               ckpt_h=None, ckpt_c=None, stream=None):
    """lstm_approx_run_static on torch CUDA tensors (no handle, no device allocation).

    Vx [4][K][D], Vh [4][K][H], U [4][H][K], sigma [4][K], bias [4][H] or None:
    fp32 factors in the library's packed layout.  Synchronous.
    """
    import torch
    lib = load()
    T, B, D = x.shape
    H = Vh.shape[-1]
    if stream is None:
        stream = torch.cuda.current_stream()
    cps = (ctypes.c_int * max(1, len(checkpoints)))(*checkpoints)
    msg = ctypes.create_string_buffer(512)
    rc = lib.lstm_approx_run_static(_ptr(Vx), _ptr(Vh), _ptr(U), _ptr(sigma), _ptr(bias), D, H, K, _ptr(x), T, B,
                                    _ptr(h0), _ptr(c0), _ptr(out_h), _ptr(out_c), cps, len(checkpoints),
                                    _ptr(ckpt_h), _ptr(ckpt_c), ctypes.c_void_p(stream.cuda_stream), msg, 512)
    if rc != OK:
        raise LSTMApproxError(rc, msg.value.decode())


def dense_run(Wx, Wh, bias, x, out_h, h0=None, c0=None, out_c=None, workspace=None, stream=None):
    """lstm_approx_dense_run on torch tensors (device, fp32): the dense LSTM
    comparator.  `workspace` (a uint8 device tensor of at least
    dense_workspace_bytes(H, T, B) bytes) is allocated here when not given."""
    import torch
    lib = load()
    T, B, D = x.shape
    H = Wh.shape[1]
    need = lib.lstm_approx_dense_workspace_bytes(H, T, B)
    if workspace is None:
        workspace = torch.empty(need + 256, dtype=torch.uint8, device=x.device)
        off = (-workspace.data_ptr()) % 256
        workspace = workspace[off:off + need]
    s = stream if stream is not None else torch.cuda.current_stream(x.device)
    msg = ctypes.create_string_buffer(256)
    rc = lib.lstm_approx_dense_run(_ptr(Wx), _ptr(Wh), _ptr(bias), D, H, _ptr(x), T, B, _ptr(h0), _ptr(c0),
                                   _ptr(out_h), _ptr(out_c), workspace.data_ptr(), workspace.numel(),
                                   ctypes.c_void_p(s.cuda_stream), msg, 256)
    if rc != OK:
        raise LSTMApproxError(rc, msg.value.decode())


def dense_workspace_bytes(H: int, T: int, B: int) -> int:
    return int(load().lstm_approx_dense_workspace_bytes(H, T, B))


def dense_set_launch_order(order: int) -> None:
    """lstm_approx_dense_set_launch_order (process-wide)."""
    rc = load().lstm_approx_dense_set_launch_order(order)
    if rc != OK:
        raise LSTMApproxError(rc, f"bad launch order {order}")


def plan(dtype: int, hidden: int, T: int, B: int, K: int, checkpoints: Sequence[int] = (), force_path: int = 0,
         cluster: int = 0, variant: int = 0) -> dict:
    """lstm_approx_plan: the kernels a run of one layer of this shape takes,
    as a dict keyed by PLAN_KEYS (host only, no device needed)."""
    lib = load()
    cps = (ctypes.c_int * max(1, len(checkpoints)))(*checkpoints)
    out = (ctypes.c_int * PLAN_ITEMS)()
    msg = ctypes.create_string_buffer(512)
    rc = lib.lstm_approx_plan(dtype, hidden, T, B, K, cps, len(checkpoints), force_path, cluster, variant, out,
                              PLAN_ITEMS, msg, 512)
    if rc != OK:
        raise LSTMApproxError(rc, msg.value.decode())
    return dict(zip(PLAN_KEYS, list(out)))


class LSTMApprox:
    """One handle of the library.

    `stream` is a torch.cuda.Stream (default: torch's current stream on the
    current device); tensors passed to :meth:`run` must live on that device.
    """

    def __init__(self, num_layers: int, input_dims: Sequence[int], hidden: int, max_rank: int,
                 max_batch: int, dtype: str = "fp32", stream=None):
        import torch
        self.lib = load()
        self.L, self.H = num_layers, hidden
        self.input_dims = list(input_dims)
        self.dtype = dtype
        if stream is None:
            stream = torch.cuda.current_stream()
        self.stream = stream
        dims = (ctypes.c_int * num_layers)(*self.input_dims)
        h = ctypes.c_void_p()
        rc = self.lib.lstm_approx_create(ctypes.byref(h), num_layers, dims, hidden, max_rank, max_batch,
                                         BF16 if dtype == "bf16" else FP32,
                                         ctypes.c_void_p(stream.cuda_stream))
        if rc != OK:
            raise LSTMApproxError(rc, "lstm_approx_create failed")
        self.h = h

    # -- helpers ---------------------------------------------------------
    def _check(self, rc: int):
        if rc != OK:
            msg = self.lib.lstm_approx_last_error(self.h).decode()
            raise LSTMApproxError(rc, msg)

    def close(self):
        if getattr(self, "h", None):
            self.lib.lstm_approx_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # -- entry points ----------------------------------------------------
    def set_factors(self, layer: int, gate: int, sigma, u, idx, val, bias=None):
        sigma = np.ascontiguousarray(sigma, dtype=np.float64)
        u = np.ascontiguousarray(u, dtype=np.float64)
        idx = np.ascontiguousarray(idx, dtype=np.int32)
        val = np.ascontiguousarray(val, dtype=np.float64)
        K, nz = idx.shape
        b = None if bias is None else np.ascontiguousarray(bias, dtype=np.float64)
        self._check(self.lib.lstm_approx_set_factors(self.h, layer, gate, K, nz, _np_ptr(sigma), _np_ptr(u),
                                                     _np_ptr(idx), _np_ptr(val), _np_ptr(b)))

    def set_layer(self, layer: int, gates):
        """gates: four dicts with sigma, u, idx, val (and optional bias)."""
        for g, f in enumerate(gates):
            self.set_factors(layer, g, f["sigma"], f["u"], f["idx"], f["val"], f.get("bias"))

    def run(self, x, K: int, out_h, h0=None, c0=None, out_c=None, checkpoints=(), ckpt_h=None, ckpt_c=None):
        """Device run; x [T][B][D] fp32 CUDA tensor, out_h [T][B][H]."""
        T, B = x.shape[0], x.shape[1]
        cps = (ctypes.c_int * max(1, len(checkpoints)))(*checkpoints)
        self._check(self.lib.lstm_approx_run(self.h, _ptr(x), T, B, K, _ptr(h0), _ptr(c0), _ptr(out_h),
                                             _ptr(out_c), cps, len(checkpoints), _ptr(ckpt_h), _ptr(ckpt_c)))

    def run_host(self, x: np.ndarray, K: int, out_h: np.ndarray, h0=None, c0=None, out_c=None,
                 checkpoints=(), ckpt_h=None, ckpt_c=None):
        """Host-buffer run (float32 numpy arrays, C order); synchronous."""
        for a in (x, out_h, h0, c0, out_c, ckpt_h, ckpt_c):
            if a is not None and (a.dtype != np.float32 or not a.flags["C_CONTIGUOUS"]):
                raise ValueError("host buffers must be C-contiguous float32")
        T, B = x.shape[0], x.shape[1]
        cps = (ctypes.c_int * max(1, len(checkpoints)))(*checkpoints)
        self._check(self.lib.lstm_approx_run_host(self.h, _np_ptr(x), T, B, K, _np_ptr(h0), _np_ptr(c0),
                                                  _np_ptr(out_h), _np_ptr(out_c), cps, len(checkpoints),
                                                  _np_ptr(ckpt_h), _np_ptr(ckpt_c)))

    def sync(self):
        self._check(self.lib.lstm_approx_sync(self.h))

    def get_mask(self, layer: int, gate: int, k: int) -> np.ndarray:
        C = self.input_dims[layer] + self.H
        out = np.zeros(C, dtype=np.int32)
        n = ctypes.c_int(0)
        self._check(self.lib.lstm_approx_get_mask(self.h, layer, gate, k, _np_ptr(out), ctypes.byref(n)))
        return out[: n.value].copy()

    def get_term(self, layer: int, gate: int, k: int):
        """(sigma, u [H], dense v [C]) of one stored term, as fp32 numpy arrays."""
        C = self.input_dims[layer] + self.H
        sigma = np.zeros(1, dtype=np.float32)
        u = np.zeros(self.H, dtype=np.float32)
        v = np.zeros(C, dtype=np.float32)
        self._check(self.lib.lstm_approx_get_term(self.h, layer, gate, k, _np_ptr(sigma), _np_ptr(u), _np_ptr(v)))
        return float(sigma[0]), u, v

    def query(self, key: int) -> int:
        v = ctypes.c_longlong(0)
        self._check(self.lib.lstm_approx_query(self.h, key, ctypes.byref(v)))
        return v.value

    def set_option(self, key: int, value: int):
        self._check(self.lib.lstm_approx_set_option(self.h, key, value))

    def phase_times(self):
        ms = (ctypes.c_float * 3)()
        self._check(self.lib.lstm_approx_phase_times(self.h, ms))
        return list(ms)
