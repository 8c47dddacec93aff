"""The C-ABI library loads and exports every entry point its header declares.

Runs without a GPU: no call here launches or computes anything.
"""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    names = set()
    inc = os.path.join(ROOT, "include")
    for f in os.listdir(inc):
        if f.endswith(".h"):
            text = open(os.path.join(inc, f)).read()
            text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
            names |= set(re.findall(r"\b(lstm_approx_\w+)\s*\(", text))
    return names


@pytest.fixture(scope="module")
def built_lib():
    from paper_1905_00689_gb300 import build as b
    b.build()
    from paper_1905_00689_gb300 import _binding
    return _binding.load()


def test_header_declares_the_boundary():
    names = _declared()
    for n in ("lstm_approx_create", "lstm_approx_set_factors", "lstm_approx_run", "lstm_approx_destroy",
              "lstm_approx_get_mask", "lstm_approx_last_error"):
        assert n in names


def test_library_exports_every_declared_symbol(built_lib):
    for n in sorted(_declared()):
        assert hasattr(built_lib, n), f"{n} declared in include/ but not exported"


def test_binding_covers_every_declared_symbol():
    from paper_1905_00689_gb300 import _binding
    assert set(_binding.EXPORTS) == _declared()


def test_invalid_arguments_rejected_before_any_device_work(built_lib):
    h = ctypes.c_void_p()
    dims = (ctypes.c_int * 2)(16, 99)
    # layer 1's input must equal the hidden size
    assert built_lib.lstm_approx_create(ctypes.byref(h), 2, dims, 8, 4, 1, 0, None) == 1
    assert built_lib.lstm_approx_create(ctypes.byref(h), 0, dims, 8, 4, 1, 0, None) == 1
    assert built_lib.lstm_approx_create(ctypes.byref(h), 1, dims, 8, 4, 1, 7, None) == 1
    assert built_lib.lstm_approx_create(None, 1, dims, 8, 4, 1, 0, None) == 1
    assert h.value is None
    # NULL handles are rejected, destroy is NULL-safe
    assert built_lib.lstm_approx_run(None, None, 1, 1, 1, None, None, None, None, None, 0, None, None) == 1
    assert built_lib.lstm_approx_sync(None) == 1
    built_lib.lstm_approx_destroy(None)
    assert built_lib.lstm_approx_last_error(None) == b"invalid handle (NULL)"
    # the dense comparator's process-wide launch order: 0 or 1 only
    assert built_lib.lstm_approx_dense_set_launch_order(2) == 1
    assert built_lib.lstm_approx_dense_set_launch_order(-1) == 1
    assert built_lib.lstm_approx_dense_set_launch_order(1) == 0
    assert built_lib.lstm_approx_dense_set_launch_order(0) == 0


def test_no_cpu_fallback_without_a_device(built_lib):
    import torch
    if torch.cuda.is_available():
        pytest.skip("a CUDA device is present")
    h = ctypes.c_void_p()
    dims = (ctypes.c_int * 1)(16)
    assert built_lib.lstm_approx_create(ctypes.byref(h), 1, dims, 8, 4, 1, 0, None) == 3  # ECUDA
    assert h.value is None


def test_header_is_c_and_a_c_client_links(built_lib, tmp_path):
    """tests/c_client.c, compiled as strict C99 against the header and linked
    to the library, gets the documented answers from the device-free calls."""
    import shutil
    import subprocess
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    pkg = os.path.join(ROOT, "paper_1905_00689_gb300")
    exe = str(tmp_path / "c_client")
    subprocess.run([cc, "-std=c99", "-Wall", "-Wextra", "-Werror", "-pedantic", "-I", os.path.join(ROOT, "include"),
                    os.path.join(ROOT, "tests", "c_client.c"), "-L", pkg, "-llstm_approx", "-Wl,-rpath," + pkg,
                    "-o", exe], check=True, capture_output=True, text=True)
    lines = subprocess.run([exe], check=True, capture_output=True, text=True).stdout.splitlines()
    assert lines[0] == "plan 0 path 2 variant 1 cluster 16"
    assert lines[1].startswith("forced 1 ") and "fp32 factors only" in lines[1]
    import torch
    if not torch.cuda.is_available():
        assert lines[2] == "create 3 null"  # ECUDA: no CPU fallback
    assert lines[3] == "error invalid handle (NULL)"
    assert lines[4] == "tensor plan 0 tau splits 4 tau streams 64"
    assert lines[5] == "dense order 0 0"


def test_product_path_does_not_import_the_oracle():
    pkg = os.path.join(ROOT, "paper_1905_00689_gb300")
    for dirpath, _, files in os.walk(pkg):
        for f in files:
            if f.endswith((".py", ".cu", ".cuh", ".h")):
                text = open(os.path.join(dirpath, f)).read()
                assert not re.search(r"^\s*(from|import)\s+oracle", text, flags=re.M), f
                assert "oracle/" not in text, f


def _header_enum(prefix):
    """name -> value of the header's enumerators starting with `prefix`."""
    text = open(os.path.join(ROOT, "include", "lstm_approx.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return {m.group(1): int(m.group(2)) for m in re.finditer(r"\b(" + prefix + r"\w+)\s*=\s*(\d+)", text)}


def test_binding_constants_match_the_header():
    """The Python binding's option, query, path and status numbers are the
    header's, so a key added on one side cannot drift from the other."""
    from paper_1905_00689_gb300 import _binding as b
    for prefix, strip in (("LSTM_APPROX_OPT_", "LSTM_APPROX_"), ("LSTM_APPROX_Q_", "LSTM_APPROX_"),
                          ("LSTM_APPROX_PATH_", "LSTM_APPROX_"), ("LSTM_APPROX_PLAN_", "LSTM_APPROX_")):
        enum = _header_enum(prefix)
        assert enum, prefix
        for name, value in enum.items():
            py = name[len(strip):]
            assert getattr(b, py) == value, (py, getattr(b, py, None), value)


def test_bench_helpers():
    """p90 is the nearest-rank 90th percentile; the captured DRAM traffic is
    reported only while the recurrence kernel's sources match the capture."""
    import sys
    sys.path.insert(0, ROOT)
    import bench
    assert bench.p90([5.0]) == 5.0
    assert bench.p90(list(range(1, 11))) == 9
    assert bench.p90(list(range(100))) == 89
    assert bench.captured_traffic() in (None, bench.TRAFFIC_CAPTURE["bytes"])
    saved = dict(bench.TRAFFIC_CAPTURE)
    try:
        bench.TRAFFIC_CAPTURE["sha256"] = "0" * 64  # sources that no longer match the capture
        assert bench.captured_traffic() is None
    finally:
        bench.TRAFFIC_CAPTURE.update(saved)


def test_reference_arm_prints_the_contract_line():
    """bench.py --impl reference (the oracle on the host cores) prints one
    JSON line with every key the benchmark contract names."""
    import json
    import subprocess
    import sys
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--steps", "1",
                        "--warmup", "3"], capture_output=True, text=True, timeout=600, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    for key in ("impl", "metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better",
                "scaling", "vs_baseline", "dtype", "data", "config", "cpu_baseline", "e2e"):
        assert key in d, key
    assert d["impl"] == "reference" and d["steps"] == 1 and d["warmup"] == 3 and d["value"] > 0
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["value"] == d["value"]
    assert d["e2e"] == {"value": d["value"], "unit": d["unit"], "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}
    assert "workload" in d["config"]


def test_bench_refuses_fewer_than_three_warmup_steps():
    import subprocess
    import sys
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--warmup", "2"], capture_output=True,
                       text=True, timeout=300, cwd=ROOT)
    assert r.returncode != 0 and "--warmup must be >= 3" in r.stderr
