"""Every C-ABI entry point, built for the host from the kernel and API sources
with AddressSanitizer and UBSan, called through ctypes the way a user calls
it, on buffers of exactly the sizes include/qx.h states; results against the
oracle (tests/emulation/api_check.py); and the Python binding driven against
that build (tests/emulation/binding_check.py).  No GPU; the library never
loads this build."""
import os
import shutil
import subprocess
import sys

import pytest

HERE = os.path.join(os.path.dirname(os.path.abspath(__file__)), "emulation")


def _run_under_sanitizers(emulation_dir, script, marker):
    gxx = shutil.which("g++")
    if gxx is None:
        pytest.skip("g++ is not available")
    sys.path.insert(0, HERE)
    import translate

    lib = translate.build(gxx, str(emulation_dir), "library")
    runtimes = [subprocess.run([gxx, f"-print-file-name={n}"], capture_output=True, text=True).stdout.strip()
                for n in ("libasan.so", "libubsan.so")]
    # the emulation runs kernels thousands of times slower than a GPU: its bounded
    # waits get minutes, not the default two seconds
    env = dict(os.environ, LD_PRELOAD=" ".join(runtimes), ASAN_OPTIONS="detect_leaks=0", QX_EMU_SMS="3",
               QX_WAIT_LIMIT_MS="300000")
    r = subprocess.run([sys.executable, os.path.join(HERE, script), lib], capture_output=True, text=True,
                       env=env, timeout=1800)
    assert r.returncode == 0 and marker in r.stdout, (r.stdout[-2000:] + r.stderr[-4000:])


def test_every_entry_point_under_the_sanitizers(emulation_dir):
    _run_under_sanitizers(emulation_dir, "api_check.py", "api ok")


def test_python_binding_under_the_sanitizers(emulation_dir):
    """The wrappers of paper_2505_07531_gb300/qx.py (Q4X calls, recipe selection
    with a Q4X candidate, GemvChain, DecodeStep) with host tensors standing in
    for device tensors (tests/emulation/binding_check.py)."""
    _run_under_sanitizers(emulation_dir, "binding_check.py", "binding ok")
