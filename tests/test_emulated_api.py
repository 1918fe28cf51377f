"""Every C-ABI entry point, built for the host from the kernel and API sources
with AddressSanitizer and UBSan, called through ctypes the way a user calls
it, on buffers of exactly the sizes include/qx.h states; results against the
oracle (tests/emulation/api_check.py).  No GPU; the library never loads this
build."""
import os
import shutil
import subprocess
import sys

import pytest

HERE = os.path.join(os.path.dirname(os.path.abspath(__file__)), "emulation")


def test_every_entry_point_under_the_sanitizers(emulation_dir):
    gxx = shutil.which("g++")
    if gxx is None:
        pytest.skip("g++ is not available")
    sys.path.insert(0, HERE)
    import translate

    lib = translate.build(gxx, str(emulation_dir), "library")
    runtimes = [subprocess.run([gxx, f"-print-file-name={n}"], capture_output=True, text=True).stdout.strip()
                for n in ("libasan.so", "libubsan.so")]
    env = dict(os.environ, LD_PRELOAD=" ".join(runtimes), ASAN_OPTIONS="detect_leaks=0", QX_EMU_SMS="3")
    r = subprocess.run([sys.executable, os.path.join(HERE, "api_check.py"), lib], capture_output=True, text=True,
                       env=env, timeout=1800)
    assert r.returncode == 0 and "api ok" in r.stdout, (r.stdout[-2000:] + r.stderr[-4000:])
