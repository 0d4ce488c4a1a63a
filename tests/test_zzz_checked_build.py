"""The range-checked build (``-DVOXZIP_CHECKED``) on the GPU parity cases.

In that build every kernel checks the index of each guarded global access against its buffer
before making it; a violation skips the access and sets VOXZIP_DEV_BOUNDS in the status word.
The GPU parity tests already demand a zero status word after each call, so running them again
with ``VOXZIP_CHECKED=1`` (which makes the binding load ``libvoxzip_checked.so``) shows that no
kernel indexes outside its buffers on any of those cases, and that the checks leave every result
unchanged.
"""
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PARITY_FILES = ["tests/test_gpu_parity.py", "tests/test_gpu_paged.py", "tests/test_gpu_policies.py",
                "tests/test_gpu_embed.py", "tests/test_zzzz_no_alloc.py"]


@pytest.mark.gpu
def test_checked_build_passes_the_parity_cases_with_no_bounds_bits():
    from paper_2608_08569_gb300.build import CHECKED_LIB_PATH, build_library

    assert build_library(checked=True) == CHECKED_LIB_PATH
    env = dict(os.environ, VOXZIP_CHECKED="1")
    probe = subprocess.run(
        [sys.executable, "-c",
         "import paper_2608_08569_gb300._native as N; N.lib(); "
         "print([l.split()[-1] for l in open('/proc/self/maps') if 'libvoxzip' in l][0])"],
        cwd=ROOT, env=env, capture_output=True, text=True, timeout=300)
    assert probe.returncode == 0, probe.stderr
    assert probe.stdout.strip() == CHECKED_LIB_PATH
    r = subprocess.run([sys.executable, "-m", "pytest", *PARITY_FILES, "-m", "gpu", "-x", "-q", "-p",
                        "no:cacheprovider"], cwd=ROOT, env=env, capture_output=True, text=True, timeout=1500)
    assert r.returncode == 0, r.stdout[-4000:] + r.stderr[-2000:]
