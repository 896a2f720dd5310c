"""The parity suite against the debug build of the library.

That build (kernels compiled with TB_DEBUG_BOUNDS) checks every global-memory
index of every kernel against the extents the kernel was given; a failed check
skips the access and is counted.  This test builds it and runs every other GPU
test in a child process that loads it (TB_DEBUG_BOUNDS=1), with the guard
canaries in place; after each of those tests the count of failed checks must
be zero.  It also checks that the normal build reports no debug checks."""
import os
import subprocess
import sys

import pytest

torch = pytest.importorskip("torch")
tv = pytest.importorskip("paper_2606_27550_gb300")

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_normal_build_has_no_debug_checks():
    from paper_2606_27550_gb300 import build

    build.build()
    torch.cuda.set_device(0)
    if os.environ.get("TB_DEBUG_BOUNDS") == "1":
        assert tv.tb_debug_bounds_build()
    else:
        assert not tv.tb_debug_bounds_build()
        assert tv.tb_debug_bounds_violations() == 0


@pytest.mark.skipif(os.environ.get("TB_DEBUG_BOUNDS") == "1", reason="already running against the debug build")
def test_parity_suite_in_debug_bounds_build():
    from paper_2606_27550_gb300 import build

    build.build(debug_bounds=True)
    env = dict(os.environ, TB_DEBUG_BOUNDS="1")
    cmd = [sys.executable, "-m", "pytest", os.path.join(ROOT, "tests"), "-m", "gpu", "-x", "-q", "-p",
           "no:cacheprovider", "--deselect", "tests/test_gpu_debug_bounds.py::test_parity_suite_in_debug_bounds_build"]
    r = subprocess.run(cmd, cwd=ROOT, env=env, capture_output=True, text=True)
    tail = (r.stdout + r.stderr)[-4000:]
    assert r.returncode == 0, tail
    assert " passed" in tail and "failed" not in tail, tail
