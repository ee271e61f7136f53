"""The checked build (-DMIKV_DEBUG) against the normal parity cases: in a process of its own with MIKV_DEBUG=1, the
package builds and loads libmikv_debug.so; its index checks must stay silent on valid inputs (the attention,
decode-step and fused-step parity tests pass unchanged and the status words stay clear) and must report invalid
ones (tests/test_gpu_debug_checks.py)."""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_checked_build_passes_the_normal_cases():
    env = dict(os.environ, MIKV_DEBUG="1", MIKV_REQUIRE_DEBUG="1")
    cases = ["tests/test_gpu_debug_checks.py",
             "tests/test_gpu_attention.py::test_decode_steps_trajectory",
             "tests/test_gpu_attention.py::test_attention_matches_oracle",
             "tests/test_gpu_step_fused.py",
             "tests/test_gpu_kch.py::test_kch_decode_steps_across_a_group",
             "tests/test_gpu_hiquant.py::test_coded_important_set_decode_steps"]
    r = subprocess.run([sys.executable, "-m", "pytest", "-q", "-x", "-m", "gpu", "-p", "no:cacheprovider", *cases],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=1500)
    assert r.returncode == 0, r.stdout[-3000:] + r.stderr[-2000:]
    assert " passed" in r.stdout and "skipped" not in r.stdout, r.stdout[-2000:]
