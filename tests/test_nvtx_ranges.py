"""NVTX ranges of the C ABI (profiling aid): every compute entry point pushes one range named after itself and
pops it on every return path. A small NVTX tool (tests/nvtx_record_tool.c, written against the NVTX v3 injection
interface of the CUDA toolkit's headers) records the pushes and pops of a child process that calls each entry
point with arguments its validation rejects, so no GPU is needed. Without a tool the ranges are inert: the same
calls return the same status with an injection path that does not load."""
import os
import shutil
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
TOOL_SRC = os.path.join(ROOT, "tests", "nvtx_record_tool.c")
NVTX_INCLUDE = "/usr/local/cuda/include"

# every compute entry point of include/mikv.h with arguments its validation rejects (null shape or sizes)
CALLS = {
    "mikv_compute_balancer": (None, None, None, 0, None, None, 0, None),
    "mikv_quantize_pack": (None, None, None, None, None, 0, None, 0, 0, None),
    "mikv_prefill_scores": (None, None, None, 0, 1.0, None, None, 0, None),
    "mikv_decode_attention": (None, None, 0, None, 1.0, None, 0, None, None, None, 0, None),
    "mikv_update_importance": (None, None, None, None, None),
    "mikv_select_demote": (0, 0, None, None, 0, 0, 0, None, None, None),
    "mikv_insert_token": (None, None, None, None, 0, None, None),
    "mikv_gather_hi": (None, None, None, None, None, None, 0, None, 0, None),
    "mikv_decode_step": (None, None, 0, None, None, None, 0, None, 1.0, None, 0, None, 0, None),
    "mikv_decode_attention_noalloc": (None, None, 0, None, 1.0, None, 0, None, None, None),
}

CHILD = """
import sys
sys.path.insert(0, {root!r})
import paper_2402_18096_gb300 as pkg
lib = pkg.load()
calls = {calls!r}
for name, args in calls.items():
    rc = getattr(lib, name)(*args)
    assert rc == 1, (name, rc)  # MIKV_ERR_ARG
print("ok")
"""


def _run_child(env_extra):
    import paper_2402_18096_gb300 as pkg
    pkg.load()  # build (if needed) in this process, not in the child
    env = dict(os.environ, **env_extra)
    r = subprocess.run([sys.executable, "-c", CHILD.format(root=ROOT, calls=CALLS)], env=env, capture_output=True,
                       text=True, timeout=300)
    assert r.returncode == 0, r.stderr
    assert r.stdout.strip().endswith("ok")


def test_every_entry_point_has_one_balanced_range(tmp_path):
    cc = shutil.which("gcc") or shutil.which("cc")
    if not cc or not os.path.exists(os.path.join(NVTX_INCLUDE, "nvtx3", "nvToolsExt.h")):
        pytest.skip("needs a C compiler and the CUDA toolkit's nvtx3 headers")
    tool = str(tmp_path / "libnvtx_record.so")
    subprocess.run([cc, "-shared", "-fPIC", "-O1", "-I", NVTX_INCLUDE, TOOL_SRC, "-o", tool], check=True)
    log = tmp_path / "ranges.txt"
    _run_child({"NVTX_INJECTION64_PATH": tool, "MIKV_NVTX_LOG": str(log)})
    lines = log.read_text().split("\n")[:-1]
    expected = []
    for name in CALLS:
        expected += [f"push {name}", "pop"]
    assert lines == expected


def test_ranges_inert_without_a_tool(tmp_path):
    _run_child({"NVTX_INJECTION64_PATH": str(tmp_path / "no_such_tool.so")})
