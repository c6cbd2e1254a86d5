"""The bounds-checking debug build (SSD_DEBUG_BOUNDS=1, libssd_debug.so):
built here, then a subset of the GPU parity tests runs against it in a child
process (SSD_LIBRARY=debug makes the binding load it).  The checks record
SSD_ERR_DEVICE_BOUNDS and skip the access instead of trapping, so on valid
inputs they must pass silently and change no result: the subset's parity
assertions and status checks are the test."""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

SUBSET = [
    "tests/test_gpu_debug_bounds.py::test_the_loaded_library_is_the_debug_build",
    "tests/test_gpu_attention.py::test_config1_shape",
    "tests/test_gpu_attention.py::test_long_cache_many_splits",
    "tests/test_gpu_attention.py::test_mma_sync_and_tensor_core_paths_agree",
    "tests/test_gpu_attention.py::test_split_merge_ignores_workspace_contents",
    "tests/test_gpu_step.py::test_committed_draw_is_the_full_draw_bit_for_bit",
    "tests/test_gpu_lmhead.py::test_fused_lmhead_matches_oracle",
    "tests/test_zz_no_alloc.py",
]


def test_the_loaded_library_is_the_debug_build():
    if os.environ.get("SSD_LIBRARY") != "debug":
        pytest.skip("runs in the child process of the debug-build test")
    import paper_2606_20543_gb300 as m
    assert m.load()._name.endswith("libssd_debug.so")


def test_debug_bounds_build_passes_a_parity_subset():
    if os.environ.get("SSD_LIBRARY") == "debug":
        pytest.skip("the child process runs the subset itself")
    from paper_2606_20543_gb300 import build
    assert build.build(debug_bounds=True).endswith("libssd_debug.so")
    env = dict(os.environ, SSD_LIBRARY="debug")
    r = subprocess.run([sys.executable, "-m", "pytest", "-q", "-x", "-m", "gpu",
                        "-p", "no:cacheprovider", *SUBSET],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=1500)
    print(r.stdout[-1500:])
    assert r.returncode == 0, r.stdout[-4000:] + r.stderr[-2000:]
    assert " passed" in r.stdout and "skipped" not in r.stdout.splitlines()[-1]
