"""The checked build: the library compiled with -DCLOVER_CHECKED, whose kernels
check every index they compute before the global access it guards and, on a
failed check, set CLOVER_ERR_CHECK (128) in the status word and skip the
access instead of trapping.

The test builds that variant and runs a selection of the parity tests in a
child process that loads it (CLOVER_VERIFY_CHECKED=1).  Those tests assert
status 0 after every call and compare with the oracle, so a check that fires
on a valid input, or a check that changes a result, fails them.  The child
first confirms that the library it loaded reports the checked build.
"""

import os
import subprocess
import sys

import pytest

from paper_2405_00263_gb300 import _lib
from paper_2405_00263_gb300 import build as _build

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

# parity tests that reach every checked site: both attention kernels with
# split-KV merges and every launch mode, the paged attention, the commit and
# compaction kernels, and the accept kernel's commit
SELECTION = [
    "tests/test_gpu_parity.py::test_small_step_matches_oracle",
    "tests/test_gpu_parity.py::test_small_step_inputs_ready_plan",
    "tests/test_gpu_parity.py::test_pair_kernel_step_matches_oracle",
    "tests/test_gpu_parity.py::test_full_row_tiles_with_empty_splits",
    "tests/test_gpu_parity.py::test_split_counts_and_row_groups",
    "tests/test_gpu_parity.py::test_step_attention_launch_modes",
    "tests/test_gpu_parity.py::test_commit_and_compact_schedules_agree",
    "tests/test_gpu_parity.py::test_kv_commit_matches_oracle",
    "tests/test_gpu_parity.py::test_one_workspace_serves_smaller_capacities",
    "tests/test_gpu_paged.py",
]


def test_checked_build_passes_parity(cuda):
    _build.build(checked=True)
    env = dict(os.environ, **{_lib.CHECKED_ENV: "1"})
    probe = ("import paper_2405_00263_gb300 as p; from paper_2405_00263_gb300 import _lib; "
             "assert p.clover_build_flags() & _lib.BUILD_CHECKED, 'not the checked build'; "
             "print(_lib.library_path())")
    r = subprocess.run([sys.executable, "-c", probe], cwd=ROOT, env=env, capture_output=True, text=True,
                       timeout=300)
    assert r.returncode == 0, r.stdout + r.stderr
    assert r.stdout.strip() == _build.CHECKED_LIB
    r = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-m", "gpu", "-p", "no:cacheprovider",
                        *SELECTION], cwd=ROOT, env=env, capture_output=True, text=True, timeout=1800)
    assert r.returncode == 0, (r.stdout + r.stderr)[-4000:]
    assert " passed" in r.stdout
