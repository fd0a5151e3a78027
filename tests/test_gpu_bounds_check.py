"""The bounds-checked build on the GPU, on valid inputs.

libtreepo_checked.so (TP_BOUNDS_CHECK) checks every schedule-derived index
in every kernel before the access: tile words against the pool, unit
records against the schedule's sections, occurrence entries, partial
slots, merge ranges, token-append slots and schedule patch positions. On
valid input no check may fail and the results must be those of the default
build: the parity, prefill, rollout (token appends, schedule patches),
gather and host-buffer tests run again in a child process that loads the
checked library (TREEPO_BOUNDS_CHECK=1). Each of them synchronises through
tp_sync, which raises on any flagged check. Only valid inputs are used: the
predicates themselves are tested with planted bad words on the host
(test_bounds_check.py), never on the GPU.
"""
import os
import subprocess
import sys

import pytest
import torch

from conftest import ROOT

pytestmark = pytest.mark.gpu

CASES = [
    "tests/test_gpu_parity.py",
    "tests/test_gpu_prefill.py",
    "tests/test_gpu_rollout.py",
    "tests/test_gpu_host_buffers.py",
]


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2508_17445_gb300 import build
    build.build(checked=True)


def test_child_loads_the_checked_library():
    env = dict(os.environ, TREEPO_BOUNDS_CHECK="1")
    out = subprocess.run([sys.executable, "-c", "import paper_2508_17445_gb300 as tp; tp.load_library(); "
                          "print(tp.library_path())"], cwd=ROOT, env=env, capture_output=True, text=True, timeout=300)
    assert out.returncode == 0, out.stderr
    assert out.stdout.strip().endswith("libtreepo_checked.so")


def test_valid_inputs_pass_every_check_with_the_same_results():
    env = dict(os.environ, TREEPO_BOUNDS_CHECK="1")
    # the full-size sampled cases are skipped for time; every other case of
    # those files runs under the checked build
    cmd = [sys.executable, "-m", "pytest", "-q", "-x", "-m", "gpu", "-p", "no:cacheprovider", "-k",
           "not full_size", *CASES]
    res = subprocess.run(cmd, cwd=ROOT, env=env, capture_output=True, text=True, timeout=1500)
    tail = "\n".join((res.stdout + res.stderr).splitlines()[-25:])
    assert res.returncode == 0, tail
    assert " passed" in tail and "failed" not in tail, tail
