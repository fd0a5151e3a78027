"""Tracing: every attention call of the C ABI is one named NVTX range.

A profiler (nsys, ncu's NVTX filters) sees each call's host scheduling and
launches under a range named for the entry point. No GPU is needed to check
the ranges: a small injection library (``nvtx_probe.c``) takes NVTX's
range calls over in a child process and logs them, and the calls are made
on a metadata-only tree, where they fail validation after the range opens.
"""
import os
import subprocess
import sys

import pytest

from conftest import ROOT

CUDA_INCLUDE = os.path.join(os.environ.get("CUDA_HOME", "/usr/local/cuda"), "include")

CHILD = r"""
import ctypes, sys
sys.path.insert(0, sys.argv[1])
import paper_2508_17445_gb300 as tp
probe = ctypes.CDLL(sys.argv[2])
probe.probe_log.restype = ctypes.c_char_p
f = tp.Forest(8, 2, 64, pool_blocks=16, device=None)
root = f.add_root()
f.append(root, n_tokens=5)
lib = tp.load_library()
leaves = (ctypes.c_int32 * 1)(root)
counts = (ctypes.c_int32 * 1)(5)
codes = [lib.tp_decode_ex(f.handle, leaves, 1, None, None, None, 0),
         lib.tp_prefill(f.handle, leaves, counts, 1, None, None, None, 0),
         lib.tp_decode_host(f.handle, leaves, 1, None, None, None, 0),
         lib.tp_decode_noalloc(f.handle, leaves, 1, None, None, None, 0)]
print("CODES", codes)
print(probe.probe_log().decode(), end="")
"""


@pytest.fixture(scope="module")
def probe(tmp_path_factory):
    if not os.path.exists(os.path.join(CUDA_INCLUDE, "nvtx3", "nvToolsExt.h")):
        pytest.skip("NVTX headers not found")
    out = str(tmp_path_factory.mktemp("nvtx") / "libnvtx_probe.so")
    subprocess.check_call(["gcc", "-O1", "-shared", "-fPIC", "-I", CUDA_INCLUDE,
                           os.path.join(ROOT, "tests", "nvtx_probe.c"), "-o", out])
    return out


def test_each_attention_call_is_one_named_range(probe):
    from paper_2508_17445_gb300 import build
    build.build()
    env = dict(os.environ, NVTX_INJECTION64_PATH=probe)
    res = subprocess.run([sys.executable, "-c", CHILD, ROOT, probe], env=env, capture_output=True, text=True,
                         timeout=120)
    assert res.returncode == 0, res.stderr
    lines = res.stdout.strip().splitlines()
    assert lines[0] == "CODES [-1, -1, -1, -1]"       # metadata-only tree: TP_ERR_INVALID_ARG, after the range opened
    assert lines[1:] == ["push tp_decode_ex", "pop", "push tp_prefill", "pop", "push tp_decode_host", "pop",
                         "push tp_decode_noalloc", "pop"]
