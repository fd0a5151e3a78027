"""tp_decode_noalloc: the decode entry point that allocates no device memory.

Some callers cannot call cudaMalloc while they decode -- a serving process
that carves up all device memory at start-up, or a latency-critical loop that
cannot take cudaMalloc's implicit synchronisation. For them the library keeps
the decode scratch (schedule and fp32 partials) in one static device array.
These tests call that entry point through the C ABI and compare it with
tp_decode_ex, on two calls in a row (the array keeps the previous call's
contents, so the second call must not depend on them). This file is
collected last on purpose.
"""
import numpy as np
import pytest
import torch

import paper_2508_17445_gb300 as tp
import workloads

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
TOL_O, TOL_LSE = 1e-2, 1e-3


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2508_17445_gb300 import build
    build.build()


def _forest(script):
    h = script.heads
    f = tp.Forest(h.num_q_heads, h.num_kv_heads, h.head_dim,
                  pool_blocks=script.upper_bound_blocks(32) + 64, device=DEV)
    ids = f.replay(script.ops, kv_fn=lambda kv_id: script.kv(kv_id, DEV))
    return f, [ids[x] for x in script.leaves]


@pytest.mark.parametrize("script", [workloads.qwen7b(seed=3, n_prompts=2),
                                    workloads.random_tree(seed=4, heads=workloads.Heads(8, 2, 64), n_prompts=3)],
                         ids=["qwen7b-2-prompts", "random-forest-hd64"])
def test_noalloc_matches_decode_on_two_calls(script):
    f, leaves = _forest(script)
    Q = script.q(DEV)
    O_ref, LSE_ref = f.decode(leaves, Q)
    f.sync()
    for _ in range(2):
        O = torch.full_like(O_ref, float("nan"))
        LSE = torch.full_like(LSE_ref, float("nan"))
        tp.tp_decode_noalloc(f.handle, leaves, Q, O, LSE)
        f.sync()
        d_o = (O.float() - O_ref.float()).abs().max().item()
        d_lse = (LSE - LSE_ref).abs().max().item()
        assert np.isfinite(d_o) and np.isfinite(d_lse)
        assert d_o <= TOL_O and d_lse <= TOL_LSE, (d_o, d_lse)
    f.close()


def test_noalloc_rejects_work_beyond_its_scratch():
    # 32 Qwen-shaped prompts need ~37 MB of fp32 partials: over the 32 MiB array
    script = workloads.qwen7b(seed=5, n_prompts=32)
    f, leaves = _forest(script)
    Q = script.q(DEV)
    O = torch.empty((len(leaves), 28, 128), dtype=torch.bfloat16, device=DEV)
    LSE = torch.empty((len(leaves), 28), dtype=torch.float32, device=DEV)
    with pytest.raises(tp.TreepoError) as e:
        tp.tp_decode_noalloc(f.handle, leaves, Q, O, LSE)
    assert e.value.code == "OOM" and "static scratch" in str(e.value)
    f.sync()
    f.close()
