"""The multi-GPU path of bench.py, on CPU with gloo (world size 2).

Prompts are independent, so a job shards the forest by prompt: every rank
builds and decodes its own trees (no collective on the data path) and the
job's time is the slowest rank's. These tests run the rank-side host work
(workload sharding, tree building and scheduling through the C ABI on a
metadata-only tree) in two gloo processes and check the reductions bench.py
uses.
"""
import os
import socket
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    import torch.distributed as dist

    import bench
    import paper_2508_17445_gb300 as tp

    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        class A:
            workload, seed, prompts = "qwen7b", 7, 2
        script = bench.make_script(A, bench.shard_seed(A.seed, rank))
        desc = bench.describe(script)
        h = script.heads
        f = tp.Forest(h.num_q_heads, h.num_kv_heads, h.head_dim, pool_blocks=1 << 16, device=None)
        ids = f.replay(script.ops)
        sched = tp.tp_debug_schedule(f.handle, [ids[x] for x in script.leaves])
        fake_ms = 10.0 + 5.0 * rank          # rank 1 is the slow one
        ms = bench.max_over_ranks([fake_ms, float(desc["unique_kv_tokens"])])
        first_prompt = [op for op in script.ops if op[0] == "append"][0][3]
        prompts = bench.max_over_ranks([float(first_prompt) if r == rank else -1.0 for r in range(world)])
        out[rank] = {"ms": ms[0], "tokens_max": ms[1], "tokens": desc["unique_kv_tokens"],
                     "leaves": desc["leaves"], "units": len(sched["units"]), "prompts": prompts,
                     "rate": bench.job_rate(desc["leaves"], world, 4, ms[0])}
        f.close()
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_shard_by_prompt():
    world = 2
    with mp.Manager() as m:
        out = m.dict()
        mp.start_processes(_rank_main, args=(world, _free_port(), out), nprocs=world, start_method="spawn")
        res = dict(out)
    assert set(res) == {0, 1}
    # both ranks see the slowest rank's time and agree on every reduction
    assert res[0]["ms"] == res[1]["ms"] == 15.0
    assert res[0]["tokens_max"] == res[1]["tokens_max"] == max(res[0]["tokens"], res[1]["tokens"])
    assert res[0]["prompts"] == res[1]["prompts"]
    # the shards are different forests of the same shape
    assert res[0]["prompts"][0] != res[0]["prompts"][1]
    assert res[0]["leaves"] == res[1]["leaves"] == 32
    assert res[0]["units"] > 0 and res[1]["units"] > 0
    # whole-job rate: all ranks' leaves over the slowest rank's time
    assert res[0]["rate"] == pytest.approx(32 * 2 * 4 / 0.015)
