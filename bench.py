"""Tree-decode benchmark: leaf-queries/s of libtreepo's tp_decode on GB300.

One step = one tp_decode call over every live leaf of a seeded synthetic
forest shaped like TreePO rollouts (all rows of the hot path: tree-walk
schedule -> split-KV attention over shared path segments -> LSE merge).
Inputs (pool K/V, Q) are resident in HBM when the timed region starts; the
unique KV read per step (>= 1.8 GB for the full workloads) is far larger
than L2 (129 MB), so no flush is needed between steps.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
  python bench.py --impl reference ...   # the CPU oracle, timed on host cores

With torchrun, each rank builds its own forest (its prompts drawn with seed
+ rank) and decodes it on its own GPU: prompts are independent, so the job
shards with no collective on the data path (weak scaling).
Prints one JSON line on rank 0.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "tree-decode leaf-queries/s; HBM GB/s on unique KV bytes vs GB300 peak"
UNIT = "leaf-queries/s"
DEFAULT_WORKLOAD = "qwen7b"
FALLBACK_HBM_GBS = 6800.0


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=20)
    p.add_argument("--warmup", type=int, default=5)
    p.add_argument("--workload", default=DEFAULT_WORKLOAD,
                   choices=["tiny", "qwen7b", "random_divergence", "wide_prefix", "no_sharing"])
    p.add_argument("--seed", type=int, default=0)
    p.add_argument("--prompts", type=int, default=None,
                   help="scale the workload down to this many prompts (small cases for ncu captures)")
    p.add_argument("--impl", default="ours", choices=["ours", "reference"])
    p.add_argument("--flags", type=int, default=0, help="tp_decode_ex flags for the timed steps")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--cpu-seconds", type=float, default=12.0, help="CPU-baseline work budget")
    return p.parse_args()


# --------------------------------------------------------------------------
# workload description (structure only)
# --------------------------------------------------------------------------
def describe(script):
    """Unique and per-leaf path tokens of the live leaves, from the script."""
    par = script.parents()
    tok = script.node_tokens()
    seen, per_leaf = set(), []
    for lf in script.leaves:
        n, x = 0, lf
        while x != -1:
            seen.add(x)
            n += tok[x]
            x = par[x]
        per_leaf.append(n)
    h = script.heads
    kv_bytes_per_token = 2 * h.num_kv_heads * h.head_dim * 2
    uniq = sum(tok[x] for x in seen)
    return {
        "leaves": len(script.leaves),
        "unique_kv_tokens": uniq,
        "unique_kv_bytes": uniq * kv_bytes_per_token,
        "no_share_kv_bytes": sum(per_leaf) * kv_bytes_per_token,
        "q_bytes": len(script.leaves) * h.num_q_heads * h.head_dim * 2,
        "o_bytes": len(script.leaves) * h.num_q_heads * h.head_dim * 2,
        "lse_bytes": len(script.leaves) * h.num_q_heads * 4,
        "flops": sum(per_leaf) * 4 * h.num_q_heads * h.head_dim,
    }


def make_script(args, seed):
    import workloads
    kw = {"seed": seed}
    if args.prompts is not None:
        kw["n_seqs" if args.workload == "no_sharing" else "n_prompts"] = args.prompts
    return workloads.by_name(args.workload, **kw)


def shard_seed(seed, rank):
    """Rank r of a multi-GPU job decodes its own forest: prompts drawn with
    seed + r, so ranks hold independent trees and share nothing."""
    return seed + rank


def max_over_ranks(values, device="cpu"):
    """Element-wise max over ranks (the job's time is its slowest rank's)."""
    import torch
    import torch.distributed as dist
    t = torch.tensor(values, dtype=torch.float64, device=device)
    if dist.is_available() and dist.is_initialized() and dist.get_world_size() > 1:
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return t.tolist()


def job_rate(leaves_per_rank, world, steps, ms_total):
    """Whole-job leaf-queries/s: every rank's leaves, over the slowest rank's time."""
    return leaves_per_rank * world * steps / (ms_total / 1e3)


def workload_label(script):
    h = script.heads
    return f"{script.name}: {script.description}; {h.num_q_heads} q / {h.num_kv_heads} kv heads, head_dim {h.head_dim}, bf16"


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def kernel_source_hash():
    h = hashlib.sha256()
    for name in ("kernels.cu", "forest.h"):
        with open(os.path.join(ROOT, "paper_2508_17445_gb300", "csrc", name), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def recorded_traffic(workload):
    """DRAM bytes per decode launch from a committed ncu summary, if it was
    taken on the current kernel source; else None."""
    path = os.path.join(ROOT, "profiles", "decode_kernel_traffic.json")
    try:
        with open(path) as f:
            d = json.load(f)
        if d.get("kernel_source_hash") != kernel_source_hash():
            return None
        return d.get("per_launch_bytes", {}).get(workload)
    except Exception:
        return None


# --------------------------------------------------------------------------
# clocks sampled during the timed region
# --------------------------------------------------------------------------
class ClockSampler:
    FIELDS = ("pci.bus_id,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, bus_id):
        self.bus_id = (bus_id or "").lower()
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader",
                                          "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if not self.proc:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.t.join(timeout=2)
        rows = []
        for ln in self.lines:
            parts = [x.strip() for x in ln.split(",")]
            if len(parts) != 9:
                continue
            bus = parts[0].lower()
            if self.bus_id and not (bus.endswith(self.bus_id[-12:]) or self.bus_id.endswith(bus[-12:])):
                continue
            try:
                rows.append((float(parts[1].split()[0]), float(parts[2].split()[0]), parts[3], parts[4:]))
            except ValueError:
                continue
        if not rows:
            return None
        sm = [r[0] for r in rows]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i, v in enumerate(r[3][1:]) if v.lower() == "active"})
        loaded = [x for x in sm if x > 0.5 * max(sm)] or sm
        return {"sm_mhz": statistics.median(loaded), "sm_max_mhz": max(r[1] for r in rows), "reasons": reasons,
                "samples": len(rows)}


# --------------------------------------------------------------------------
# CPU oracle timing (the reported baseline; never on the product path)
# --------------------------------------------------------------------------
class OracleTimer:
    """Times the fp64 oracle on leaf samples of one forest, on all host cores.
    K/V of sampled paths are fetched into a host cache before timing."""

    def __init__(self, script, kv_device):
        import oracle
        self.oracle = oracle
        self.script = script
        self.kv_device = kv_device
        self.model = oracle.OracleForest(block_tokens=32, pool_blocks=script.upper_bound_blocks(32) + 64).replay(script)
        self.q = script.q("cpu")
        self.cores = os.cpu_count() or 1
        self.cache = {}

    def fetch(self, rows):
        for i in rows:
            for kv_id in self.model.path_chunks(self.script.leaves[i]):
                if kv_id not in self.cache:
                    k, v = self.script.kv(kv_id, self.kv_device)
                    self.cache[kv_id] = (self.oracle.bf16_bits(k.cpu()), self.oracle.bf16_bits(v.cpu()))

    def seconds(self, rows):
        self.fetch(rows)
        t0 = time.perf_counter()
        self.model.decode(self.script.leaves, self.q, lambda i: self.cache[i], threads=self.cores, indices=rows)
        return time.perf_counter() - t0

    def sample(self, budget_s, rng_seed):
        """A seeded leaf sample sized to about budget_s of oracle work."""
        import numpy as np
        n = len(self.script.leaves)
        order = np.random.default_rng(rng_seed).permutation(n).tolist()
        if not hasattr(self, "per_leaf"):
            probe = order[: min(n, max(self.cores, 8))]
            self.per_leaf = self.seconds(probe) / len(probe)
        k = int(min(n, max(min(n, self.cores), budget_s / max(self.per_leaf, 1e-9))))
        return order[:k]


def oracle_rate(script, kv_device, budget_s, rng_seed=0):
    """Leaf-queries/s of the fp64 oracle on a bounded sample of leaves."""
    t = OracleTimer(script, kv_device)
    rows = t.sample(budget_s, rng_seed)
    dt = t.seconds(rows)
    n = len(script.leaves)
    return {"value": len(rows) / dt, "unit": UNIT, "cores": t.cores, "kind": "oracle",
            "sample": f"{len(rows)} of {n} leaves of the same forest, fp64 C oracle (path materialised, naive "
                      f"softmax attention), threads over leaves; {dt:.1f} s", "seconds": dt, "leaves": len(rows)}


def run_reference(args, rank, world):
    """--impl reference: the CPU oracle on the host cores, same metric/config.
    Each step decodes a seeded leaf sample sized so warm-up + steps take a
    few minutes; the rate is sampled leaves / oracle time."""
    if rank != 0:
        return
    script = make_script(args, args.seed)
    desc = describe(script)
    per_step_budget = max(1.0, 150.0 / max(1, args.steps + args.warmup))
    timer = OracleTimer(script, "cpu")
    leaves_done, secs, ks = 0, 0.0, []
    for step in range(args.warmup + args.steps):
        rows = timer.sample(per_step_budget, rng_seed=step)
        dt = timer.seconds(rows)
        if step >= args.warmup:
            leaves_done += len(rows)
            secs += dt
            ks.append(len(rows))
    value = leaves_done / secs
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": desc["leaves"] / value * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": workload_label(script), "leaves": desc["leaves"],
                   "unique_kv_bytes": desc["unique_kv_bytes"]},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": timer.cores, "kind": "oracle",
                         "sample": f"each step: {min(ks)}-{max(ks)} of {desc['leaves']} leaves (seeded sample), "
                                   f"fp64 C oracle, threads over leaves; ms_per_step scaled to all leaves"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# --------------------------------------------------------------------------
# the GPU arm
# --------------------------------------------------------------------------
def main():
    args = parse()
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        run_reference(args, rank, world)
        return

    import torch
    import torch.distributed as dist

    import paper_2508_17445_gb300 as tp
    import workloads
    from paper_2508_17445_gb300 import build as lib_build

    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device(f"cuda:{local}"))
    torch.cuda.set_device(local)
    dev = f"cuda:{local}"
    if rank == 0:
        lib_build.build()
    if world > 1:
        dist.barrier()

    script = make_script(args, shard_seed(args.seed, rank))
    desc = describe(script)
    h = script.heads
    t_setup = time.perf_counter()
    forest = tp.Forest(h.num_q_heads, h.num_kv_heads, h.head_dim,
                       pool_blocks=script.upper_bound_blocks(32) + 64, device=dev)
    ids = forest.replay(script.ops, kv_fn=lambda i: script.kv(i, dev))
    leaves = [ids[x] for x in script.leaves]
    Q = script.q(dev)
    n = len(leaves)
    O = torch.empty((n, h.num_q_heads, h.head_dim), dtype=torch.bfloat16, device=dev)
    LSE = torch.empty((n, h.num_q_heads), dtype=torch.float32, device=dev)
    torch.cuda.synchronize()
    t_setup = time.perf_counter() - t_setup
    stream = torch.cuda.current_stream()

    def steps(k, flags):
        for _ in range(k):
            tp.tp_decode_ex(forest.handle, leaves, Q, O, LSE, flags)

    def timed(k, flags):
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        steps(k, flags)
        b.record(stream)
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()
        return a.elapsed_time(b)

    # ---- warm-up, then the timed region (kernel times recorded live)
    steps(args.warmup, args.flags)
    torch.cuda.synchronize()
    bus = getattr(torch.cuda.get_device_properties(local), "pci_bus_id", None)
    sampler = ClockSampler(bus if isinstance(bus, str) else None)
    sampler.start()
    time.sleep(0.3)
    tp.tp_profile_start(forest.handle)
    ms_total = timed(args.steps, args.flags)
    ktimes = tp.tp_profile_stop(forest.handle)
    clocks = sampler.stop()
    forest.sync()

    # ---- controls: schedule rebuilt every call, and no prefix sharing
    ms_uncached = timed(args.steps, args.flags | tp.TP_DECODE_NO_CACHE)
    steps(2, tp.TP_DECODE_NO_SHARE)
    ms_noshare = timed(args.steps, tp.TP_DECODE_NO_SHARE)
    steps(2, args.flags)

    # ---- end to end through the public API: pinned host Q in, O/LSE out
    Qh = Q.cpu().pin_memory()
    Oh = torch.empty(O.shape, dtype=O.dtype, pin_memory=True)
    Lh = torch.empty(LSE.shape, dtype=LSE.dtype, pin_memory=True)
    Qd = torch.empty_like(Q)

    def e2e_step():
        Qd.copy_(Qh, non_blocking=True)
        tp.tp_decode_ex(forest.handle, leaves, Qd, O, LSE, args.flags)
        Oh.copy_(O, non_blocking=True)
        Lh.copy_(LSE, non_blocking=True)
        stream.synchronize()

    for _ in range(2):
        e2e_step()
    if world > 1:
        dist.barrier()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        e2e_step()
    e2e_s = time.perf_counter() - t0
    forest.sync()

    # ---- max over ranks
    ms_total, ms_uncached, ms_noshare, e2e_s = max_over_ranks([ms_total, ms_uncached, ms_noshare, e2e_s], dev)
    leaves_all = n * world

    if rank == 0:
        ms_step = ms_total / args.steps
        value = job_rate(n, world, args.steps, ms_total)
        peak, peak_kind = peaks()
        dec = ktimes["decode"]
        mer = ktimes["merge"]
        dec_ms = dec["ms"] / max(dec["launches"], 1)
        algo_dec = desc["unique_kv_bytes"] + desc["q_bytes"]
        achieved = algo_dec / (dec_ms / 1e3) / 1e9
        call_bytes = desc["unique_kv_bytes"] + desc["q_bytes"] + desc["o_bytes"] + desc["lse_bytes"]
        call_gbs = call_bytes / (ms_step / 1e3) / 1e9
        traffic = recorded_traffic(args.workload)
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": workload_label(script), "leaves_per_gpu": n, "seed": args.seed,
                       "unique_kv_bytes_per_gpu": desc["unique_kv_bytes"],
                       "no_share_kv_bytes_per_gpu": desc["no_share_kv_bytes"],
                       "l2": f"inputs larger than L2: {desc['unique_kv_bytes'] / 1e9:.2f} GB unique KV read per step "
                             "(L2 129 MB), no flush",
                       "parallelism": f"forest sharded by prompt over {world} GPU(s), no collective",
                       "decode_flags": args.flags},
            "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                         "frac": achieved / peak, "traffic": traffic, "kernel": "decode_kernel",
                         "algorithmic_bytes_per_launch": algo_dec, "launch_ms": dec_ms,
                         "peak_source": f"{peak_kind} hbm_gbs"},
            "call_roofline": {"bytes": call_bytes, "achieved": call_gbs, "frac": call_gbs / peak,
                              "note": "unique KV + Q + O + LSE per tp_decode call / ms_per_step"},
            "kernel_ms_per_step": {"decode": dec_ms, "merge": mer["ms"] / max(mer["launches"], 1)},
            "ms_per_step_schedule_uncached": ms_uncached / args.steps,
            "no_share_ms_per_step": ms_noshare / args.steps,
            "sharing_speedup": ms_noshare / ms_total,
            "e2e": {"value": leaves_all * args.steps / e2e_s, "unit": UNIT,
                    "h2d_bytes_per_step": Q.numel() * Q.element_size(),
                    "d2h_bytes_per_step": O.numel() * O.element_size() + LSE.numel() * LSE.element_size()},
            "gpu_launches": int(dec["launches"] + mer["launches"]),
            "clocks": clocks,
            "setup_s": t_setup,
        }
        if world == 1 and not args.no_cpu_baseline:
            cb = oracle_rate(script, dev, args.cpu_seconds)
            line["cpu_baseline"] = {k: cb[k] for k in ("value", "unit", "cores", "kind", "sample")}
        print(json.dumps(line), flush=True)
    forest.close()
    if world > 1:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
