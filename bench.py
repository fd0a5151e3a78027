"""Tree-decode benchmark: leaf-queries/s of libtreepo's tp_decode on GB300.

One step = one tp_decode call over every live leaf of a seeded synthetic
forest shaped like TreePO rollouts (all rows of the hot path: tree-walk
schedule -> split-KV attention over shared path segments -> LSE merge).
Inputs (pool K/V, Q) are resident in HBM when the timed region starts; the
unique KV read per step (>= 1.8 GB for the full workloads) is far larger
than L2 (129 MB), so no flush is needed between steps. The K timed calls
run as a user makes them; the same K calls then run again with every call's
kernels bracketed by CUDA events on the tree's stream, which gives the kernel
durations the roofline divides by (the brackets themselves cost a call a few
microseconds, so the rate comes from the first region).

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
DEFAULT_WORKLOAD = "random_divergence"
FALLBACK_HBM_GBS = 6800.0
FALLBACK_BF16_TFLOPS = 1900.0
FALLBACK_BF16_TFLOPS_SUSTAINED = 1700.0


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=20)
    p.add_argument("--warmup", type=int, default=5)
    p.add_argument("--workload", default=DEFAULT_WORKLOAD,
                   choices=["tiny", "qwen7b", "random_divergence", "wide_prefix", "no_sharing", "rollout", "prefill",
                            "advantage"],
                   help="a decode forest (the default line), or one of the other measured paths: rollout "
                        "(Algorithm 1 with decode after every token), prefill (causal multi-query attention), "
                        "advantage (Eq. tree_ae)")
    p.add_argument("--seed", type=int, default=0)
    p.add_argument("--prompts", type=int, default=None,
                   help="scale the workload down to this many prompts (small cases for ncu captures)")
    p.add_argument("--impl", default="ours", choices=["ours", "reference"])
    p.add_argument("--flags", type=int, default=0, help="tp_decode_ex flags for the timed steps")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-others", action="store_true",
                   help="skip the short measurements of the other workloads that follow the default line")
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


def peaks(key="hbm_gbs"):
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d[key]), "measured"
    except Exception:
        return {"hbm_gbs": FALLBACK_HBM_GBS, "bf16_tflops_sustained": FALLBACK_BF16_TFLOPS_SUSTAINED}.get(
            key, FALLBACK_BF16_TFLOPS), "fallback"


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
        self.window = "sampler started 0.3 s before the timed region, stopped after it"

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
                "samples": len(rows), "window": self.window}


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

    def seconds(self, rows, threads=None):
        self.fetch(rows)
        t0 = time.perf_counter()
        self.model.decode(self.script.leaves, self.q, lambda i: self.cache[i], threads=threads or self.cores,
                          indices=rows)
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
    # the same oracle on one core, over a prefix of the sample worth ~2 s
    rows1 = rows[:max(1, min(len(rows), int(2.0 / max(t.per_leaf * t.cores, 1e-9))))]
    dt1 = t.seconds(rows1, threads=1)
    return {"value": len(rows) / dt, "unit": UNIT, "cores": t.cores, "kind": "oracle",
            "sample": f"{len(rows)} of {n} leaves of the same forest, fp64 C oracle (path materialised, naive "
                      f"softmax attention), threads over leaves; {dt:.1f} s", "seconds": dt, "leaves": len(rows),
            "value_one_core": len(rows1) / dt1, "one_core_sample": f"{len(rows1)} of those leaves, 1 thread, "
                                                                   f"{dt1:.1f} s"}


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
# the other paths: rollout driver, prefill attention, tree advantage
# --------------------------------------------------------------------------
ROLLOUT_SHAPE = dict(n_prompts=64, width=16, max_depth=14, seg_tokens=512, init_branches=2, p_eos=1 / 2048,
                     p_boxed=0.03, p_fail=0.03, p_correct=0.5)


def rollout_prompts(n, seed):
    import numpy as np
    return [int(x) for x in np.random.default_rng(seed).integers(256, 1025, n)]


def rollout_decode_bytes(events, heads):
    """Algorithmic bytes of every decode call of a rollout run with decode on,
    from its events: per call, the unique K/V tokens of the paths still
    generating (their leaf holding t + 1 tokens at token step t) plus their
    query rows."""
    EV_ROOT, EV_FORK, EV_SEGMENT = 1, 2, 3
    parent, tok = {}, {}
    kv_tok = 2 * heads.num_kv_heads * heads.head_dim * 2
    q_row = heads.num_q_heads * heads.head_dim * 2
    total = rows = 0
    i, n = 0, len(events)
    while i < n:
        kind = int(events[i][0])
        if kind == EV_ROOT:
            parent[int(events[i][2])] = -1
            tok[int(events[i][2])] = int(events[i][3])
            i += 1
        elif kind == EV_FORK:
            for c in range(int(events[i][3]), int(events[i][3]) + int(events[i][4])):
                parent[c] = int(events[i][2])
            i += 1
        elif kind == EV_SEGMENT:                     # one loop pass: its whole queue
            seg = []
            while i < n and int(events[i][0]) == EV_SEGMENT:
                seg.append((int(events[i][2]), int(events[i][4])))
                i += 1
            cnt, base = {}, 0
            for node, _ in seg:
                x = parent[node]
                while x != -1:
                    if cnt.get(x, 0) == 0:
                        base += tok[x]
                    cnt[x] = cnt.get(x, 0) + 1
                    x = parent[x]
            alive, t = len(seg), 0
            for node, ln in sorted(seg, key=lambda s: s[1]):
                steps = ln - t                       # token steps t .. ln-1 with this many paths alive
                if steps > 0:
                    leaf_tok = alive * (steps * (t + 1 + ln)) // 2
                    total += (base * steps + leaf_tok) * kv_tok
                    rows += alive * steps
                    t = ln
                alive -= 1
                x = parent[node]
                while x != -1:
                    cnt[x] -= 1
                    if cnt[x] == 0:
                        base -= tok[x]
                    x = parent[x]
            for node, ln in seg:
                tok[node] = ln
        else:
            i += 1
    return total + rows * q_row, rows


LOAD_WINDOW_S = 0.5  # untimed work of the same kind run just before a short timed region


def _clocks_start(load=None, device=0):
    """Start the clock sampler. A timed region of a few milliseconds would see
    no sample of its own (nvidia-smi reports every 100 ms), so `load` -- one
    untimed call of the timed work -- is repeated for about LOAD_WINDOW_S
    seconds first; the calls are left queued, so the GPU runs the same work
    from the sampler's start up to and through the timed region (which
    synchronises before it starts)."""
    import torch
    bus = getattr(torch.cuda.get_device_properties(device), "pci_bus_id", None)
    sampler = ClockSampler(bus if isinstance(bus, str) else None)
    sampler.start()
    if load is None:
        time.sleep(0.3)
        return sampler
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    load()
    torch.cuda.synchronize()
    per_call = max(time.perf_counter() - t0, 1e-5)
    n = min(20000, max(1, int(LOAD_WINDOW_S / per_call)))
    sampler.window = f"{n} untimed calls of the timed work (~{LOAD_WINDOW_S} s) just before the timed region, then the region"
    for _ in range(n):
        load()
    return sampler


def bench_rollout(args):
    """Algorithm 1 at the paper's tree shape (64 prompts, w = 16, 14 x 512
    segments, binary budget) with decode attention after every generated
    token; one step = one whole rollout on the same forest."""
    import torch

    import paper_2508_17445_gb300 as tp
    from paper_2508_17445_gb300 import build as lib_build
    lib_build.build()
    sh = dict(ROLLOUT_SHAPE)
    if args.prompts is not None:
        sh["n_prompts"] = args.prompts
    import workloads
    heads = workloads.Heads(28, 4, 128)
    prompts = rollout_prompts(sh["n_prompts"], args.seed)
    # pool for the largest possible trees: every query's budgeted segments
    segs = sum(min(sh["init_branches"] * 2 ** j, sh["width"]) for j in range(sh["max_depth"]))
    blocks = sum(-(-p // 32) for p in prompts) + sh["n_prompts"] * segs * (-(-sh["seg_tokens"] // 32))
    forest = tp.Forest(heads.num_q_heads, heads.num_kv_heads, heads.head_dim, pool_blocks=blocks + 1024,
                       device="cuda:0")

    def params(step):
        return tp.rollout_params(prompts, width=sh["width"], max_depth=sh["max_depth"], seg_tokens=sh["seg_tokens"],
                                 init_branches=sh["init_branches"], p_eos=sh["p_eos"], p_boxed=sh["p_boxed"],
                                 p_fail=sh["p_fail"], p_correct=sh["p_correct"], seed=args.seed * 1000 + step,
                                 decode=1, decode_flags=args.flags)
    for w in range(args.warmup):
        forest.rollout(params(w))
    forest.sync()
    sampler = _clocks_start()
    t0 = time.perf_counter()
    stats, algo_bytes, rows = [], 0, 0
    for k in range(args.steps):
        ev, st = forest.rollout(params(args.warmup + k))
        stats.append(st)
        b, r = rollout_decode_bytes(ev, heads)
        algo_bytes += b
        rows += r
    forest.sync()
    wall = time.perf_counter() - t0
    # the same rollouts again with every kernel bracketed by CUDA events: the
    # kernel times (the brackets cost each of the thousands of small calls a
    # few microseconds, so the rate comes from the region above)
    tp.tp_profile_start(forest.handle)
    for k in range(args.steps):
        forest.rollout(params(args.warmup + k))
    kt = tp.tp_profile_stop(forest.handle)
    clocks = sampler.stop()
    tokens = sum(st["tokens"] for st in stats)
    trajs = sum(st["outputs"] for st in stats)
    assert rows == sum(st["decode_rows"] for st in stats)
    dec_ms = kt["decode"]["ms"]
    peak, kind = peaks()
    achieved = algo_bytes / (dec_ms / 1e3) / 1e9
    launches = sum(v["launches"] for v in kt.values())
    line = {
        "metric": "tree rollout generated tokens/s (Algorithm 1, decode attention after every token)",
        "value": tokens / wall, "unit": "tokens/s", "n_gpus": 1, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": wall / args.steps * 1e3, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16", "data": "synthetic",
        "config": {"workload": f"rollout: {sh['n_prompts']} prompts (256..1024 tokens), w={sh['width']}, "
                               f"{sh['max_depth']} x {sh['seg_tokens']}-token segments, b0={sh['init_branches']}, "
                               f"binary budget, p_eos={sh['p_eos']:.2g}/token, p_boxed={sh['p_boxed']}, "
                               f"p_fail={sh['p_fail']}; 28 q / 4 kv heads, head_dim 128",
                   "decode_flags": args.flags, "l2": "decode reads up to GBs of path KV per call, no flush"},
        "trajectories_per_s": trajs / wall,
        "decode_calls_per_step": sum(st["decode_calls"] for st in stats) / args.steps,
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s", "frac": achieved / peak,
                     "traffic": None, "kernel": "decode kernels inside the rollout",
                     "algorithmic_bytes_per_step": algo_bytes / args.steps,
                     "peak_source": f"{kind} hbm_gbs"},
        "kernel_ms_per_step": {k: v["ms"] / args.steps for k, v in kt.items()},
        "kernel_times": "CUDA events around every kernel, over a second run of the same rollouts",
        "host_ms_per_step": (wall * 1e3 - sum(v["ms"] for v in kt.values())) / args.steps,
        "e2e": {"value": tokens / wall, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0,
                "note": "the rollout is host-driven end to end: value is already wall-clock through tp_rollout"},
        "gpu_launches": int(launches), "clocks": clocks,
    }
    if not args.no_cpu_baseline:
        line["cpu_baseline"] = rollout_cpu_baseline(prompts, sh, args, heads, min(args.cpu_seconds, 20.0))
    print(json.dumps(line), flush=True)
    forest.close()


def rollout_cpu_baseline(prompts, sh, args, heads, budget_s):
    """The oracle on the host cores: Algorithm 1's decisions for the same
    rollout, plus fp64 path attention for a seeded sample of its decode rows,
    scaled to tokens/s."""
    import numpy as np

    import oracle
    import oracle.rollout as R
    op = R.RolloutParams(prompt_tokens=prompts, width=sh["width"], max_depth=sh["max_depth"],
                         seg_tokens=sh["seg_tokens"], init_branches=sh["init_branches"], p_eos=sh["p_eos"],
                         p_boxed=sh["p_boxed"], p_fail=sh["p_fail"], p_correct=sh["p_correct"], seed=args.seed * 1000)
    t0 = time.perf_counter()
    res = R.rollout(op)
    t_dec = time.perf_counter() - t0
    segs = [e for e in res.events if e[0] == R.EV_SEGMENT]
    tokens = sum(e[4] for e in segs)
    rng = np.random.default_rng(0)
    cores = os.cpu_count() or 1
    done, t_att = 0, 0.0
    while t_att < budget_s * 0.7 and done < 4096:
        e = segs[int(rng.integers(0, len(segs)))]
        node, t = int(e[2]), int(rng.integers(0, e[4]))
        kb, vb = R.path_kv(res, op.seed, node, t + 1, heads.num_kv_heads, heads.head_dim)
        qb = R.synth_rows(op.seed, R.TAG_Q, [node], [t], heads.num_q_heads, heads.head_dim)[0]
        t1 = time.perf_counter()
        oracle.path_attention(qb, kb, vb)
        t_att += time.perf_counter() - t1
        done += 1
    per_row = t_att / done
    total = t_dec + tokens * per_row
    return {"value": tokens / total, "unit": "tokens/s", "cores": 1, "kind": "oracle",
            "sample": f"oracle Algorithm 1 over the whole rollout ({t_dec:.1f} s) + fp64 path attention for "
                      f"{done} sampled (leaf, token) decode rows ({per_row * 1e3:.2f} ms each), scaled to its "
                      f"{tokens} generated tokens; single thread"}


PREFILL_SHAPE = (16, 1024, 512)  # leaves per prompt, prompt tokens, segment tokens (all queries)


def prefill_setup(seed, n_prompts):
    """The segment-prefill forest on cuda:0, its query tensors and its flops."""
    import torch

    import paper_2508_17445_gb300 as tp
    import workloads
    fan, plen, seg = PREFILL_SHAPE
    script = workloads.segment_prefill(seed=seed, n_prompts=n_prompts, prompt_len=plen, fanout=fan, seg_len=seg)
    h = script.heads
    forest = tp.Forest(h.num_q_heads, h.num_kv_heads, h.head_dim, pool_blocks=script.upper_bound_blocks(32) + 64,
                       device="cuda:0")
    ids = forest.replay(script.ops, kv_fn=lambda i: script.kv(i, "cuda:0"))
    nodes = [ids[x] for x in script.leaves]
    counts = [seg] * len(nodes)
    total = sum(counts)
    g = torch.Generator(device="cpu").manual_seed(seed)
    Q = torch.randn(total, h.num_q_heads, h.head_dim, generator=g).to(torch.bfloat16).to("cuda:0")
    O = torch.empty_like(Q)
    L = torch.empty(total, h.num_q_heads, dtype=torch.float32, device="cuda:0")
    flops = 4 * h.head_dim * h.num_q_heads * len(nodes) * sum(plen + j + 1 for j in range(seg))
    return script, forest, nodes, counts, Q, O, L, flops


def bench_prefill(args):
    """Causal multi-query attention over tree paths: 64 prompts of 1024
    tokens, each forked into 16 leaves holding a 512-token segment; one step
    = one tp_prefill over every leaf's whole segment (524288 query tokens)."""
    import torch

    import paper_2508_17445_gb300 as tp
    import workloads
    from paper_2508_17445_gb300 import build as lib_build
    lib_build.build()
    n_prompts = args.prompts or 64
    fan, plen, seg = PREFILL_SHAPE
    script, forest, nodes, counts, Q, O, L, flops = prefill_setup(args.seed, n_prompts)
    total = sum(counts)
    for _ in range(args.warmup):
        tp.tp_prefill(forest.handle, nodes, counts, Q, O, L, args.flags)
    torch.cuda.synchronize()
    stream = torch.cuda.current_stream()
    sampler = _clocks_start(lambda: tp.tp_prefill(forest.handle, nodes, counts, Q, O, L, args.flags))
    torch.cuda.synchronize()
    tp.tp_profile_start(forest.handle)
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(stream)
    for _ in range(args.steps):
        tp.tp_prefill(forest.handle, nodes, counts, Q, O, L, args.flags)
    b.record(stream)
    torch.cuda.synchronize()
    ms = a.elapsed_time(b) / args.steps
    kt = tp.tp_profile_stop(forest.handle)
    clocks = sampler.stop()
    forest.sync()
    dec_ms = kt["decode"]["ms"] / args.steps  # one attention bracket per call (its kernels run together)
    # the region runs after LOAD_WINDOW_S of the same dense work, where the
    # 1.4 kW cap holds the clocks: the sustained GEMM figure is the peak
    peak, kind = peaks("bf16_tflops_sustained")
    burst, _ = peaks("bf16_tflops")
    achieved = flops / (dec_ms / 1e3) / 1e12
    # end to end through the host-buffer call: pinned host Q in, O and LSE
    # back, every step; calls back to back (the library overlaps a call's
    # copies with its neighbours' attention), then one tp_sync
    Qh, Oh = Q.cpu().pin_memory(), torch.empty(O.shape, dtype=O.dtype, pin_memory=True)
    Lh = torch.empty(L.shape, dtype=L.dtype, pin_memory=True)
    tp.tp_prefill_host(forest.handle, nodes, counts, Qh, Oh, Lh, args.flags)
    forest.sync()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        tp.tp_prefill_host(forest.handle, nodes, counts, Qh, Oh, Lh, args.flags)
    forest.sync()
    e2e_s = (time.perf_counter() - t0) / args.steps
    t0 = time.perf_counter()
    for _ in range(args.steps):  # the same with a wait after every call
        tp.tp_prefill_host(forest.handle, nodes, counts, Qh, Oh, Lh, args.flags)
        forest.sync()
    e2e_sync_s = (time.perf_counter() - t0) / args.steps
    line = {
        "metric": "tree prefill query tokens/s (causal multi-query attention over root-to-node paths); "
                  "TFLOP/s vs GB300 bf16 peak",
        "value": total / (ms / 1e3), "unit": "query-tokens/s", "n_gpus": 1, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16", "data": "synthetic",
        "config": {"workload": f"segment_prefill: {n_prompts} prompts of {plen} tokens x {fan} leaves, each leaf's "
                               f"{seg}-token segment as causal queries ({total} query tokens); 28 q / 4 kv heads, "
                               f"head_dim 128",
                   "flags": args.flags, "l2": "K/V re-read from L2 by the query blocks of a path; no flush"},
        "tflops_call": flops / (ms / 1e3) / 1e12,
        "roofline": {"bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                     "frac": achieved / peak, "traffic": None, "kernel": "decode_tc_kernel (causal)",
                     "algorithmic_flops_per_launch": flops, "launch_ms": dec_ms,
                     "peak_source": f"{kind} bf16_tflops_sustained (timed after {LOAD_WINDOW_S} s of the same load)",
                     "frac_of_burst_peak": achieved / burst},
        "kernel_ms_per_step": {"attention": dec_ms, "merge": kt["merge"]["ms"] / args.steps},
        "e2e": {"value": total / e2e_s, "unit": "query-tokens/s", "h2d_bytes_per_step": Q.numel() * 2,
                "d2h_bytes_per_step": O.numel() * 2 + L.numel() * 4,
                "call": "tp_prefill_host, calls back to back then tp_sync",
                "value_wait_each_call": total / e2e_sync_s},
        "gpu_launches": int(kt["decode"]["launches"] + kt["merge"]["launches"]), "clocks": clocks,
    }
    if not args.no_cpu_baseline:
        line["cpu_baseline"] = prefill_cpu_baseline(script, counts, Q, min(args.cpu_seconds, 20.0))
    print(json.dumps(line), flush=True)
    forest.close()


def prefill_cpu_baseline(script, counts, Q, budget_s):
    import numpy as np

    import oracle
    model = oracle.OracleForest(block_tokens=32, pool_blocks=script.upper_bound_blocks(32) + 64).replay(script)
    cache = {}

    def src(i):
        if i not in cache:
            k, v = script.kv(i, "cpu")
            cache[i] = (oracle.bf16_bits(k), oracle.bf16_bits(v))
        return cache[i]
    total = sum(counts)
    rng = np.random.default_rng(0)
    cores = os.cpu_count() or 1
    rows = sorted(set(int(x) for x in rng.integers(0, total, cores * 4)))
    qc = Q.cpu()
    model.prefill(list(script.leaves), counts, qc, src, indices=rows[:cores])   # materialise the paths
    t0 = time.perf_counter()
    model.prefill(list(script.leaves), counts, qc, src, indices=rows, threads=cores)
    dt = time.perf_counter() - t0
    n = len(rows)
    while dt < budget_s / 4 and n < total:
        more = sorted(set(int(x) for x in rng.integers(0, total, n)))
        t0 = time.perf_counter()
        model.prefill(list(script.leaves), counts, qc, src, indices=more, threads=cores)
        dt += time.perf_counter() - t0
        n += len(more)
    return {"value": n / dt, "unit": "query-tokens/s", "cores": cores, "kind": "oracle",
            "sample": f"{n} seeded query rows of the same call, fp64 C oracle over each row's causal path prefix, "
                      f"threads over rows; {dt:.1f} s"}


def bench_advantage(args):
    """Eq. tree_ae over the output trees of a paper-shaped rollout batch
    (64 prompts, w = 16): one step = one tp_tree_advantage call."""
    import numpy as np
    import torch

    import paper_2508_17445_gb300 as tp
    from paper_2508_17445_gb300 import build as lib_build
    lib_build.build()
    sh = dict(ROLLOUT_SHAPE)
    n_prompts = args.prompts or sh["n_prompts"]
    prompts = rollout_prompts(n_prompts, args.seed)
    dry = tp.Forest(28, 4, 128, pool_blocks=1 << 22, device=None)
    ev, st = dry.rollout(tp.rollout_params(prompts, width=sh["width"], max_depth=sh["max_depth"],
                                           seg_tokens=sh["seg_tokens"], init_branches=sh["init_branches"],
                                           p_eos=sh["p_eos"], p_boxed=0.1, p_fail=sh["p_fail"], p_correct=0.5,
                                           seed=args.seed))
    n_nodes = int(st["nodes"])
    parent = [dry.node_info(x)["parent"] for x in range(n_nodes)]
    outs = ev[ev[:, 0] == 4]
    leaves = outs[:, 2].astype(np.int32)
    rewards = outs[:, 5].astype(np.float32)
    dev = "cuda:0"
    P = torch.tensor(parent, dtype=torch.int32, device=dev)
    Lf = torch.tensor(leaves, dtype=torch.int32, device=dev)
    Rw = torch.tensor(rewards, dtype=torch.float32, device=dev)
    adv = torch.empty(len(leaves), dtype=torch.float32, device=dev)
    stats = torch.zeros(4, dtype=torch.float64, device=dev)
    ws = torch.empty(max(tp.tp_advantage_workspace_bytes(n_nodes, len(leaves)), 8), dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream()
    for _ in range(args.warmup):
        tp.tp_tree_advantage(P, Lf, Rw, adv, stats, ws, stream.cuda_stream)
    torch.cuda.synchronize()
    sampler = _clocks_start(lambda: tp.tp_tree_advantage(P, Lf, Rw, adv, stats, ws, stream.cuda_stream))
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(stream)
    for _ in range(args.steps):
        tp.tp_tree_advantage(P, Lf, Rw, adv, stats, ws, stream.cuda_stream)
    b.record(stream)
    torch.cuda.synchronize()
    ms = a.elapsed_time(b) / args.steps
    clocks = sampler.stop()
    depth = float(np.mean(outs[:, 3]))
    algo = 4 * n_nodes + 12 * len(leaves) + 4 * int(len(leaves) * depth) * 2
    peak, kind = peaks()
    Lh, Rh = Lf.cpu().pin_memory(), Rw.cpu().pin_memory()
    Ah = torch.empty(adv.shape, dtype=adv.dtype, pin_memory=True)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        Lf.copy_(Lh, non_blocking=True)
        Rw.copy_(Rh, non_blocking=True)
        tp.tp_tree_advantage(P, Lf, Rw, adv, stats, ws, stream.cuda_stream)
        Ah.copy_(adv, non_blocking=True)
        stream.synchronize()
    e2e_s = (time.perf_counter() - t0) / args.steps
    line = {
        "metric": "tree advantage trajectories/s (Eq. tree_ae: sub-group means over the node table, "
                  "mean pooling, global std)",
        "value": len(leaves) / (ms / 1e3), "unit": "trajectories/s", "n_gpus": 1, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "f64 accumulation, f32 out", "data": "synthetic",
        "config": {"workload": f"output trees of a {n_prompts}-prompt rollout batch (w=16, 14 x 512): "
                               f"{len(leaves)} trajectories, {n_nodes} nodes, mean depth {depth:.1f}"},
        "roofline": {"bound": "hbm", "achieved": algo / (ms / 1e3) / 1e9, "peak": peak, "unit": "GB/s",
                     "frac": algo / (ms / 1e3) / 1e9 / peak, "traffic": None,
                     "kernel": "advantage_{init,walk,means,abar}_kernel",
                     "note": "four small launches (fp64 sub-group sums, means, pooled A_i, normalisation); a few "
                             "hundred KB per call: launch- and latency-bound, not bandwidth-bound",
                     "peak_source": f"{kind} hbm_gbs"},
        "e2e": {"value": len(leaves) / e2e_s, "unit": "trajectories/s", "h2d_bytes_per_step": 8 * len(leaves),
                "d2h_bytes_per_step": 4 * len(leaves)},
        "gpu_launches": 4 * args.steps, "clocks": clocks,
    }
    if not args.no_cpu_baseline:
        import oracle.advantage as OA
        t0 = time.perf_counter()
        k = 0
        while time.perf_counter() - t0 < min(args.cpu_seconds, 5.0) or k == 0:
            OA.tree_advantage(parent, leaves.tolist(), rewards.astype(np.float64).tolist())
            k += 1
        dt = (time.perf_counter() - t0) / k
        line["cpu_baseline"] = {"value": len(leaves) / dt, "unit": "trajectories/s", "cores": 1, "kind": "oracle",
                                "sample": f"the whole call, {k} repetitions, fp64 Python loops, single thread"}
    print(json.dumps(line), flush=True)


# --------------------------------------------------------------------------
# the GPU arm
# --------------------------------------------------------------------------
OTHER_DECODE = ("tiny", "qwen7b", "wide_prefix", "no_sharing")


def other_workloads(dev, steps, warmup):
    """Short measurements of the other workloads, after the default line's
    and on the same GPU, so that one run records every configuration: each
    other decode forest (leaf-queries/s over `steps` calls timed like the
    default line's, its attention kernels' and whole call's fractions of the
    measured copy peak, the no-share speedup) and the prefill path at full
    size (query tokens/s; TFLOP/s of its attention kernels). Clocks are
    sampled for the default line only."""
    import torch

    import paper_2508_17445_gb300 as tp
    import workloads
    peak, _ = peaks()
    stream = torch.cuda.current_stream()

    def timed(fn):
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        fn()
        b.record(stream)
        torch.cuda.synchronize()
        return a.elapsed_time(b)

    out = {"note": f"each: {warmup} warm-up calls, then {steps} timed calls (CUDA events); attention kernel times "
                   "from a second run of the same calls with event brackets"}
    for name in OTHER_DECODE:
        script = workloads.by_name(name, seed=0)
        desc = describe(script)
        h = script.heads
        forest = tp.Forest(h.num_q_heads, h.num_kv_heads, h.head_dim,
                           pool_blocks=script.upper_bound_blocks(32) + 64, device=dev)
        ids = forest.replay(script.ops, kv_fn=lambda i, s=script: s.kv(i, dev))
        leaves = [ids[x] for x in script.leaves]
        Q = script.q(dev)
        O = torch.empty((len(leaves), h.num_q_heads, h.head_dim), dtype=torch.bfloat16, device=dev)
        L = torch.empty((len(leaves), h.num_q_heads), dtype=torch.float32, device=dev)

        def run(k, flags=0):
            for _ in range(k):
                tp.tp_decode_ex(forest.handle, leaves, Q, O, L, flags)
        run(warmup)
        ms = timed(lambda: run(steps)) / steps
        tp.tp_profile_start(forest.handle)
        timed(lambda: run(steps))
        kt = tp.tp_profile_stop(forest.handle)
        run(2, tp.TP_DECODE_NO_SHARE)
        ms_noshare = timed(lambda: run(steps, tp.TP_DECODE_NO_SHARE)) / steps
        forest.sync()
        forest.close()
        algo = desc["unique_kv_bytes"] + desc["q_bytes"]
        call = algo + desc["o_bytes"] + desc["lse_bytes"]
        dec_ms = kt["decode"]["ms"] / steps
        out[name] = {"value": len(leaves) / (ms / 1e3), "unit": UNIT, "ms_per_step": ms,
                     "attention_frac_of_hbm": algo / (dec_ms / 1e3) / 1e9 / peak,
                     "call_frac_of_hbm": call / (ms / 1e3) / 1e9 / peak,
                     "sharing_speedup": ms_noshare / ms, "workload": workload_label(script)}
        del Q, O, L
        torch.cuda.empty_cache()
    script, forest, nodes, counts, Q, O, L, flops = prefill_setup(0, 64)
    for _ in range(warmup):
        tp.tp_prefill(forest.handle, nodes, counts, Q, O, L, 0)
    k = max(1, min(steps, 5))
    ms = timed(lambda: [tp.tp_prefill(forest.handle, nodes, counts, Q, O, L, 0) for _ in range(k)]) / k
    tp.tp_profile_start(forest.handle)
    timed(lambda: [tp.tp_prefill(forest.handle, nodes, counts, Q, O, L, 0) for _ in range(k)])
    kt = tp.tp_profile_stop(forest.handle)
    forest.sync()
    forest.close()
    att_ms = kt["decode"]["ms"] / k
    out["prefill"] = {"value": sum(counts) / (ms / 1e3), "unit": "query-tokens/s", "ms_per_step": ms,
                      "attention_tflops": flops / (att_ms / 1e3) / 1e12,
                      "frac_of_sustained_bf16": flops / (att_ms / 1e3) / 1e12 / peaks("bf16_tflops_sustained")[0],
                      "workload": "segment_prefill: 64 prompts of 1024 tokens x 16 leaves, 512-token segments as "
                                  "causal queries"}
    del Q, O, L
    torch.cuda.empty_cache()
    return out


def main():
    args = parse()
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if args.workload in ("rollout", "prefill", "advantage"):
        if rank == 0:     # single-GPU measurements of the other paths; other ranks have no work
            {"rollout": bench_rollout, "prefill": bench_prefill, "advantage": bench_advantage}[args.workload](args)
        return
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

    # ---- warm-up, then the timed region: K calls as a user makes them
    steps(args.warmup, args.flags)
    torch.cuda.synchronize()
    sampler = _clocks_start(lambda: steps(1, args.flags), device=local)
    ms_total = timed(args.steps, args.flags)
    # ---- the same K calls with each call's kernels bracketed by CUDA events
    # on the tree's stream (its attention kernels together, the merge alone):
    # the kernel durations the roofline divides by, measured live. The
    # brackets cost a call a few microseconds, so `value` comes from the
    # region above, not from this one.
    tp.tp_profile_start(forest.handle)
    ms_profiled = timed(args.steps, args.flags)
    ktimes = tp.tp_profile_stop(forest.handle)
    clocks = sampler.stop()
    forest.sync()

    # ---- controls, timed like the first region: schedule rebuilt every
    # call, and no prefix sharing
    ms_uncached = timed(args.steps, args.flags | tp.TP_DECODE_NO_CACHE)
    steps(2, tp.TP_DECODE_NO_SHARE)
    ms_noshare = timed(args.steps, tp.TP_DECODE_NO_SHARE)
    steps(2, args.flags)

    # ---- end to end through the host-buffer call: pinned host Q in, O and
    # LSE back, every step; calls back to back (the library overlaps a call's
    # copies with its neighbours' attention), then one tp_sync
    Qh = Q.cpu().pin_memory()
    Oh = torch.empty(O.shape, dtype=O.dtype, pin_memory=True)
    Lh = torch.empty(LSE.shape, dtype=LSE.dtype, pin_memory=True)
    for _ in range(2):
        tp.tp_decode_host(forest.handle, leaves, Qh, Oh, Lh, args.flags)
    forest.sync()
    if world > 1:
        dist.barrier()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        tp.tp_decode_host(forest.handle, leaves, Qh, Oh, Lh, args.flags)
    forest.sync()
    e2e_s = time.perf_counter() - t0
    t0 = time.perf_counter()
    for _ in range(args.steps):  # the same with a wait after every call
        tp.tp_decode_host(forest.handle, leaves, Qh, Oh, Lh, args.flags)
        forest.sync()
    e2e_sync_s = time.perf_counter() - t0

    # ---- max over ranks
    ms_total, ms_profiled, ms_uncached, ms_noshare, e2e_s, e2e_sync_s = max_over_ranks(
        [ms_total, ms_profiled, ms_uncached, ms_noshare, e2e_s, e2e_sync_s], dev)
    leaves_all = n * world

    if rank == 0:
        ms_step = ms_total / args.steps
        value = job_rate(n, world, args.steps, ms_total)
        peak, peak_kind = peaks()
        dec = ktimes["decode"]
        mer = ktimes["merge"]
        dec_ms = dec["ms"] / args.steps  # one bracket per call around its concurrent attention kernels
        assert dec["launches"] > 0 and dec_ms * args.steps <= ms_profiled * 1.001
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
                         "measured": "CUDA events around each call's attention kernels on the tree's stream, over "
                                     "a second timed region of the same K calls",
                         "peak_source": f"{peak_kind} hbm_gbs"},
            "call_roofline": {"bytes": call_bytes, "achieved": call_gbs, "frac": call_gbs / peak,
                              "note": "unique KV + Q + O + LSE per tp_decode call / ms_per_step"},
            "kernel_ms_per_step": {"decode": dec_ms, "merge": mer["ms"] / args.steps},
            "ms_per_step_profiled": ms_profiled / args.steps,
            "ms_per_step_schedule_uncached": ms_uncached / args.steps,
            "no_share_ms_per_step": ms_noshare / args.steps,
            "sharing_speedup": ms_noshare / ms_total,
            "e2e": {"value": leaves_all * args.steps / e2e_s, "unit": UNIT,
                    "h2d_bytes_per_step": Q.numel() * Q.element_size(),
                    "d2h_bytes_per_step": O.numel() * O.element_size() + LSE.numel() * LSE.element_size(),
                    "call": "tp_decode_host, calls back to back then tp_sync",
                    "value_wait_each_call": leaves_all * args.steps / e2e_sync_s},
            "gpu_launches": int(dec["launches"] + mer["launches"]),
            "clocks": clocks,
            "setup_s": t_setup,
        }
        if world == 1 and not args.no_cpu_baseline:
            cb = oracle_rate(script, dev, args.cpu_seconds)
            line["cpu_baseline"] = {k: cb[k] for k in ("value", "unit", "cores", "kind", "sample", "value_one_core",
                                                       "one_core_sample")}
    forest.close()
    if rank == 0:
        if (world == 1 and not args.no_others and args.workload == DEFAULT_WORKLOAD and args.prompts is None
                and args.flags == 0):
            del Q, O, LSE
            torch.cuda.empty_cache()
            try:  # extra records: a failure here must not cost the default line
                line["other_workloads"] = other_workloads(dev, min(args.steps, 10), max(args.warmup, 3))
            except Exception as e:  # noqa: BLE001
                line["other_workloads"] = {"error": f"{type(e).__name__}: {e}"[:300]}
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
