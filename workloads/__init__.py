"""Seeded synthetic inputs for decode attention over a segment tree of KV caches.

This module only *describes* inputs: the shape of each tree, as a script of
tree operations, and the bf16 Q/K/V tensors those operations carry. It holds
none of the attention arithmetic. Both sides of every parity check replay the
same script: the CUDA library through its C ABI, and the CPU oracle through
its own plain tree model.

Script operations (node ids are script-local, assigned in creation order):

    ("root",   nid)                 new tree with an empty root node
    ("append", nid, kv_id, n)       append n tokens; K/V come from ``kv(kv_id)``
    ("fork",   nid, (c0, c1, ...))  freeze nid and create children c0..ck-1
    ("prune",  nid)                 early-stop: remove leaf nid (and dead ancestors)

The tree shapes follow TreePO's segment-wise sampling (Sec. 2.2, Algorithm 1):
a prompt is the root at depth 0, every later node holds fixed-length segments,
branching forks a path, early stop prunes it. Five named configurations give
the workloads used throughout: ``tiny``, ``qwen7b``, ``random_divergence``,
``wide_prefix`` and ``no_sharing``; ``random_tree`` makes small irregular trees
(ragged blocks, prunes, forks of one) for edge-case tests.

Tensors are i.i.d. N(0, 1) rounded to bf16 (round-to-nearest-even, done by
torch's dtype conversion), drawn from torch generators whose seeds derive from
the workload seed and the tensor's index, so any node can be regenerated alone
on the CPU or on a CUDA device (the two devices give different draws).
"""
from __future__ import annotations

import dataclasses
from typing import Callable, List, Optional, Sequence, Tuple

import numpy as np
import torch

__all__ = [
    "Heads", "Script", "Peaks", "peaked", "root_appends", "last_appends", "tiny", "qwen7b", "random_divergence", "wide_prefix",
    "no_sharing", "random_tree", "single_path", "shared_prompt", "by_name", "CONFIG_NAMES",
]


@dataclasses.dataclass(frozen=True)
class Heads:
    num_q_heads: int
    num_kv_heads: int
    head_dim: int

    @property
    def group(self) -> int:
        return self.num_q_heads // self.num_kv_heads


def _mix(seed: int, stream: int, index: int) -> int:
    # splitmix64-style seed derivation so every tensor has its own generator
    x = (seed * 0x9E3779B97F4A7C15 + stream * 0xBF58476D1CE4E5B9 + index * 0x94D049BB133111EB) & (2**64 - 1)
    x ^= x >> 31
    x = (x * 0xD6E8FEB86645B1A1) & (2**64 - 1)
    x ^= x >> 29
    return x & (2**63 - 1)


@dataclasses.dataclass
class Script:
    """A seeded tree workload: operations, decode leaf set, tensor recipe."""

    name: str
    heads: Heads
    seed: int
    ops: List[tuple]
    leaves: List[int]                 # script node ids decoded, in output order
    kv_len: List[int]                 # tokens carried by each kv_id
    description: str = ""
    shape: Optional["Peaks"] = None   # peaked-score shaping of the draws (None: plain N(0,1))

    # ---- tensors -------------------------------------------------------
    def kv(self, kv_id: int, device="cpu") -> Tuple[torch.Tensor, torch.Tensor]:
        """K, V of append ``kv_id``: bf16 [n][Hkv][hd], i.i.d. N(0,1) (K
        reshaped by ``shape`` when set)."""
        n = self.kv_len[kv_id]
        h = self.heads
        g = torch.Generator(device=device)
        g.manual_seed(_mix(self.seed, 1, kv_id))
        k = torch.randn((n, h.num_kv_heads, h.head_dim), generator=g, device=device, dtype=torch.float32)
        v = torch.randn((n, h.num_kv_heads, h.head_dim), generator=g, device=device, dtype=torch.float32)
        if self.shape is not None:
            k = self.shape.shape_k(k, kv_id)
        return k.to(torch.bfloat16), v.to(torch.bfloat16)

    def q(self, device="cpu", n: Optional[int] = None) -> torch.Tensor:
        """Decode queries: bf16 [len(leaves)][Hq][hd], i.i.d. N(0,1) (reshaped
        by ``shape`` when set)."""
        n = len(self.leaves) if n is None else n
        h = self.heads
        g = torch.Generator(device=device)
        g.manual_seed(_mix(self.seed, 2, 0))
        q = torch.randn((n, h.num_q_heads, h.head_dim), generator=g, device=device, dtype=torch.float32)
        if self.shape is not None:
            q = self.shape.shape_q(q)
        return q.to(torch.bfloat16)

    # ---- structure summaries (no attention arithmetic) ------------------
    def parents(self) -> dict:
        par = {}
        for op in self.ops:
            if op[0] == "root":
                par[op[1]] = -1
            elif op[0] == "fork":
                for c in op[2]:
                    par[c] = op[1]
        return par

    def node_tokens(self) -> dict:
        tok = {}
        for op in self.ops:
            if op[0] == "root":
                tok[op[1]] = 0
            elif op[0] == "fork":
                for c in op[2]:
                    tok[c] = 0
            elif op[0] == "append":
                tok[op[1]] += op[3]
        return tok

    def n_nodes(self) -> int:
        return len(self.parents())

    def upper_bound_blocks(self, block_tokens: int) -> int:
        """Blocks a pool needs if nothing is ever freed (safe pool size)."""
        total = 0
        tok = {}
        for op in self.ops:
            if op[0] == "root":
                tok[op[1]] = 0
            elif op[0] == "fork":
                for c in op[2]:
                    tok[c] = 0
            elif op[0] == "append":
                nid, n = op[1], op[3]
                before = -(-tok[nid] // block_tokens)
                tok[nid] += n
                total += -(-tok[nid] // block_tokens) - before
        return total

    def total_appended_tokens(self) -> int:
        return int(sum(self.kv_len))


@dataclasses.dataclass(frozen=True)
class Peaks:
    """Peaked attention scores, as trained models produce them, from the same
    seeded draws: every element is transformed before the bf16 rounding.

      Q <- q_scale * Q + q_shift
      K <- k_scale * K + (ramp * t / (n - 1) + spike * [t in spikes]) * 1

    with 1 the all-ones vector, t the token index inside its append of n
    tokens. With q_shift > 0 every query has a component along 1, so a ramp
    makes the scores climb along the append (its maximum keeps moving to
    later tokens) and a spike makes one token dominate its path. ``ramp_ids``
    limits the ramp to those appends (None: every append); ``spikes`` maps an
    append to the token indices that carry the spike.
    """

    q_scale: float = 1.0
    k_scale: float = 1.0
    q_shift: float = 0.0
    ramp: float = 0.0
    ramp_ids: Optional[frozenset] = None
    spike: float = 0.0
    spikes: Tuple[Tuple[int, Tuple[int, ...]], ...] = ()

    def shape_q(self, q: torch.Tensor) -> torch.Tensor:
        return q * self.q_scale + self.q_shift

    def shape_k(self, k: torch.Tensor, kv_id: int) -> torch.Tensor:
        k = k * self.k_scale
        n = k.shape[0]
        add = torch.zeros(n, device=k.device, dtype=torch.float32)
        if self.ramp and (self.ramp_ids is None or kv_id in self.ramp_ids):
            add += self.ramp * torch.arange(n, device=k.device, dtype=torch.float32) / max(n - 1, 1)
        for kid, toks in self.spikes:
            if kid == kv_id:
                add[list(toks)] += self.spike
        return k + add[:, None, None]


def peaked(script: Script, shape: Peaks) -> Script:
    """The same workload (same tree, same seeds) with its draws reshaped."""
    return dataclasses.replace(script, shape=shape, name=script.name + "_peaked")


def root_appends(script: Script) -> frozenset:
    """kv_ids appended to root nodes (the prompts, the longest shared prefixes)."""
    roots = {op[1] for op in script.ops if op[0] == "root"}
    return frozenset(op[2] for op in script.ops if op[0] == "append" and op[1] in roots)


def last_appends(script: Script) -> dict:
    """Decoded leaf -> kv_id of the last append on it (the deepest tokens of its path)."""
    last = {}
    for op in script.ops:
        if op[0] == "append":
            last[op[1]] = op[2]
    return {lf: last[lf] for lf in script.leaves if lf in last}


# --------------------------------------------------------------------------
# script builder
# --------------------------------------------------------------------------
class _Builder:
    def __init__(self):
        self.ops: List[tuple] = []
        self.kv_len: List[int] = []
        self.next_id = 0

    def root(self) -> int:
        nid = self.next_id
        self.next_id += 1
        self.ops.append(("root", nid))
        return nid

    def append(self, nid: int, n: int) -> None:
        kv_id = len(self.kv_len)
        self.kv_len.append(int(n))
        self.ops.append(("append", nid, kv_id, int(n)))

    def fork(self, nid: int, k: int) -> List[int]:
        kids = list(range(self.next_id, self.next_id + k))
        self.next_id += k
        self.ops.append(("fork", nid, tuple(kids)))
        return kids

    def prune(self, nid: int) -> None:
        self.ops.append(("prune", nid))


def _full_fork_tree(b: _Builder, root: int, levels: Sequence[Tuple[int, Callable[[], int]]]) -> List[int]:
    """Fork every live leaf by ``k`` then append ``seg()`` tokens, per level."""
    live = [root]
    for k, seg in levels:
        nxt = []
        for nid in live:
            for c in b.fork(nid, k):
                b.append(c, seg())
                nxt.append(c)
        live = nxt
    return live


# --------------------------------------------------------------------------
# the five named workloads
# --------------------------------------------------------------------------
def tiny(seed: int = 0) -> Script:
    """1 layer, 4 query / 1 KV head, head_dim 64; prompt 128, segment 32,
    full binary tree of depth 3 (8 leaves); each leaf's last segment holds
    t ~ U{1..32} tokens and its query attends to all of them."""
    rng = np.random.default_rng(seed)
    b = _Builder()
    r = b.root()
    b.append(r, 128)
    live = [r]
    for depth in (1, 2, 3):
        nxt = []
        for nid in live:
            for c in b.fork(nid, 2):
                n = 32 if depth < 3 else int(rng.integers(1, 33))
                b.append(c, n)
                nxt.append(c)
        live = nxt
    return Script("tiny", Heads(4, 1, 64), seed, b.ops, live, b.kv_len,
                  "tiny binary tree: prompt 128, segment 32, depth 3, ragged last segment")


def qwen7b(seed: int = 0, n_prompts: int = 64, segment: int = 512, depth: int = 4,
           prompt_range: Tuple[int, int] = (256, 1024)) -> Script:
    """Qwen2.5-7B-shaped layer: 28 query / 4 KV heads, head_dim 128; prompts
    of U{256..1024} tokens, segment 512, every node forks into 2 down to depth 4
    (16 leaves per prompt)."""
    rng = np.random.default_rng(seed)
    b = _Builder()
    leaves: List[int] = []
    for _ in range(n_prompts):
        r = b.root()
        b.append(r, int(rng.integers(prompt_range[0], prompt_range[1] + 1)))
        leaves += _full_fork_tree(b, r, [(2, lambda: segment)] * depth)
    return Script("qwen7b", Heads(28, 4, 128), seed, b.ops, leaves, b.kv_len,
                  f"{n_prompts} prompts U{prompt_range}, segment {segment}, binary depth {depth}")


def random_divergence(seed: int = 0, n_prompts: int = 32, prompt: int = 1024, segment: int = 512,
                      depth: int = 14, max_leaves: int = 32, p_stop: float = 0.1,
                      heads: Heads = Heads(28, 4, 128)) -> Script:
    """Seeded random divergence.

    Each prompt is the root (depth 0). At every segment boundary (the prompt's
    included) each live leaf draws k in {1,2,3,4} with probabilities
    0.4/0.3/0.2/0.1, clamped to at least 1 and so that live leaves stay
    <= ``max_leaves`` once the leaves not yet processed are counted; k = 1
    keeps appending to the same node, k > 1 forks. After segments
    1..depth-1 each live leaf first early-stops with probability ``p_stop``
    (pruned, blocks freed); no stop test at the prompt boundary and none
    after the last segment. The leaves alive after segment ``depth`` decode.
    """
    rng = np.random.default_rng(seed)
    b = _Builder()
    leaves: List[int] = []

    def branch(live: List[int]) -> List[int]:
        draws = rng.choice(4, size=len(live), p=[0.4, 0.3, 0.2, 0.1]) + 1
        out: List[int] = []
        for i, (nid, d) in enumerate(zip(live, draws)):
            remaining = len(live) - i - 1
            k = max(1, min(int(d), max_leaves - len(out) - remaining))
            out += [nid] if k == 1 else b.fork(nid, k)
        return out

    for _ in range(n_prompts):
        r = b.root()
        b.append(r, prompt)
        live = branch([r])
        for s in range(1, depth + 1):
            for nid in live:
                b.append(nid, segment)
            if s == depth:
                break
            keep = rng.random(len(live)) >= p_stop
            for nid, kp in zip(live, keep):
                if not kp:
                    b.prune(nid)
            live = [nid for nid, kp in zip(live, keep) if kp]
            if not live:
                break
            live = branch(live)
        leaves += live
    return Script("random_divergence", heads, seed, b.ops, leaves, b.kv_len,
                  f"{n_prompts} prompts of {prompt}, segment {segment}, depth {depth}, "
                  f"fork 1-4 (0.4/0.3/0.2/0.1), cap {max_leaves} leaves, stop p={p_stop}")


def wide_prefix(seed: int = 0, n_prompts: int = 8, prompt: int = 2048, segment: int = 256,
                branch: int = 4, shared_depth: int = 3, private_segments: int = 2) -> Script:
    """64 query / 8 KV heads, head_dim 128; prompts of 2048, segment 256,
    branch factor 4 at depths 1..3 (64 leaves per prompt), then 2 further
    unshared segments appended to every leaf."""
    b = _Builder()
    leaves: List[int] = []
    for _ in range(n_prompts):
        r = b.root()
        b.append(r, prompt)
        live = _full_fork_tree(b, r, [(branch, lambda: segment)] * shared_depth)
        for nid in live:
            for _ in range(private_segments):
                b.append(nid, segment)
        leaves += live
    return Script("wide_prefix", Heads(64, 8, 128), seed, b.ops, leaves, b.kv_len,
                  f"{n_prompts} prompts of {prompt}, segment {segment}, branch {branch} "
                  f"at depths 1..{shared_depth}, {private_segments} private segments per leaf")


def no_sharing(seed: int = 0, n_seqs: int = 256, segments: int = 16, segment: int = 256,
               heads: Heads = Heads(64, 8, 128)) -> Script:
    """No-sharing control: independent single-path trees of ``segments``
    segments of ``segment`` tokens, one decode query each."""
    b = _Builder()
    leaves: List[int] = []
    for _ in range(n_seqs):
        r = b.root()
        for _ in range(segments):
            b.append(r, segment)
        leaves.append(r)
    return Script("no_sharing", heads, seed, b.ops, leaves, b.kv_len,
                  f"{n_seqs} independent paths of {segments}x{segment} tokens")


def single_path(seed: int = 0, lengths: Sequence[int] = (37, 64, 5), heads: Heads = Heads(8, 2, 64),
                fork_chain: bool = True) -> Script:
    """One path of several nodes (fork of 1 between them when ``fork_chain``)."""
    b = _Builder()
    nid = b.root()
    for i, n in enumerate(lengths):
        if i and fork_chain:
            nid = b.fork(nid, 1)[0]
        b.append(nid, n)
    return Script("single_path", heads, seed, b.ops, [nid], b.kv_len, f"single path {list(lengths)}")


def random_tree(seed: int = 0, heads: Heads = Heads(8, 2, 64), n_prompts: int = 3,
                max_depth: int = 4, prompt_range=(1, 90), seg_range=(1, 70), max_kids: int = 3,
                p_prune: float = 0.2, p_fork_one: float = 0.2, p_extra_append: float = 0.3) -> Script:
    """Small irregular forest for edge cases: ragged token counts (blocks
    partly filled mid-path), forks of one, extra appends to leaves, and prunes
    interleaved with growth so freed blocks are reused."""
    rng = np.random.default_rng(seed)
    b = _Builder()
    all_live: List[int] = []
    for _ in range(n_prompts):
        r = b.root()
        b.append(r, int(rng.integers(prompt_range[0], prompt_range[1] + 1)))
        live = [r]
        for _d in range(max_depth):
            nxt = []
            for i, nid in enumerate(live):
                u = rng.random()
                survivors_left = len(nxt) + (len(live) - i - 1)
                if u < p_prune and survivors_left > 0:
                    b.prune(nid)
                    continue
                k = 1 if rng.random() < p_fork_one else int(rng.integers(1, max_kids + 1))
                for c in b.fork(nid, k):
                    b.append(c, int(rng.integers(seg_range[0], seg_range[1] + 1)))
                    if rng.random() < p_extra_append:
                        b.append(c, int(rng.integers(seg_range[0], seg_range[1] + 1)))
                    nxt.append(c)
            live = nxt if nxt else live
        all_live += live
    # decode order: shuffled, with one leaf repeated when possible
    order = list(rng.permutation(len(all_live)))
    leaves = [all_live[i] for i in order]
    if leaves:
        leaves.append(leaves[0])
    return Script("random_tree", heads, seed, b.ops, leaves, b.kv_len, "irregular forest")


def shared_prompt(seed: int = 0, prompt: int = 2000, n_leaves: int = 3, leaf_tokens: Sequence[int] = (40, 7, 90),
                  heads: Heads = Heads(16, 2, 128)) -> Script:
    """One long prompt forked into a few short leaves (long shared node with
    few stacked rows)."""
    b = _Builder()
    r = b.root()
    b.append(r, prompt)
    kids = b.fork(r, n_leaves)
    for c, n in zip(kids, leaf_tokens):
        b.append(c, n)
    return Script("shared_prompt", heads, seed, b.ops, kids, b.kv_len,
                  f"prompt {prompt} shared by {n_leaves} leaves")


def segment_prefill(seed: int = 0, n_prompts: int = 4, prompt_len: int = 1024, fanout: int = 4,
                    seg_len: int = 512, heads: Heads = Heads(28, 4, 128)) -> Script:
    """Prefill shape: each prompt forked into `fanout` leaves that each hold
    a freshly appended segment of `seg_len` tokens (the tokens a prefill
    call processes as queries, Sec. 4.3)."""
    b = _Builder()
    leaves = []
    for _ in range(n_prompts):
        r = b.root()
        b.append(r, prompt_len)
        for c in b.fork(r, fanout):
            b.append(c, seg_len)
            leaves.append(c)
    return Script("segment_prefill", heads, seed, b.ops, leaves, b.kv_len,
                  f"{n_prompts} prompts of {prompt_len} tokens x {fanout} leaves of {seg_len}-token segments")


CONFIG_NAMES = ("tiny", "qwen7b", "random_divergence", "wide_prefix", "no_sharing")


def by_name(name: str, **kw) -> Script:
    return {"tiny": tiny, "qwen7b": qwen7b, "random_divergence": random_divergence,
            "wide_prefix": wide_prefix, "no_sharing": no_sharing}[name](**kw)
