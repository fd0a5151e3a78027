"""Oracle for TreePO's segment-level tree sampling (Sec. 2.2, Algorithm 1),
its branching budget split (Sec. 2.2 budget transfer, Sec. 4.6 probability-
based assignment) and the synthetic stand-in model that drives it.

TEST INFRASTRUCTURE ONLY: imported by ``tests/`` and ``bench.py``'s CPU legs,
never by the product library, and it imports nothing of the product.

Algorithm 1, in the paper's order: P <- Q; P <- Branching(P); while P is not
empty: S <- Inference(P); every segment s_k either goes to the outputs O
(Finish or FailedNode) or back into P as p_k (+) s_k; P <- Branching(P);
P <- Fallback(P, O). The readings where the paper leaves the rule open:

* depth-j budget (Sec. 2.2: N^d until the width w is reached; Sec. 3 "init
  divergence"): the paths of query q at depth j are forked to
  min(b0 * N^j, w - |O_q|) paths, never fewer than one per path;
* FailedNode (repetition early stop) outputs are pruned at once; Finish is
  EOS, a boxed answer or the maximum depth d; only EOS / boxed outputs are
  fallback candidates (Sec. 2.2 footnote);
* Fallback (Sec. 2.2: only when q has no active path and w_q < w): one new
  path forked from a uniformly drawn segment boundary 0 .. J-1 of a
  uniformly drawn live candidate; candidates keep their KV until q is done;
* every decision of the stand-in model is a SplitMix64 draw addressed by
  (tag, node, token, word), so the oracle and the library draw the same
  numbers without sharing code.

Everything is pinned in ``tests/test_oracle_rollout.py``: SplitMix64's
published outputs, hand-computed splits, closed-form tree shapes (full
N-ary trees, all-fail and all-boxed rollouts) and invariants over random
parameters.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from typing import Dict, List, Optional, Sequence, Tuple

import numpy as np

MASK64 = (1 << 64) - 1
GOLDEN_GAMMA = 0x9E3779B97F4A7C15

TAG_K, TAG_V, TAG_Q = 1, 2, 3
TAG_EOS, TAG_TOKEN_LOGP, TAG_SEGMENT, TAG_QUERY = 4, 5, 6, 7
SEG_SCALE, SEG_BOXED, SEG_FAIL, SEG_CORRECT = 0, 1, 2, 3
QUERY_INIT, QUERY_PICK, QUERY_DEPTH = 0, 1, 2

SEG_EOS, SEG_BOXED_BIT, SEG_FAILED, SEG_MAX_DEPTH = 1, 2, 4, 8
EV_ROOT, EV_FORK, EV_SEGMENT, EV_OUTPUT, EV_PRUNE, EV_FALLBACK, EV_DONE = 1, 2, 3, 4, 5, 6, 7
BRANCH_EVEN, BRANCH_LOGP_HIGH, BRANCH_LOGP_LOW = 0, 1, 2


# ------------------------------------------------------------- generator --
def splitmix64(seed: int, i: int) -> int:
    """Element i of the SplitMix64 stream of `seed` (Steele, Lea and Flood,
    OOPSLA 2014): mix(seed + (i + 1) * gamma) in 64-bit arithmetic."""
    z = (seed + (i + 1) * GOLDEN_GAMMA) & MASK64
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & MASK64
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & MASK64
    return z ^ (z >> 31)


def counter(tag: int, a: int, b: int, c: int = 0) -> int:
    return (tag << 60) | ((a & 0xFFFFFFF) << 32) | ((b & 0xFFFFF) << 12) | (c & 0xFFF)


def uniform(seed: int, tag: int, a: int, b: int, c: int = 0) -> float:
    """A draw in [0, 1): the top 53 bits of the counter's element."""
    return (splitmix64(seed, counter(tag, a, b, c)) >> 11) * 2.0 ** -53


def _splitmix64_np(seed: int, ctr: np.ndarray) -> np.ndarray:
    with np.errstate(over="ignore"):
        z = np.uint64(seed) + (ctr + np.uint64(1)) * np.uint64(GOLDEN_GAMMA)
        z = (z ^ (z >> np.uint64(30))) * np.uint64(0xBF58476D1CE4E5B9)
        z = (z ^ (z >> np.uint64(27))) * np.uint64(0x94D049BB133111EB)
    return z ^ (z >> np.uint64(31))


def synth_rows(seed: int, tag: int, nodes: Sequence[int], positions: Sequence[int], heads: int,
               head_dim: int) -> np.ndarray:
    """Stand-in activations: bf16 bit patterns [rows][heads][head_dim] of
    token (nodes[i], positions[i]). Each 64-bit draw gives four values, low
    16 bits first; 16 bits r give sign r[15], exponent 124 + r[7:9] and
    mantissa r[0:7], i.e. values in +-[0.125, 2) -- root mean square about
    0.9, the scale of the unit-normal inputs of the decode workloads."""
    width = heads * head_dim
    words = width // 4
    node = np.asarray(nodes, dtype=np.uint64)[:, None]
    pos = np.asarray(positions, dtype=np.uint64)[:, None]
    w = np.arange(words, dtype=np.uint64)[None, :]
    ctr = (np.uint64(tag) << np.uint64(60)) | ((node & np.uint64(0xFFFFFFF)) << np.uint64(32)) | \
          ((pos & np.uint64(0xFFFFF)) << np.uint64(12)) | w
    h = _splitmix64_np(seed, ctr)                                          # [rows][words]
    lanes = np.stack([(h >> np.uint64(16 * k)) & np.uint64(0xFFFF) for k in range(4)], axis=-1)
    r = lanes.astype(np.uint32)
    bits = (r & 0x8000) | ((124 + ((r >> 7) & 3)) << 7) | (r & 0x7F)
    return bits.astype(np.uint16).reshape(len(nodes), heads, head_dim)


def bf16_to_f64(bits: np.ndarray) -> np.ndarray:
    return (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


# ----------------------------------------------------------- branch split --
def branch_split(logp: Optional[Sequence[float]], n: int, budget: int, policy: int,
                 temperature: float = 1.0) -> List[int]:
    """Split `budget` branches over n active paths, at least one each.

    Even (budget transfer, Sec. 2.2): budget // n each, one more for the
    first budget % n paths. Probability-based (Sec. 4.6): the budget - n
    branches beyond the first are shared in proportion to
    softmax(+-logp / T) (+ favours high log-probability, - low), rounded by
    largest remainder with ties to the lower index. Double precision,
    index order."""
    if n < 0 or budget < n:
        raise ValueError("budget must be at least the number of paths")
    if n == 0:
        return []
    if policy == BRANCH_EVEN:
        return [budget // n + (1 if i < budget % n else 0) for i in range(n)]
    sign = 1.0 if policy == BRANCH_LOGP_HIGH else -1.0
    if policy not in (BRANCH_LOGP_HIGH, BRANCH_LOGP_LOW) or not temperature > 0.0:
        raise ValueError("bad policy or temperature")
    extra = budget - n
    z = [sign * float(x) / temperature for x in logp]
    m = max(z)
    e = [math.exp(x - m) for x in z]
    total = 0.0
    for x in e:
        total += x
    out, frac, used = [], [], 0
    for x in e:
        quota = extra * (x / total)
        whole = math.floor(quota)
        out.append(1 + whole)
        used += whole
        frac.append(quota - whole)
    left = min(max(extra - used, 0), n)
    for i in sorted(range(n), key=lambda i: (-frac[i], i))[:left]:
        out[i] += 1
    return out


# -------------------------------------------------------------- sampler --
@dataclass
class RolloutParams:
    prompt_tokens: Sequence[int]
    width: int = 16
    max_depth: int = 14
    seg_tokens: int = 512
    arity: int = 2
    init_branches: int = 2
    policy: int = BRANCH_EVEN
    fallback: bool = True
    temperature: float = 2.0
    p_eos: float = 0.0
    p_boxed: float = 0.0
    p_fail: float = 0.0
    p_correct: float = 0.5
    seed: int = 0


@dataclass
class Segment:
    tokens: int
    status: int
    logp: float


@dataclass
class Output:
    node: int
    depth: int
    candidate: bool
    reward: int
    alive: bool


@dataclass
class RolloutResult:
    events: List[Tuple[int, ...]]
    parent: Dict[int, int]            # node -> parent (-1 for roots)
    tokens: Dict[int, int]            # node -> tokens it holds
    depth: Dict[int, int]
    query_of: Dict[int, int]
    outputs: List[Tuple[int, Output]] = field(default_factory=list)   # (query, output) in output order

    def path(self, node: int) -> List[int]:
        """Root-first node list of node's root-to-node path."""
        chain = []
        while node != -1:
            chain.append(node)
            node = self.parent[node]
        return chain[::-1]


def draw_segment(p: RolloutParams, node: int, depth: int) -> Segment:
    """Inference of one segment by the stand-in model: token t is EOS if
    u(EOS, node, t) < p_eos; token log-probability kappa * ln(1 - u) with
    kappa = 2 u(SEGMENT, node, SCALE); segment flags from their own draws."""
    n, status = p.seg_tokens, 0
    if p.p_eos > 0.0:
        for t in range(p.seg_tokens):
            if uniform(p.seed, TAG_EOS, node, t) < p.p_eos:
                n, status = t + 1, SEG_EOS
                break
    kappa = 2.0 * uniform(p.seed, TAG_SEGMENT, node, SEG_SCALE)
    acc = 0.0
    for t in range(n):
        acc += kappa * math.log(1.0 - uniform(p.seed, TAG_TOKEN_LOGP, node, t))
    if uniform(p.seed, TAG_SEGMENT, node, SEG_BOXED) < p.p_boxed:
        status |= SEG_BOXED_BIT
    if uniform(p.seed, TAG_SEGMENT, node, SEG_FAIL) < p.p_fail:
        status |= SEG_FAILED
    if depth >= p.max_depth:
        status |= SEG_MAX_DEPTH
    return Segment(n, status, acc / n)


def rollout(p: RolloutParams, first_node: int = 0) -> RolloutResult:
    """Algorithm 1 over a model of the tree (node ids handed out in creation
    order from `first_node`, as the library's tree does)."""
    nq = len(p.prompt_tokens)
    ev: List[Tuple[int, ...]] = []
    res = RolloutResult(ev, {}, {}, {}, {})
    next_id = [first_node]
    alive = set()
    live_children: Dict[int, int] = {}

    def new_node(q: int, parent: int) -> int:
        x = next_id[0]
        next_id[0] += 1
        res.parent[x] = parent
        res.tokens[x] = 0
        res.depth[x] = 0 if parent == -1 else res.depth[parent] + 1
        res.query_of[x] = q
        live_children[x] = 0
        alive.add(x)
        if parent != -1:
            live_children[parent] += 1
        return x

    def fork(q: int, node: int, k: int) -> List[int]:
        kids = [new_node(q, node) for _ in range(k)]
        ev.append((EV_FORK, q, node, kids[0], k, 0, 0, 0))
        return kids

    def prune(q: int, leaf: int) -> None:
        ev.append((EV_PRUNE, q, leaf, 0, 0, 0, 0, 0))
        x = leaf
        while True:                                # the node and its now childless ancestors
            alive.discard(x)
            x = res.parent[x]
            if x == -1:
                break
            live_children[x] -= 1
            if live_children[x] > 0:
                break

    b0: List[int] = []
    outputs: List[List[Output]] = [[] for _ in range(nq)]
    fallbacks = [0] * nq
    done = [False] * nq

    def budget(q: int, depth: int, active: int) -> int:
        b = b0[q]
        for _ in range(depth):
            if b >= p.width:
                break
            b *= p.arity
        return max(min(b, p.width - len(outputs[q])), active)

    def branching(P: List[Tuple[int, int, Optional[float]]]) -> List[Tuple[int, int]]:
        """Fork every path so that its query holds its depth budget of paths."""
        newP = []
        for q in range(nq):
            mine = [(node, lp) for (qq, node, lp) in P if qq == q]
            if not mine:
                continue
            depth = res.depth[mine[0][0]]
            total = budget(q, depth, len(mine))
            if depth == 0:
                split = branch_split(None, len(mine), total, BRANCH_EVEN)
            else:
                split = branch_split([lp for _, lp in mine], len(mine), total, p.policy, p.temperature)
            for (node, _), k in zip(mine, split):
                newP.extend((q, c) for c in fork(q, node, k))
        return newP

    def fallback(P: List[Tuple[int, int]]) -> List[Tuple[int, int]]:
        if not p.fallback:
            return P
        for q in range(nq):
            if done[q] or any(qq == q for qq, _ in P) or len(outputs[q]) >= p.width:
                continue
            cands = [o for o in outputs[q] if o.alive]
            if not cands:
                continue
            c = cands[int(len(cands) * uniform(p.seed, TAG_QUERY, q, QUERY_PICK, fallbacks[q]))]
            j = int(c.depth * uniform(p.seed, TAG_QUERY, q, QUERY_DEPTH, fallbacks[q]))
            at = c.node
            while res.depth[at] > j:
                at = res.parent[at]
            fallbacks[q] += 1
            ev.append((EV_FALLBACK, q, c.node, at, j, 0, 0, 0))
            P = P + [(q, x) for x in fork(q, at, 1)]
        return P

    # P <- Q: one root per query, holding its prompt
    P0 = []
    for q in range(nq):
        r = new_node(q, -1)
        b0.append(p.init_branches if p.init_branches > 0
                  else 2 + int(7.0 * uniform(p.seed, TAG_QUERY, q, QUERY_INIT)))
        ev.append((EV_ROOT, q, r, p.prompt_tokens[q], b0[q], 0, 0, 0))
        res.tokens[r] = p.prompt_tokens[q]
        P0.append((q, r, None))
    P = branching(P0)

    while P:
        S = []
        for (q, node) in P:                           # Inference: one segment per path
            s = draw_segment(p, node, res.depth[node])
            res.tokens[node] = s.tokens
            S.append(s)
        for (q, node), s in zip(P, S):
            logp_bits = int(np.array([s.logp], dtype=np.float64).view(np.int64)[0])
            ev.append((EV_SEGMENT, q, node, res.depth[node], s.tokens, s.status, logp_bits, 0))
        P_last, P_cont = P, []
        for (q, node), s in zip(P_last, S):
            d = res.depth[node]
            if s.status & SEG_FAILED:                  # FailedNode: an output, pruned now
                o = Output(node, d, False, 0, False)
                outputs[q].append(o)
                res.outputs.append((q, o))
                ev.append((EV_OUTPUT, q, node, d, 0, 0, 0, 0))
                prune(q, node)
            elif s.status & (SEG_EOS | SEG_BOXED_BIT | SEG_MAX_DEPTH):   # Finish
                cand = bool(s.status & (SEG_EOS | SEG_BOXED_BIT))
                reward = int(bool(s.status & SEG_BOXED_BIT) and
                             uniform(p.seed, TAG_SEGMENT, node, SEG_CORRECT) < p.p_correct)
                keep = cand and p.fallback
                o = Output(node, d, cand, reward, keep)
                outputs[q].append(o)
                res.outputs.append((q, o))
                ev.append((EV_OUTPUT, q, node, d, int(cand), reward, 0, 0))
                if not keep:
                    prune(q, node)
            else:
                P_cont.append((q, node, s.logp))
        P = branching(P_cont)
        P = fallback(P)
        for q in range(nq):                          # queries with nothing left to sample
            if done[q] or any(qq == q for qq, _ in P):
                continue
            for o in outputs[q]:
                if o.alive:
                    o.alive = False
                    prune(q, o.node)
            done[q] = True
            ev.append((EV_DONE, q, -1, len(outputs[q]), 0, 0, 0, 0))
    return res


def events_array(res: RolloutResult) -> np.ndarray:
    return np.array(res.events, dtype=np.int64).reshape(-1, 8)


def path_kv(res: RolloutResult, seed: int, leaf: int, leaf_tokens: int, kv_heads: int,
            head_dim: int) -> Tuple[np.ndarray, np.ndarray]:
    """bf16 K and V bits [N][kv_heads][head_dim] of leaf's root-to-leaf path
    holding only the first `leaf_tokens` tokens of the leaf itself."""
    nodes, pos = [], []
    chain = res.path(leaf)
    for x in chain:
        n = leaf_tokens if x == leaf else res.tokens[x]
        nodes.extend([x] * n)
        pos.extend(range(n))
    return (synth_rows(seed, TAG_K, nodes, pos, kv_heads, head_dim),
            synth_rows(seed, TAG_V, nodes, pos, kv_heads, head_dim))
