"""CPU oracle for decode attention over a segment tree of KV caches.

TEST INFRASTRUCTURE ONLY. Only ``tests/``, ``__graft_entry__.smoke()`` and
``bench.py`` (its CPU-baseline leg and ``--impl reference``) may import this
package. The product library never loads it, and this package never imports
the product: the two share nothing but the seeded input generators in
``workloads``.

Contents
--------
``path_attention``   fp64 softmax attention of one query over one
                     materialised path (``attention.c``; definition in its
                     header). TreePO's trajectory is s_1 (+) ... (+) s_j
                     (Sec. 2.3) and a decode step attends to all of it.
``path_scores``      the fp64 scores q.k / sqrt(d) that softmax runs over
                     (for tests that locate a path's score maximum).
``lse_merge``        fp64 log-sum-exp merge of attention partials over
                     disjoint token sets (a split of the path).
``OracleForest``     plain tree model: replays a workload script (root,
                     append, fork, prune; Sec. 2.2, Algorithm 1), keeps each
                     node's tokens, models the paged pool (fixed-size blocks
                     handed out lowest index first, freed on prune) and
                     materialises each leaf's root-to-leaf path; ``decode``
                     and the causal multi-query ``prefill`` (each query sees
                     its path up to and including itself) run
                     ``path_attention`` on those paths.

Every function here is pinned by ``tests/test_oracle.py`` against values that
do not come from this code: a hand-computed two-token example, closed forms,
torch's own SDPA in fp64, brute-force path construction and a hand-computed
block-allocation example (``tests/golden/``).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading
from concurrent.futures import ThreadPoolExecutor
from typing import Callable, Dict, List, Optional, Sequence, Tuple

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "attention.c")
_LIB_PATH = os.path.join(_HERE, "_oracle_attention.so")
_lib = None
_lib_lock = threading.Lock()


def build(force: bool = False) -> str:
    """Compile ``attention.c`` with the host C compiler (plain -O2)."""
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".{os.getpid()}.tmp"
        subprocess.check_call(["gcc", "-O2", "-std=c99", "-fPIC", "-shared", _SRC, "-o", tmp, "-lm"])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lib_lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            f = lib.oracle_path_attention
            f.restype = ctypes.c_int
            f.argtypes = [ctypes.c_int64, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32,
                          ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p,
                          ctypes.c_void_p, ctypes.c_void_p]
            _lib = lib
    return _lib


def bf16_bits(x) -> np.ndarray:
    """bf16 tensor (torch) or uint16 array -> contiguous uint16 numpy array."""
    if isinstance(x, np.ndarray):
        assert x.dtype == np.uint16
        return np.ascontiguousarray(x)
    import torch
    assert x.dtype == torch.bfloat16, x.dtype
    return x.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)


def path_attention(q, k, v) -> Tuple[np.ndarray, np.ndarray]:
    """fp64 attention of one decode query over one materialised path.

    q: [Hq][d] bf16; k, v: [N][Hkv][d] bf16 (root first). Returns
    (O [Hq][d] fp64, LSE [Hq] fp64, natural log).
    """
    qb, kb, vb = bf16_bits(q), bf16_bits(k), bf16_bits(v)
    hq, d = qb.shape
    n, hkv, d2 = kb.shape
    assert d2 == d and vb.shape == kb.shape
    out = np.empty((hq, d), dtype=np.float64)
    lse = np.empty((hq,), dtype=np.float64)
    rc = _load().oracle_path_attention(n, hq, hkv, d, qb.ctypes.data, kb.ctypes.data, vb.ctypes.data,
                                       out.ctypes.data, lse.ctypes.data)
    if rc != 0:
        raise ValueError(f"oracle_path_attention rejected its arguments (N={n}, Hq={hq}, Hkv={hkv}, d={d})")
    return out, lse


def path_scores(q, k) -> np.ndarray:
    """fp64 attention scores of one decode query over one materialised path.

    q: [Hq][d] bf16; k: [N][Hkv][d] bf16 (root first). Returns s [Hq][N] with
    s[h][j] = (q_h . k_{j, h // g}) / sqrt(d), g = Hq / Hkv: the scores whose
    softmax ``path_attention`` takes (step 4 of the definition in
    ``attention.c``), so LSE = ln sum_j exp(s[h][j]). The tests read them to
    show where a path's score maximum lies.
    """
    qb, kb = bf16_bits(q), bf16_bits(k)
    q64 = (qb.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    k64 = (kb.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    hq, d = q64.shape
    n, hkv, d2 = k64.shape
    assert d2 == d and hq % hkv == 0
    g = hq // hkv
    s = np.empty((hq, n), dtype=np.float64)
    for h in range(hq):
        s[h] = k64[:, h // g, :] @ q64[h]
    return s / np.sqrt(d)


def lse_merge(parts: Sequence[Tuple[np.ndarray, np.ndarray]]) -> Tuple[np.ndarray, np.ndarray]:
    """Merge attention results over disjoint token sets of one path.

    Each part i is (O_i [H][d], LSE_i [H]) for the same queries over its own
    tokens. With LSE = ln sum_i exp(LSE_i) the merged output is
    O = sum_i exp(LSE_i - LSE) O_i -- the softmax over the union, written
    through the parts' normalisers.
    """
    lses = np.stack([p[1] for p in parts])                  # [P][H]
    m = lses.max(axis=0)
    w = np.exp(lses - m[None, :])                           # [P][H]
    total = w.sum(axis=0)
    lse = m + np.log(total)
    out = np.zeros_like(parts[0][0])
    for (o_i, _), w_i in zip(parts, w):
        out += (w_i / total)[:, None] * o_i
    return out, lse


class OracleError(Exception):
    """A tree operation the model rejects (mirrors the C ABI's error codes)."""

    def __init__(self, code: str, msg: str = ""):
        super().__init__(f"{code}: {msg}")
        self.code = code


class _Node:
    __slots__ = ("parent", "kids_live", "chunks", "n_tokens", "blocks", "state")

    def __init__(self, parent: int):
        self.parent = parent
        self.kids_live = 0
        self.chunks: List[int] = []       # kv_ids appended, in order
        self.n_tokens = 0
        self.blocks: List[int] = []
        self.state = "leaf"               # leaf | frozen | dead


class OracleForest:
    """Plain model of a forest of segment trees over a paged KV pool.

    Pool model: ``pool_blocks`` blocks of ``block_tokens`` token slots. An
    append first fills the node's partly used last block, then takes new
    blocks, lowest free index first, in ascending order; a failed allocation
    changes nothing. Token t of a node lives in slot
    ``blocks[t // BT] * BT + t % BT``. Forking freezes the node and gives it
    k empty children (no tokens move); pruning a leaf frees its blocks and
    those of every ancestor whose last live child it was.
    """

    def __init__(self, block_tokens: int = 32, pool_blocks: int = 1 << 20):
        self.bt = block_tokens
        self.pool_blocks = pool_blocks
        self.free = np.ones(pool_blocks, dtype=bool)
        self.nodes: Dict[int, _Node] = {}
        self.kv_len: Dict[int, int] = {}

    # ---- pool ---------------------------------------------------------------
    def _alloc(self, count: int) -> List[int]:
        ids = np.flatnonzero(self.free)[:count]
        if len(ids) < count:
            raise OracleError("OOM", f"need {count} blocks, {int(self.free.sum())} free")
        self.free[ids] = False
        return [int(i) for i in ids]

    def _release(self, node: _Node) -> None:
        for blk in node.blocks:
            assert not self.free[blk]
            self.free[blk] = True
        node.blocks = []
        node.state = "dead"

    # ---- operations ---------------------------------------------------------
    def _live(self, nid: int) -> _Node:
        node = self.nodes.get(nid)
        if node is None or node.state == "dead":
            raise OracleError("BAD_NODE", str(nid))
        return node

    def add_root(self, nid: int) -> None:
        assert nid not in self.nodes
        self.nodes[nid] = _Node(-1)

    def append(self, nid: int, kv_id: int, n: int) -> None:
        node = self._live(nid)
        if node.state == "frozen":
            raise OracleError("FROZEN", str(nid))
        if n == 0:
            return
        need = -(-(node.n_tokens + n) // self.bt) - len(node.blocks)
        node.blocks += self._alloc(need) if need > 0 else []
        node.chunks.append(kv_id)
        self.kv_len[kv_id] = n
        node.n_tokens += n

    def fork(self, nid: int, kids: Sequence[int]) -> None:
        """Freeze ``nid`` and give it children; forking a frozen node adds
        more children (a later branch from the same point)."""
        node = self._live(nid)
        if len(kids) < 1:
            raise OracleError("INVALID_ARG", "fork needs k >= 1")
        node.state = "frozen"
        node.kids_live += len(kids)
        for c in kids:
            assert c not in self.nodes
            self.nodes[c] = _Node(nid)

    def prune(self, nid: int) -> None:
        node = self._live(nid)
        if node.state != "leaf":
            raise OracleError("NOT_LEAF", str(nid))
        self._release(node)
        p = node.parent
        while p != -1:
            par = self.nodes[p]
            par.kids_live -= 1
            if par.kids_live > 0:
                break
            self._release(par)
            p = par.parent

    def replay(self, script) -> "OracleForest":
        for op in script.ops:
            kind = op[0]
            if kind == "root":
                self.add_root(op[1])
            elif kind == "append":
                self.append(op[1], op[2], op[3])
            elif kind == "fork":
                self.fork(op[1], op[2])
            elif kind == "prune":
                self.prune(op[1])
            else:
                raise ValueError(kind)
        return self

    # ---- paths --------------------------------------------------------------
    def path_nodes(self, leaf: int, any_node: bool = False) -> List[int]:
        """Node ids from the root down to ``leaf`` (any live node with
        ``any_node``)."""
        node = self._live(leaf)
        if node.state != "leaf" and not any_node:
            raise OracleError("NOT_LEAF", str(leaf))
        out = []
        x = leaf
        while x != -1:
            out.append(x)
            x = self.nodes[x].parent
        return out[::-1]

    def path_slots(self, leaf: int) -> np.ndarray:
        """Pool slot of every token on the path, root first."""
        slots = []
        for x in self.path_nodes(leaf):
            node = self.nodes[x]
            for t in range(node.n_tokens):
                slots.append(node.blocks[t // self.bt] * self.bt + t % self.bt)
        return np.asarray(slots, dtype=np.int64)

    def path_chunks(self, leaf: int, any_node: bool = False) -> List[int]:
        """kv_ids on the path, root first, in append order."""
        out = []
        for x in self.path_nodes(leaf, any_node):
            out += self.nodes[x].chunks
        return out

    def path_kv(self, leaf: int, kv_source: Callable[[int], tuple],
                any_node: bool = False) -> Tuple[np.ndarray, np.ndarray]:
        """Materialise the path: K, V as uint16 bf16 bits [N][Hkv][d]."""
        ks, vs = [], []
        for kv_id in self.path_chunks(leaf, any_node):
            k, v = kv_source(kv_id)
            ks.append(bf16_bits(k))
            vs.append(bf16_bits(v))
        if not ks:
            raise OracleError("EMPTY_PATH", str(leaf))
        return np.concatenate(ks), np.concatenate(vs)

    def decode(self, leaves: Sequence[int], q, kv_source: Callable[[int], tuple],
               threads: Optional[int] = None, indices: Optional[Sequence[int]] = None):
        """fp64 O [n][Hq][d] and LSE [n][Hq] for ``leaves`` (rows of ``q``).

        ``indices`` restricts the work to those rows (others are NaN).
        Threads run over leaves; the C routine releases the GIL.
        """
        qb = bf16_bits(q)
        n = len(leaves)
        hq, d = qb.shape[1], qb.shape[2]
        out = np.full((n, hq, d), np.nan)
        lse = np.full((n, hq), np.nan)
        todo = list(range(n)) if indices is None else list(indices)

        def one(i):
            k, v = self.path_kv(leaves[i], kv_source)
            out[i], lse[i] = path_attention(qb[i], k, v)

        threads = threads or min(len(todo), os.cpu_count() or 1) or 1
        if threads <= 1:
            for i in todo:
                one(i)
        else:
            with ThreadPoolExecutor(max_workers=threads) as ex:
                list(ex.map(one, todo))
        return out, lse

    def prefill(self, nodes: Sequence[int], n_queries: Sequence[int], q, kv_source: Callable[[int], tuple],
                threads: Optional[int] = None, indices: Optional[Sequence[int]] = None):
        """Causal multi-query attention: fp64 O [sum m][Hq][d], LSE [sum m][Hq].

        The last m_i tokens of nodes[i] are queries (rows of ``q`` packed
        node by node); query j sits at path position P_i - m_i + j and
        attends to the path's first P_i - m_i + j + 1 tokens -- the decode
        definition applied to each prefix of the path.
        """
        qb = bf16_bits(q)
        total = int(sum(n_queries))
        hq, d = qb.shape[1], qb.shape[2]
        out = np.full((total, hq, d), np.nan)
        lse = np.full((total, hq), np.nan)
        rows = []                                   # (row, node index, visible tokens)
        r = 0
        for i, (x, m) in enumerate(zip(nodes, n_queries)):
            node = self._live(x)
            path_len = sum(self.nodes[y].n_tokens for y in self.path_nodes(x, True))
            if m > node.n_tokens:
                raise OracleError("INVALID_ARG", f"node {x} holds {node.n_tokens} tokens, {m} queries asked")
            for j in range(m):
                rows.append((r, i, path_len - m + j + 1))
                r += 1
        want = None if indices is None else set(indices)
        paths: Dict[int, Tuple[np.ndarray, np.ndarray]] = {}

        def one(item):
            row, i, vis = item
            if i not in paths:
                paths[i] = self.path_kv(nodes[i], kv_source, any_node=True)
            k, v = paths[i]
            out[row], lse[row] = path_attention(qb[row], k[:vis], v[:vis])

        todo = [it for it in rows if want is None or it[0] in want]
        for it in todo:                              # materialise paths once, then fan out
            if it[1] not in paths:
                paths[it[1]] = self.path_kv(nodes[it[1]], kv_source, any_node=True)
        threads = threads or min(len(todo), os.cpu_count() or 1) or 1
        if threads <= 1:
            for it in todo:
                one(it)
        else:
            with ThreadPoolExecutor(max_workers=threads) as ex:
                list(ex.map(one, todo))
        return out, lse

    # ---- stats ----------------------------------------------------------------
    def live_blocks(self) -> int:
        return int((~self.free).sum())

    def unique_path_tokens(self, leaves: Sequence[int]) -> int:
        seen = set()
        for lf in leaves:
            seen.update(self.path_nodes(lf))
        return sum(self.nodes[x].n_tokens for x in seen)
