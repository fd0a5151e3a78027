"""Python binding of libtreepo: decode attention over a segment tree of KV
caches on one GB300 (sm_103a).

Every function here has the name of the C entry point it calls (declared in
``include/treepo.h``) and only marshals arguments: tensors become device
pointers, node lists become int32 host arrays, status codes become
``TreepoError``. All computation happens in the library's CUDA kernels; when
the library is missing this module raises instead of falling back.

``Forest`` is a small owner object: it allocates the pool arena with PyTorch
(PyTorch is used for device memory and streams only) and frees the tree.
"""
from __future__ import annotations

import ctypes
import os
from typing import Dict, Iterable, List, Optional, Sequence

import numpy as np

__all__ = [
    "TreepoError", "load_library", "library_path", "tp_pool_bytes", "tp_tree_create", "tp_tree_destroy",
    "tp_set_stream", "tp_add_root", "tp_append_segment", "tp_fork", "tp_prune", "tp_decode", "tp_decode_ex",
    "tp_sync", "tp_last_error", "tp_get_node_info", "tp_get_stats", "tp_profile_start", "tp_profile_stop",
    "tp_debug_path", "tp_debug_gather",
    "tp_debug_schedule", "tp_debug_check_schedule", "tp_decode_noalloc", "tp_append_tokens", "tp_synth_tokens", "tp_branch_assign",
    "tp_rollout", "tp_advantage_workspace_bytes", "tp_tree_advantage", "tp_prefill", "tp_debug_prefill_schedule", "tp_decode_host", "tp_prefill_host", "tp_debug_wait_probe", "TpRolloutParams", "TpRolloutStats",
    "TpRolloutProbe", "rollout_params", "TP_BRANCH_EVEN", "TP_BRANCH_LOGP_HIGH", "TP_BRANCH_LOGP_LOW",
    "EVENT_NAMES", "TP_SEG_EOS", "TP_SEG_BOXED", "TP_SEG_FAILED", "TP_SEG_MAX_DEPTH", "Forest", "TP_DECODE_NO_SHARE", "TP_DECODE_CUDA_CORE_SMALL", "TP_DECODE_NO_CACHE", "TP_DECODE_TCGEN05", "TP_DECODE_ALL_TCGEN05", "TP_MMA_SYNC",
    "EXPORTED_SYMBOLS",
]

_HERE = os.path.dirname(os.path.abspath(__file__))
# TREEPO_BOUNDS_CHECK=1 selects the bounds-checked build (same ABI; every
# kernel checks its schedule indices before each access)
BOUNDS_CHECKED = os.environ.get("TREEPO_BOUNDS_CHECK", "0") == "1"
_LIB_PATH = os.path.join(_HERE, "libtreepo_checked.so" if BOUNDS_CHECKED else "libtreepo.so")
_lib: Optional[ctypes.CDLL] = None

TP_DECODE_NO_SHARE = 1
TP_DECODE_CUDA_CORE_SMALL = 2
TP_DECODE_NO_CACHE = 4
TP_DECODE_TCGEN05 = 8
TP_DECODE_ALL_TCGEN05 = 16
TP_MMA_SYNC = 32

TP_BRANCH_EVEN = 0
TP_BRANCH_LOGP_HIGH = 1
TP_BRANCH_LOGP_LOW = 2
TP_SEG_EOS, TP_SEG_BOXED, TP_SEG_FAILED, TP_SEG_MAX_DEPTH = 1, 2, 4, 8
EVENT_NAMES = {1: "root", 2: "fork", 3: "segment", 4: "output", 5: "prune", 6: "fallback", 7: "done"}

STATUS_NAMES = {0: "OK", -1: "INVALID_ARG", -2: "OOM", -3: "BAD_NODE", -4: "FROZEN", -5: "NOT_LEAF",
                -6: "EMPTY_PATH", -7: "CUDA", -8: "DEVICE"}

EXPORTED_SYMBOLS = (
    "tp_pool_bytes", "tp_tree_create", "tp_tree_destroy", "tp_set_stream", "tp_add_root",
    "tp_append_segment", "tp_fork", "tp_prune", "tp_decode", "tp_decode_ex", "tp_sync", "tp_last_error",
    "tp_get_node_info", "tp_get_stats", "tp_profile_start", "tp_profile_stop", "tp_debug_path",
    "tp_debug_gather", "tp_debug_schedule", "tp_decode_noalloc", "tp_append_tokens", "tp_synth_tokens",
    "tp_branch_assign", "tp_rollout", "tp_advantage_workspace_bytes", "tp_tree_advantage", "tp_prefill",
    "tp_debug_prefill_schedule", "tp_decode_host", "tp_prefill_host", "tp_debug_wait_probe",
    "tp_debug_check_schedule",
)


class TreepoError(RuntimeError):
    def __init__(self, status: int, message: str):
        self.status = status
        self.code = STATUS_NAMES.get(status, str(status))
        super().__init__(f"TP_ERR_{self.code}: {message}")


class TpConfig(ctypes.Structure):
    _fields_ = [("num_q_heads", ctypes.c_int32), ("num_kv_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("block_tokens", ctypes.c_int32),
                ("pool_blocks", ctypes.c_int64), ("pool", ctypes.c_void_p), ("cuda_stream", ctypes.c_void_p)]


class TpNodeInfo(ctypes.Structure):
    _fields_ = [("parent", ctypes.c_int32), ("state", ctypes.c_int32), ("n_tokens", ctypes.c_int32),
                ("n_live_children", ctypes.c_int32), ("path_tokens", ctypes.c_int64)]


class TpKernelTimes(ctypes.Structure):
    _fields_ = [("launches", ctypes.c_int64 * 4), ("milliseconds", ctypes.c_double * 4)]


KERNEL_KINDS = ("decode", "merge", "append", "gather")


class TpRolloutParams(ctypes.Structure):
    _fields_ = [("n_queries", ctypes.c_int32), ("prompt_tokens", ctypes.c_void_p), ("width", ctypes.c_int32),
                ("max_depth", ctypes.c_int32), ("seg_tokens", ctypes.c_int32), ("arity", ctypes.c_int32),
                ("init_branches", ctypes.c_int32), ("policy", ctypes.c_int32), ("fallback", ctypes.c_int32),
                ("decode", ctypes.c_int32), ("decode_flags", ctypes.c_uint32), ("reserved", ctypes.c_int32),
                ("temperature", ctypes.c_double), ("p_eos", ctypes.c_double), ("p_boxed", ctypes.c_double),
                ("p_fail", ctypes.c_double), ("p_correct", ctypes.c_double), ("seed", ctypes.c_uint64)]


class TpRolloutStats(ctypes.Structure):
    _fields_ = [(f, ctypes.c_int64) for f in ("iterations", "segments", "tokens", "prompt_tokens", "outputs",
                                               "fallbacks", "decode_calls", "decode_rows", "events",
                                               "peak_blocks", "nodes")]


class TpRolloutProbe(ctypes.Structure):
    _fields_ = [("call", ctypes.c_int64), ("cap", ctypes.c_int32), ("reserved", ctypes.c_int32),
                ("o", ctypes.c_void_p), ("lse", ctypes.c_void_p), ("rows", ctypes.c_void_p),
                ("n_rows", ctypes.c_void_p)]


class TpStats(ctypes.Structure):
    _fields_ = [("pool_blocks", ctypes.c_int64), ("free_blocks", ctypes.c_int64),
                ("live_nodes", ctypes.c_int64), ("total_nodes", ctypes.c_int64)]


def library_path() -> str:
    return _LIB_PATH


def load_library() -> ctypes.CDLL:
    """Load libtreepo.so (built in-tree by ``paper_2508_17445_gb300.build``)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(_LIB_PATH):
        flag = " --checked" if BOUNDS_CHECKED else ""
        raise ImportError(f"{_LIB_PATH} is missing: run `python -m paper_2508_17445_gb300.build{flag}` "
                          "(there is no fallback implementation)")
    lib = ctypes.CDLL(_LIB_PATH)
    P, I32, I64, U32 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_uint32
    sig = {
        "tp_pool_bytes": (I64, [P]),
        "tp_tree_create": (I32, [P, P]),
        "tp_tree_destroy": (I32, [P]),
        "tp_set_stream": (I32, [P, P]),
        "tp_add_root": (I32, [P, P]),
        "tp_append_segment": (I32, [P, I32, I32, P, P]),
        "tp_fork": (I32, [P, I32, I32, P]),
        "tp_prune": (I32, [P, I32]),
        "tp_decode": (I32, [P, P, I32, P, P, P]),
        "tp_decode_ex": (I32, [P, P, I32, P, P, P, U32]),
        "tp_decode_noalloc": (I32, [P, P, I32, P, P, P, U32]),
        "tp_sync": (I32, [P]),
        "tp_last_error": (ctypes.c_char_p, [P]),
        "tp_get_node_info": (I32, [P, I32, P]),
        "tp_get_stats": (I32, [P, P]),
        "tp_profile_start": (I32, [P]),
        "tp_profile_stop": (I32, [P, P]),
        "tp_debug_path": (I32, [P, I32, P, I64, P]),
        "tp_debug_gather": (I32, [P, I32, P, P, I64, P]),
        "tp_debug_schedule": (I32, [P, P, I32, U32, P, I64, P]),
        "tp_append_tokens": (I32, [P, P, I32, P, P]),
        "tp_synth_tokens": (I32, [P, ctypes.c_uint64, I32, I32, I32, P, P, P]),
        "tp_branch_assign": (I32, [P, I32, I32, I32, ctypes.c_double, P]),
        "tp_rollout": (I32, [P, P, P, I64, P, P]),
        "tp_advantage_workspace_bytes": (I64, [I32, I32]),
        "tp_tree_advantage": (I32, [P, I32, P, P, I32, P, P, P, I64, P]),
        "tp_prefill": (I32, [P, P, P, I32, P, P, P, U32]),
        "tp_decode_host": (I32, [P, P, I32, P, P, P, U32]),
        "tp_prefill_host": (I32, [P, P, P, I32, P, P, P, U32]),
        "tp_debug_wait_probe": (I32, [P, I64]),
        "tp_debug_prefill_schedule": (I32, [P, P, P, I32, U32, P, I64, P]),
        "tp_debug_check_schedule": (I32, [P, P, I64, P]),
    }
    for name, (res, args) in sig.items():
        f = getattr(lib, name)
        f.restype = res
        f.argtypes = args
    _lib = lib
    return lib


def _check(handle, status: int) -> None:
    if status != 0:
        msg = load_library().tp_last_error(handle)
        raise TreepoError(status, msg.decode() if msg else "")


def _ptr(t) -> Optional[int]:
    if t is None:
        return None
    return t.data_ptr()


def _node_array(nodes: Sequence[int]) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(nodes, dtype=np.int32).reshape(-1))


# ---------------------------------------------------------------- C calls --
def tp_pool_bytes(cfg: TpConfig) -> int:
    return int(load_library().tp_pool_bytes(ctypes.byref(cfg)))


def tp_tree_create(cfg: TpConfig) -> ctypes.c_void_p:
    h = ctypes.c_void_p()
    _check(None, load_library().tp_tree_create(ctypes.byref(cfg), ctypes.byref(h)))
    return h


def tp_tree_destroy(h) -> None:
    _check(None, load_library().tp_tree_destroy(h))


def tp_set_stream(h, stream_ptr: int) -> None:
    _check(h, load_library().tp_set_stream(h, stream_ptr))


def tp_add_root(h) -> int:
    out = ctypes.c_int32()
    _check(h, load_library().tp_add_root(h, ctypes.byref(out)))
    return out.value


def tp_append_segment(h, node: int, n_tokens: int, K=None, V=None) -> None:
    """K, V: device bf16 [n_tokens][Hkv][hd] tensors (None on a metadata-only tree)."""
    _check(h, load_library().tp_append_segment(h, node, n_tokens, _ptr(K), _ptr(V)))


def tp_fork(h, node: int, k: int) -> List[int]:
    out = (ctypes.c_int32 * max(k, 1))()
    _check(h, load_library().tp_fork(h, node, k, out))
    return list(out[:k])


def tp_prune(h, leaf: int) -> None:
    _check(h, load_library().tp_prune(h, leaf))


def tp_decode_ex(h, leaves: Sequence[int], Q, O, LSE, flags: int = 0) -> None:
    arr = _node_array(leaves)
    _check(h, load_library().tp_decode_ex(h, arr.ctypes.data, len(arr), _ptr(Q), _ptr(O), _ptr(LSE), flags))


def tp_decode(h, leaves: Sequence[int], Q, O, LSE) -> None:
    arr = _node_array(leaves)
    _check(h, load_library().tp_decode(h, arr.ctypes.data, len(arr), _ptr(Q), _ptr(O), _ptr(LSE)))


def tp_decode_noalloc(h, leaves: Sequence[int], Q, O, LSE, flags: int = 0) -> None:
    """tp_decode_ex without device allocation (scratch in the library's static array)."""
    arr = _node_array(leaves)
    _check(h, load_library().tp_decode_noalloc(h, arr.ctypes.data, len(arr), _ptr(Q), _ptr(O), _ptr(LSE), flags))


def tp_sync(h) -> None:
    _check(h, load_library().tp_sync(h))


def tp_last_error(h) -> str:
    m = load_library().tp_last_error(h)
    return m.decode() if m else ""


def tp_get_node_info(h, node: int) -> Dict[str, int]:
    info = TpNodeInfo()
    _check(h, load_library().tp_get_node_info(h, node, ctypes.byref(info)))
    return {f: getattr(info, f) for f, _ in TpNodeInfo._fields_}


def tp_get_stats(h) -> Dict[str, int]:
    st = TpStats()
    _check(h, load_library().tp_get_stats(h, ctypes.byref(st)))
    return {f: getattr(st, f) for f, _ in TpStats._fields_}


def tp_profile_start(h) -> None:
    _check(h, load_library().tp_profile_start(h))


def tp_profile_stop(h) -> Dict[str, Dict[str, float]]:
    """{kernel kind: {"launches": n, "ms": summed event time}}."""
    kt = TpKernelTimes()
    _check(h, load_library().tp_profile_stop(h, ctypes.byref(kt)))
    return {k: {"launches": int(kt.launches[i]), "ms": float(kt.milliseconds[i])} for i, k in enumerate(KERNEL_KINDS)}


def tp_debug_path(h, leaf: int) -> np.ndarray:
    n = ctypes.c_int64()
    lib = load_library()
    info = tp_get_node_info(h, leaf)
    cap = max(int(info["path_tokens"]), 1)
    out = np.zeros(cap, dtype=np.int64)
    _check(h, lib.tp_debug_path(h, leaf, out.ctypes.data, cap, ctypes.byref(n)))
    return out[: n.value]


def tp_debug_gather(h, leaf: int, K_out, V_out) -> int:
    n = ctypes.c_int64()
    _check(h, load_library().tp_debug_gather(h, leaf, _ptr(K_out), _ptr(V_out), K_out.shape[0], ctypes.byref(n)))
    return n.value


def tp_prefill(h, nodes: Sequence[int], n_queries: Sequence[int], Q, O, LSE, flags: int = 0) -> None:
    """Q, O: device bf16 [sum n_queries][Hq][hd]; LSE: device fp32 [sum n_queries][Hq]."""
    arr = _node_array(nodes)
    m = np.ascontiguousarray(np.asarray(n_queries, dtype=np.int32).reshape(-1))
    _check(h, load_library().tp_prefill(h, arr.ctypes.data if len(arr) else None,
                                        m.ctypes.data if len(m) else None, len(arr), _ptr(Q), _ptr(O), _ptr(LSE),
                                        flags))


def _host_ptr(t) -> int:
    if t.is_cuda or not t.is_contiguous():
        raise ValueError("host-buffer calls take contiguous CPU tensors (pinned for overlap)")
    return t.data_ptr()


def tp_decode_host(h, leaves: Sequence[int], Q, O, LSE, flags: int = 0) -> None:
    """tp_decode_ex with host Q/O/LSE (contiguous CPU tensors, ideally pinned);
    asynchronous: read O and LSE after tp_sync."""
    arr = _node_array(leaves)
    _check(h, load_library().tp_decode_host(h, arr.ctypes.data if len(arr) else None, len(arr), _host_ptr(Q),
                                            _host_ptr(O), _host_ptr(LSE), flags))


def tp_prefill_host(h, nodes: Sequence[int], n_queries: Sequence[int], Q, O, LSE, flags: int = 0) -> None:
    """tp_prefill with host Q/O/LSE (contiguous CPU tensors, ideally pinned);
    asynchronous: read O and LSE after tp_sync."""
    arr = _node_array(nodes)
    m = np.ascontiguousarray(np.asarray(n_queries, dtype=np.int32).reshape(-1))
    _check(h, load_library().tp_prefill_host(h, arr.ctypes.data if len(arr) else None,
                                             m.ctypes.data if len(m) else None, len(arr), _host_ptr(Q),
                                             _host_ptr(O), _host_ptr(LSE), flags))


def tp_debug_wait_probe(h, limit_ns: int) -> None:
    """Launch the bounded-wait probe: the next tp_sync raises TreepoError DEVICE."""
    _check(h, load_library().tp_debug_wait_probe(h, int(limit_ns)))


def _parse_schedule(w: np.ndarray) -> Dict[str, np.ndarray]:
    assert w[0] == 0x54505344
    n_units, n_tiles, n_occ, n, n_slots, n_merge, g, n_tensor, n_tc = (int(x) for x in w[1:10])
    off = 16
    units = w[off: off + 8 * n_units].reshape(n_units, 8)
    off += 8 * n_units
    tiles = w[off: off + n_tiles]
    off += n_tiles
    occ = w[off: off + n_occ]
    off += n_occ
    merge_off = w[off: off + n + 1]
    off += n + 1
    merge_slot = w[off: off + n_merge]
    off += n_merge
    out = {"units": units, "tiles": tiles, "occ": occ, "merge_off": merge_off, "merge_slot": merge_slot,
           "n_slots": n_slots, "group": g, "n_tensor_units": n_tensor, "n_tc_units": n_tc, "words": w}
    if w[10] == 1:
        out["unit_pos"] = w[off: off + n_units]
        out["vis"] = w[off + n_units: off + n_units + n]
        off += n_units + n
    rw = int(w[11])
    if rw:
        out["merge_rec"] = w[off: off + n * rw].reshape(n, rw)
    return out


def tp_debug_prefill_schedule(h, nodes: Sequence[int], n_queries: Sequence[int], flags: int = 0):
    """The schedule tp_prefill would run, decoded into arrays."""
    arr = _node_array(nodes)
    m = np.ascontiguousarray(np.asarray(n_queries, dtype=np.int32).reshape(-1))
    lib = load_library()
    n_words = ctypes.c_int64()
    args = (arr.ctypes.data if len(arr) else None, m.ctypes.data if len(m) else None, len(arr), flags)
    _check(h, lib.tp_debug_prefill_schedule(h, *args, None, 0, ctypes.byref(n_words)))
    buf = np.zeros(max(n_words.value, 1), dtype=np.int32)
    _check(h, lib.tp_debug_prefill_schedule(h, *args, buf.ctypes.data, len(buf), ctypes.byref(n_words)))
    return _parse_schedule(buf[: n_words.value])


def tp_debug_schedule(h, leaves: Sequence[int], flags: int = 0) -> Dict[str, np.ndarray]:
    """The schedule tp_decode_ex(flags) would run, decoded into arrays."""
    arr = _node_array(leaves)
    lib = load_library()
    n_words = ctypes.c_int64()
    _check(h, lib.tp_debug_schedule(h, arr.ctypes.data if len(arr) else None, len(arr), flags, None, 0,
                                     ctypes.byref(n_words)))
    buf = np.zeros(max(n_words.value, 1), dtype=np.int32)
    _check(h, lib.tp_debug_schedule(h, arr.ctypes.data if len(arr) else None, len(arr), flags,
                                     buf.ctypes.data, len(buf), ctypes.byref(n_words)))
    return _parse_schedule(buf[: n_words.value])


CHECK_CATEGORIES = ("units", "tiles", "occ", "merge_ranges", "merge_slots")


def tp_debug_check_schedule(h, words: np.ndarray) -> Dict[str, int]:
    """Violation counts of a schedule's words under the bounds-checked
    kernels' index predicates (zero everywhere for a valid schedule)."""
    w = np.ascontiguousarray(np.asarray(words, dtype=np.int32))
    out = (ctypes.c_int64 * 5)()
    _check(h, load_library().tp_debug_check_schedule(h, w.ctypes.data, len(w), out))
    return dict(zip(CHECK_CATEGORIES, (int(x) for x in out)))


def tp_append_tokens(h, nodes: Sequence[int], K=None, V=None) -> None:
    """One token per node; K, V: device bf16 [n][Hkv][hd] (None on a metadata-only tree)."""
    arr = _node_array(nodes)
    _check(h, load_library().tp_append_tokens(h, arr.ctypes.data if len(arr) else None, len(arr), _ptr(K), _ptr(V)))


def tp_synth_tokens(h, seed: int, node: int, pos0: int, n_tokens: int, K=None, V=None, Q=None) -> None:
    _check(h, load_library().tp_synth_tokens(h, seed, node, pos0, n_tokens, _ptr(K), _ptr(V), _ptr(Q)))


def tp_branch_assign(logp: Optional[Sequence[float]], n: int, budget: int, policy: int,
                     temperature: float = 1.0) -> List[int]:
    lp = None if logp is None else np.ascontiguousarray(np.asarray(logp, dtype=np.float64))
    out = np.zeros(max(n, 1), dtype=np.int32)
    st = load_library().tp_branch_assign(None if lp is None else lp.ctypes.data, n, budget, policy,
                                         float(temperature), out.ctypes.data)
    if st != 0:
        raise TreepoError(st, "tp_branch_assign rejected its arguments")
    return [int(x) for x in out[:n]]


def rollout_params(prompt_tokens: Sequence[int], **kw) -> TpRolloutParams:
    """Parameters with defaults: w=16, d=14, l=512, binary, b0=2, even split,
    fallback on, no decode, T=2.0; ``prompt_tokens`` is kept alive on the
    returned object."""
    arr = np.ascontiguousarray(np.asarray(prompt_tokens, dtype=np.int32))
    d = dict(width=16, max_depth=14, seg_tokens=512, arity=2, init_branches=2, policy=TP_BRANCH_EVEN, fallback=1,
             decode=0, decode_flags=0, temperature=2.0, p_eos=0.0, p_boxed=0.0, p_fail=0.0, p_correct=0.5, seed=0)
    d.update(kw)
    p = TpRolloutParams(n_queries=len(arr), prompt_tokens=arr.ctypes.data, reserved=0, **d)
    p._prompts = arr
    return p


def tp_rollout(h, params: TpRolloutParams, cap_events: int = 1 << 20, probe: Optional[TpRolloutProbe] = None):
    """Run Algorithm 1; returns (events int64 [n][8], stats dict)."""
    ev = np.zeros((max(cap_events, 1), 8), dtype=np.int64)
    st = TpRolloutStats()
    _check(h, load_library().tp_rollout(h, ctypes.byref(params), ev.ctypes.data, cap_events,
                                        ctypes.byref(probe) if probe is not None else None, ctypes.byref(st)))
    stats = {f: int(getattr(st, f)) for f, _ in TpRolloutStats._fields_}
    if stats["events"] > cap_events:
        raise TreepoError(-1, f"{stats['events']} events exceed cap_events={cap_events}")
    return ev[: stats["events"]].copy(), stats


def tp_advantage_workspace_bytes(n_nodes: int, n_out: int) -> int:
    return int(load_library().tp_advantage_workspace_bytes(n_nodes, n_out))


def tp_tree_advantage(parent, leaf, reward, adv, stats=None, workspace=None, stream: int = 0) -> None:
    """parent int32 [n_nodes], leaf int32 [n_out], reward / adv float32 [n_out], stats float64 [4] (device tensors)."""
    ws_bytes = tp_advantage_workspace_bytes(int(parent.shape[0]), int(leaf.shape[0]))
    if workspace is None:
        import torch
        workspace = torch.empty(max(ws_bytes, 8), dtype=torch.uint8, device=parent.device)
    st = load_library().tp_tree_advantage(_ptr(parent), int(parent.shape[0]), _ptr(leaf), _ptr(reward),
                                          int(leaf.shape[0]), _ptr(adv), _ptr(stats), _ptr(workspace),
                                          int(workspace.numel()), stream)
    _check(None, st)


# ------------------------------------------------------------------ owner --
class Forest:
    """A tp_tree plus the pool arena it owns.

    ``device=None`` builds a metadata-only tree (no CUDA, no pool): the host
    logic runs, appends copy nothing, decode is refused.
    """

    def __init__(self, num_q_heads: int, num_kv_heads: int, head_dim: int, pool_blocks: int,
                 block_tokens: int = 32, device=None, stream=None):
        self.cfg = TpConfig(num_q_heads, num_kv_heads, head_dim, block_tokens, pool_blocks, None, None)
        self.device = device
        self.pool = None
        if device is not None:
            import torch
            nbytes = tp_pool_bytes(self.cfg)
            if nbytes <= 0:
                raise TreepoError(-1, "bad tree configuration")
            self.pool = torch.empty(nbytes, dtype=torch.uint8, device=device)
            self.cfg.pool = self.pool.data_ptr()
            s = stream if stream is not None else torch.cuda.current_stream(device)
            self.cfg.cuda_stream = s.cuda_stream
        self.handle = tp_tree_create(self.cfg)

    def close(self) -> None:
        if getattr(self, "handle", None) is not None:
            tp_tree_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    # thin methods
    def add_root(self) -> int:
        return tp_add_root(self.handle)

    def append(self, node: int, K=None, V=None, n_tokens: Optional[int] = None) -> None:
        n = int(K.shape[0]) if K is not None else int(n_tokens)
        tp_append_segment(self.handle, node, n, K, V)

    def fork(self, node: int, k: int) -> List[int]:
        return tp_fork(self.handle, node, k)

    def prune(self, leaf: int) -> None:
        tp_prune(self.handle, leaf)

    def decode(self, leaves: Sequence[int], Q, flags: int = 0, out=None):
        import torch
        n, hq, hd = Q.shape
        if out is None:
            O = torch.empty((n, hq, hd), dtype=torch.bfloat16, device=Q.device)
            LSE = torch.empty((n, hq), dtype=torch.float32, device=Q.device)
        else:
            O, LSE = out
        tp_decode_ex(self.handle, leaves, Q, O, LSE, flags)
        return O, LSE

    def decode_host(self, leaves: Sequence[int], Q, flags: int = 0, out=None):
        """decode with host Q (CPU tensor, ideally pinned); O and LSE are
        pinned host tensors, valid after sync()."""
        import torch
        n, hq, hd = Q.shape
        if out is None:
            O = torch.empty((n, hq, hd), dtype=torch.bfloat16).pin_memory()
            LSE = torch.empty((n, hq), dtype=torch.float32).pin_memory()
        else:
            O, LSE = out
        tp_decode_host(self.handle, leaves, Q, O, LSE, flags)
        return O, LSE

    def prefill(self, nodes: Sequence[int], n_queries: Sequence[int], Q, flags: int = 0, out=None):
        """Causal attention of the last n_queries[i] tokens of nodes[i] over
        their paths; Q: [sum n_queries][Hq][hd] on the device."""
        import torch
        n, hq, hd = Q.shape
        if out is None:
            O = torch.empty((n, hq, hd), dtype=torch.bfloat16, device=Q.device)
            LSE = torch.empty((n, hq), dtype=torch.float32, device=Q.device)
        else:
            O, LSE = out
        tp_prefill(self.handle, nodes, n_queries, Q, O, LSE, flags)
        return O, LSE

    def append_tokens(self, nodes: Sequence[int], K=None, V=None) -> None:
        tp_append_tokens(self.handle, nodes, K, V)

    def rollout(self, params: TpRolloutParams, cap_events: int = 1 << 20, probe=None):
        return tp_rollout(self.handle, params, cap_events, probe)

    def sync(self) -> None:
        tp_sync(self.handle)

    def stats(self) -> Dict[str, int]:
        return tp_get_stats(self.handle)

    def node_info(self, node: int) -> Dict[str, int]:
        return tp_get_node_info(self.handle, node)

    def replay(self, ops: Iterable[tuple], kv_fn=None) -> Dict[int, int]:
        """Apply a script of tree operations; returns script id -> node id.

        ops: ("root", sid) | ("append", sid, kv_id, n) | ("fork", sid, (c..)) |
        ("prune", sid). kv_fn(kv_id) -> (K, V) device tensors; with no kv_fn
        (metadata-only tree) appends carry no data.
        """
        ids: Dict[int, int] = {}
        for op in ops:
            kind = op[0]
            if kind == "root":
                ids[op[1]] = self.add_root()
            elif kind == "append":
                if kv_fn is None:
                    tp_append_segment(self.handle, ids[op[1]], op[3], None, None)
                else:
                    K, V = kv_fn(op[2])
                    self.append(ids[op[1]], K, V)
            elif kind == "fork":
                kids = self.fork(ids[op[1]], len(op[2]))
                for sid, nid in zip(op[2], kids):
                    ids[sid] = nid
            elif kind == "prune":
                self.prune(ids[op[1]])
            else:
                raise ValueError(f"unknown op {kind!r}")
        return ids
