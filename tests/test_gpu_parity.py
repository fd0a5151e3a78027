"""GPU parity: libtreepo's CUDA path against the fp64 CPU oracle.

Every case replays the same seeded workload script on both sides: through
the C ABI on cuda:0 (K/V/Q drawn on the device by the workload's seeded
generators) and through the oracle's plain tree model on the CPU (the same
tensors, copied to the host). Outputs are compared element by element.

Tolerances. The contract bar is max|dO| <= 1e-2 and max|dLSE| <= 1e-3 (bf16
inputs, fp32 accumulation). A second, tighter bar follows from the
arithmetic. bf16 round-to-nearest has unit roundoff u = 2^-8. O is rounded
to bf16 once (<= u|O|); on the tensor path each probability is rounded to
bf16 before P.V, which moves O by at most u * A with A = sum_j p_j |v_j|
(the attention output over |V|, computed by the oracle); fp32 sums and the
exp2 approximation add ~1e-6. So |dO| <= u (|O| + A) + 1e-5 and
|dLSE| <= 5e-5 (LSE never sees a rounded probability) -- the LSE bar fails
when a single token of a long path is dropped or counted twice.
"""
import numpy as np
import pytest
import torch

import oracle
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


def _kv_source(script):
    cache = {}

    def src(kv_id):
        if kv_id not in cache:
            k, v = script.kv(kv_id, DEV)
            cache[kv_id] = (k.cpu(), v.cpu())
        return cache[kv_id]
    return src


def build_forest(script, extra_blocks=64):
    h = script.heads
    f = tp.Forest(h.num_q_heads, h.num_kv_heads, h.head_dim,
                  pool_blocks=script.upper_bound_blocks(32) + extra_blocks, device=DEV)
    ids = f.replay(script.ops, kv_fn=lambda kv_id: script.kv(kv_id, DEV))
    return f, ids


def check(o_gpu, lse_gpu, o_ref, lse_ref, a_ref=None, rows=None):
    o = o_gpu.float().cpu().numpy().astype(np.float64)
    lse = lse_gpu.cpu().numpy().astype(np.float64)
    if rows is not None:
        o, lse, o_ref, lse_ref = o[rows], lse[rows], o_ref[rows], lse_ref[rows]
        a_ref = None if a_ref is None else a_ref[rows]
    d_o = np.abs(o - o_ref)
    d_lse = np.abs(lse - lse_ref)
    assert np.isfinite(o).all() and np.isfinite(lse).all()
    assert d_o.max() <= TOL_O, f"max|dO| = {d_o.max():.3g}"
    assert d_lse.max() <= TOL_LSE, f"max|dLSE| = {d_lse.max():.3g}"
    if a_ref is not None:
        bound = 2.0 ** -8 * (np.abs(o_ref) + a_ref) + 1e-5
        worst = (d_o - bound).max()
        assert worst <= 0, f"|dO| exceeds 2^-8 (|O| + A) + 1e-5 by {worst:.3g}"
    assert d_lse.max() <= 5e-5, f"max|dLSE| = {d_lse.max():.3g}"
    return float(d_o.max()), float(d_lse.max())


def oracle_outputs(model, leaves_sid, q_cpu, src, rows=None):
    """Oracle O, LSE and A = attention output over |V| (for the rounding bound)."""
    o_ref, lse_ref = model.decode(leaves_sid, q_cpu, src, indices=rows)

    def abs_src(kv_id):
        k, v = src(kv_id)
        return k, oracle.bf16_bits(v) & np.uint16(0x7FFF)
    a_ref, _ = model.decode(leaves_sid, q_cpu, abs_src, indices=rows)
    return o_ref, lse_ref, a_ref


def run_and_compare(script, flags=0, sample=None, leaves=None, q=None):
    f, ids = build_forest(script)
    leaves_sid = script.leaves if leaves is None else leaves
    leaf_ids = [ids[x] for x in leaves_sid]
    Q = script.q(DEV, n=len(leaf_ids)) if q is None else q
    O, LSE = f.decode(leaf_ids, Q, flags=flags)
    f.sync()
    model = oracle.OracleForest(block_tokens=32, pool_blocks=f.cfg.pool_blocks).replay(script)
    rows = None if sample is None else sorted(sample)
    o_ref, lse_ref, a_ref = oracle_outputs(model, leaves_sid, Q.cpu(), _kv_source(script), rows)
    err = check(O, LSE, o_ref, lse_ref, a_ref, rows=rows)
    f.close()
    return O, LSE, err


# default routing, CUDA-core small units, no sharing, all mma.sync, and
# tcgen05 forced (calls under 1 MiB of K/V default to mma.sync only)
FLAG_SETS = [0, tp.TP_DECODE_CUDA_CORE_SMALL, tp.TP_DECODE_NO_SHARE, tp.TP_MMA_SYNC, tp.TP_DECODE_ALL_TCGEN05]


# --------------------------------------------------------------------------
# small cases: every output compared
# --------------------------------------------------------------------------
@pytest.mark.parametrize("flags", FLAG_SETS)
def test_tiny_config(flags):
    run_and_compare(workloads.tiny(seed=0), flags)


@pytest.mark.parametrize("seed", range(4))
@pytest.mark.parametrize("heads", [workloads.Heads(8, 2, 64), workloads.Heads(28, 4, 128),
                                   workloads.Heads(64, 8, 128), workloads.Heads(16, 16, 128)])
def test_random_forests(seed, heads):
    s = workloads.random_tree(seed=seed, heads=heads, n_prompts=3, max_depth=5,
                              prompt_range=(1, 400), seg_range=(1, 200))
    run_and_compare(s, flags=FLAG_SETS[seed % 4])
    run_and_compare(s, flags=tp.TP_DECODE_ALL_TCGEN05)


@pytest.mark.parametrize("heads", [workloads.Heads(32, 2, 64), workloads.Heads(24, 2, 128)])
def test_gqa_groups_wider_than_eight(heads):
    # g = 16 and 12 q heads per kv head: 128-row tensor units hold 8 and 10
    # occurrences, 64-row mma.sync units 4 and 5
    s = workloads.random_tree(seed=7, heads=heads, n_prompts=2, max_depth=4,
                              prompt_range=(1, 300), seg_range=(1, 150))
    for flags in FLAG_SETS:
        run_and_compare(s, flags)


@pytest.mark.parametrize("flags", FLAG_SETS)
def test_qwen7b_shape_reduced(flags):
    # two prompts: ragged prompt lengths, 512-token segments, rows 112/56/28/14/7
    run_and_compare(workloads.qwen7b(seed=1, n_prompts=2), flags)


@pytest.mark.parametrize("flags", FLAG_SETS)
def test_random_divergence_reduced(flags):
    run_and_compare(workloads.random_divergence(seed=2, n_prompts=3, depth=5), flags)


@pytest.mark.parametrize("flags", [0, tp.TP_DECODE_NO_SHARE, tp.TP_DECODE_TCGEN05, tp.TP_MMA_SYNC])
def test_wide_prefix_one_prompt(flags):
    # root shared by 64 leaves x 8 heads = 512 rows: 8 tensor units per chunk
    run_and_compare(workloads.wide_prefix(seed=3, n_prompts=1), flags)


def test_no_sharing_reduced():
    run_and_compare(workloads.no_sharing(seed=4, n_seqs=6))


# --------------------------------------------------------------------------
# edge cases
# --------------------------------------------------------------------------
@pytest.mark.parametrize("lengths", [(1,), (31,), (32,), (33,), (1, 1, 1), (64, 1), (5, 27, 32, 1, 64, 200),
                                     (4096,)])
@pytest.mark.parametrize("heads", [workloads.Heads(4, 1, 64), workloads.Heads(8, 1, 128)])
def test_single_paths_with_ragged_blocks(lengths, heads):
    for flags in FLAG_SETS:
        run_and_compare(workloads.single_path(seed=len(lengths), lengths=lengths, heads=heads), flags)


@pytest.mark.parametrize("flags", FLAG_SETS)
def test_long_shared_prompt_is_chunked(flags):
    # 2000 tokens shared by 3 leaves x 8 heads = 24 rows: the prompt item is
    # cut into several chunks, each writing 24-row partials merged per leaf
    s = workloads.shared_prompt(seed=9)
    f, ids = build_forest(s)
    sched = tp.tp_debug_schedule(f.handle, [ids[x] for x in s.leaves], flags)
    f.close()
    if not flags & tp.TP_DECODE_NO_SHARE:
        assert max(np.diff(sched["merge_off"])) >= 3
    run_and_compare(s, flags)


@pytest.mark.parametrize("flags", FLAG_SETS)
def test_more_slots_than_one_merge_chunk(flags):
    # a 12000-token path at head_dim 128 is cut into more than 32 chunks: the
    # merge folds the slots 32 at a time and rescales across the chunks
    s = workloads.single_path(seed=12, lengths=(12000,), heads=workloads.Heads(8, 1, 128))
    f, ids = build_forest(s)
    sched = tp.tp_debug_schedule(f.handle, [ids[x] for x in s.leaves], flags)
    f.close()
    assert max(np.diff(sched["merge_off"])) > 32
    run_and_compare(s, flags)


def test_repeated_leaf_gives_bitwise_identical_rows():
    s = workloads.random_tree(seed=5, heads=workloads.Heads(28, 4, 128), n_prompts=2)
    f, ids = build_forest(s)
    leaf = ids[s.leaves[0]]
    q1 = s.q(DEV, n=1)
    Q = q1.repeat(5, 1, 1).contiguous()
    for flags in FLAG_SETS:
        O, LSE = f.decode([leaf] * 5, Q, flags=flags)
        f.sync()
        for r in range(1, 5):
            assert torch.equal(O[0], O[r]) and torch.equal(LSE[0], LSE[r])
    f.close()


def test_identical_siblings_give_bitwise_identical_outputs():
    # two siblings whose last segments carry the same K/V and the same query
    heads = workloads.Heads(8, 2, 128)
    gen = torch.Generator(device=DEV).manual_seed(7)
    f = tp.Forest(8, 2, 128, pool_blocks=256, device=DEV)
    r = f.add_root()
    k = torch.randn(300, 2, 128, generator=gen, device=DEV).to(torch.bfloat16)
    v = torch.randn(300, 2, 128, generator=gen, device=DEV).to(torch.bfloat16)
    f.append(r, k, v)
    a, b = f.fork(r, 2)
    k2 = torch.randn(70, 2, 128, generator=gen, device=DEV).to(torch.bfloat16)
    v2 = torch.randn(70, 2, 128, generator=gen, device=DEV).to(torch.bfloat16)
    f.append(a, k2, v2)
    f.append(b, k2, v2)
    q = torch.randn(1, 8, 128, generator=gen, device=DEV).to(torch.bfloat16).repeat(2, 1, 1).contiguous()
    for flags in FLAG_SETS:
        O, LSE = f.decode([a, b], q, flags=flags)
        f.sync()
        assert torch.equal(O[0], O[1]) and torch.equal(LSE[0], LSE[1])
    f.close()


def test_empty_leaf_set_is_a_no_op():
    s = workloads.tiny()
    f, ids = build_forest(s)
    Q = torch.empty(0, 4, 64, dtype=torch.bfloat16, device=DEV)
    O, LSE = f.decode([], Q)
    f.sync()
    assert O.shape == (0, 4, 64)
    f.close()


def test_decode_errors_on_device_tree():
    s = workloads.tiny()
    f, ids = build_forest(s)
    Q = s.q(DEV, n=1)
    root = ids[0]
    with pytest.raises(tp.TreepoError) as e:
        f.decode([root], Q)
    assert e.value.code == "NOT_LEAF"
    leaf = ids[s.leaves[0]]
    f.prune(leaf)
    with pytest.raises(tp.TreepoError) as e:
        f.decode([leaf], Q)
    assert e.value.code == "BAD_NODE"
    bad_q = torch.empty(2 * 4 * 64 + 1, dtype=torch.bfloat16, device=DEV)[1:].view(2, 4, 64)
    with pytest.raises(tp.TreepoError) as e:
        f.decode([ids[s.leaves[1]], ids[s.leaves[2]]], bad_q)   # misaligned Q
    assert e.value.code == "INVALID_ARG"
    f.sync()
    f.close()


def test_pruned_blocks_are_reused_and_results_stay_exact():
    # grow, prune half, grow again into freed blocks, decode everything alive
    s = workloads.random_divergence(seed=6, n_prompts=2, depth=4, segment=96, prompt=200,
                                    heads=workloads.Heads(28, 4, 128))
    run_and_compare(s)


def test_gather_reproduces_paths_bit_for_bit():
    s = workloads.random_tree(seed=8, heads=workloads.Heads(28, 4, 128), n_prompts=3, max_depth=4)
    f, ids = build_forest(s)
    model = oracle.OracleForest(block_tokens=32, pool_blocks=f.cfg.pool_blocks).replay(s)
    src = _kv_source(s)
    for sid in set(s.leaves):
        k_ref, v_ref = model.path_kv(sid, src)
        n = k_ref.shape[0]
        K = torch.empty((n, 4, 128), dtype=torch.bfloat16, device=DEV)
        V = torch.empty_like(K)
        assert tp.tp_debug_gather(f.handle, ids[sid], K, V) == n
        assert np.array_equal(oracle.bf16_bits(K), k_ref)
        assert np.array_equal(oracle.bf16_bits(V), v_ref)
    f.sync()
    f.close()


def test_schedule_cache_follows_tree_changes():
    s = workloads.tiny(seed=2)
    f, ids = build_forest(s)
    model = oracle.OracleForest(block_tokens=32, pool_blocks=f.cfg.pool_blocks).replay(s)
    leaves = [ids[x] for x in s.leaves]
    Q = s.q(DEV)
    f.decode(leaves, Q)
    # grow one leaf by 5 tokens; the cached schedule must not be reused
    gen = torch.Generator(device=DEV).manual_seed(1)
    k = torch.randn(5, 1, 64, generator=gen, device=DEV).to(torch.bfloat16)
    v = torch.randn(5, 1, 64, generator=gen, device=DEV).to(torch.bfloat16)
    f.append(leaves[0], k, v)
    O, LSE = f.decode(leaves, Q)
    f.sync()
    model.append(s.leaves[0], 10_000, 5)
    src = _kv_source(s)

    def src2(kv_id):
        return (k.cpu(), v.cpu()) if kv_id == 10_000 else src(kv_id)
    o_ref, lse_ref, a_ref = oracle_outputs(model, s.leaves, Q.cpu(), src2)
    check(O, LSE, o_ref, lse_ref, a_ref)
    f.close()


def test_bounded_wait_reports_and_the_tree_stays_usable():
    # a kernel whose bounded wait (the attention kernels' helper, 20 ms limit
    # instead of 2 s) runs out on a barrier nothing completes: tp_sync reports
    # it, clears the flag, and the same tree decodes bit-identically afterwards
    s = workloads.tiny(seed=1)
    f, ids = build_forest(s)
    leaves = [ids[x] for x in s.leaves]
    Q = s.q(DEV)
    O1, L1 = f.decode(leaves, Q)
    f.sync()
    O1, L1 = O1.clone(), L1.clone()
    with pytest.raises(tp.TreepoError) as e:
        tp.tp_debug_wait_probe(f.handle, 10)  # below the 1 us floor
    assert e.value.code == "INVALID_ARG"
    tp.tp_debug_wait_probe(f.handle, 20_000_000)
    with pytest.raises(tp.TreepoError) as e:
        f.sync()
    assert e.value.code == "DEVICE"
    f.sync()  # the flag was cleared
    O2, L2 = f.decode(leaves, Q)
    f.sync()
    assert torch.equal(O1.view(torch.int16), O2.view(torch.int16)) and torch.equal(L1, L2)
    f.close()


@pytest.mark.parametrize("flags", [0, tp.TP_MMA_SYNC, tp.TP_DECODE_CUDA_CORE_SMALL])
def test_profile_counts_kernel_launches(flags):
    s = workloads.tiny()
    f, ids = build_forest(s)
    leaves = [ids[x] for x in s.leaves]
    d = tp.tp_debug_schedule(f.handle, leaves, flags)
    n_units, n_tc, n_mma = len(d["units"]), d["n_tc_units"], d["n_tensor_units"]
    per_call = (n_tc > 0) + (n_mma > 0) + (n_units > n_tc + n_mma)  # attention kernels of one call
    assert per_call >= 1
    Q = s.q(DEV)
    f.decode(leaves, Q, flags=flags)  # builds and caches the schedule
    tp.tp_profile_start(f.handle)
    for _ in range(3):
        f.decode(leaves, Q, flags=flags)
    t = tp.tp_profile_stop(f.handle)
    assert t["decode"]["launches"] == 3 * per_call and t["merge"]["launches"] == 3
    assert t["decode"]["ms"] > 0
    f.sync()
    f.close()


# --------------------------------------------------------------------------
# full-size workloads, sampled outputs, in the configuration bench.py times
# --------------------------------------------------------------------------
def _sample(n, k, seed):
    rng = np.random.default_rng(seed)
    return sorted(rng.choice(n, size=min(k, n), replace=False).tolist())


@pytest.mark.parametrize("name,k", [("qwen7b", 24), ("random_divergence", 12), ("wide_prefix", 16),
                                    ("no_sharing", 12)])
def test_full_size_sampled(name, k):
    s = workloads.by_name(name, seed=0)
    f, ids = build_forest(s)
    leaf_ids = [ids[x] for x in s.leaves]
    Q = s.q(DEV)
    model = oracle.OracleForest(block_tokens=32, pool_blocks=f.cfg.pool_blocks).replay(s)
    rows = _sample(len(leaf_ids), k, seed=len(name))
    src = _kv_source(s)
    o_ref, lse_ref, a_ref = oracle_outputs(model, s.leaves, Q.cpu(), src, rows)
    for flags in (0, tp.TP_DECODE_CUDA_CORE_SMALL, tp.TP_MMA_SYNC, tp.TP_DECODE_TCGEN05):
        O, LSE = f.decode(leaf_ids, Q, flags=flags)
        f.sync()
        check(O, LSE, o_ref, lse_ref, a_ref, rows=rows)
        assert torch.isfinite(O.float()).all() and torch.isfinite(LSE).all()
    f.close()


# --------------------------------------------------------------------------
# randomized sweep: more seeds, head shapes and routing flags
# --------------------------------------------------------------------------
SWEEP_HEADS = [workloads.Heads(4, 1, 64), workloads.Heads(8, 2, 64), workloads.Heads(28, 4, 128),
               workloads.Heads(64, 8, 128), workloads.Heads(16, 16, 128), workloads.Heads(32, 2, 64)]


@pytest.mark.parametrize("seed", range(100, 124))
def test_random_forest_sweep(seed):
    rng = np.random.default_rng(seed)
    heads = SWEEP_HEADS[seed % len(SWEEP_HEADS)]
    s = workloads.random_tree(seed=seed, heads=heads, n_prompts=int(rng.integers(1, 5)),
                              max_depth=int(rng.integers(1, 7)), prompt_range=(1, int(rng.integers(2, 700))),
                              seg_range=(1, int(rng.integers(2, 300))), max_kids=int(rng.integers(1, 5)))
    run_and_compare(s, flags=FLAG_SETS[(seed // len(SWEEP_HEADS)) % len(FLAG_SETS)])
