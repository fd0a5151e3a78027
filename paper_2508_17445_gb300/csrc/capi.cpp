// capi.cpp -- the extern "C" entry points declared in include/treepo.h.
#include <algorithm>
#include <cmath>
#include <cstring>
#include <new>
#include <string>

#include <nvtx3/nvToolsExt.h>

#include "forest.h"

using tp::fail;

namespace tp {

// One NVTX range per attention call, named for the entry point (a profiler
// shows each call's host scheduling and launches under it; without a tool
// attached the push and pop cost a few nanoseconds).
struct CallRange {
    explicit CallRange(const char* name) { nvtxRangePushA(name); }
    ~CallRange() { nvtxRangePop(); }
    CallRange(const CallRange&) = delete;
    CallRange& operator=(const CallRange&) = delete;
};

tp_status cuda_fail(tp_tree* t, cudaError_t e, const char* what) {
    return fail(t, TP_ERR_CUDA, std::string(what) + ": " + cudaGetErrorString(e));
}

tp_status ensure_device_bytes(tp_tree* t, void** ptr, int64_t* cap, int64_t need, const char* what) {
    if (need <= *cap) return TP_OK;
    int64_t want = std::max<int64_t>(need, *cap + *cap / 2);
    if (*ptr) {
        cudaStreamSynchronize(t->stream);
        cudaFree(*ptr);
        *ptr = nullptr;
        *cap = 0;
    }
    cudaError_t e = cudaMalloc(ptr, (size_t)want);
    if (e != cudaSuccess) {
        *ptr = nullptr;
        cudaGetLastError();
        return fail(t, e == cudaErrorMemoryAllocation ? TP_ERR_OOM : TP_ERR_CUDA,
                    std::string(what) + ": " + cudaGetErrorString(e));
    }
    *cap = want;
    return TP_OK;
}

tp_status stage_upload(tp_tree* t, int32_t* dst, const int32_t* src, int64_t words) {
    const int k = t->pinned_next;
    t->pinned_next ^= 1;
    if (t->h_pinned_ev[k] == nullptr) {
        cudaError_t e = cudaEventCreateWithFlags(&t->h_pinned_ev[k], cudaEventDisableTiming);
        if (e != cudaSuccess) return cuda_fail(t, e, "cudaEventCreate");
    }
    cudaError_t e = cudaEventSynchronize(t->h_pinned_ev[k]);  // previous copy out of this buffer done
    if (e != cudaSuccess) return cuda_fail(t, e, "cudaEventSynchronize");
    if (t->h_pinned_cap[k] < words) {
        if (t->h_pinned[k]) cudaFreeHost(t->h_pinned[k]);
        t->h_pinned[k] = nullptr;
        t->h_pinned_cap[k] = 0;
        int64_t want = std::max<int64_t>(words, 1 << 16);
        e = cudaHostAlloc((void**)&t->h_pinned[k], (size_t)want * 4, cudaHostAllocDefault);
        if (e != cudaSuccess) return cuda_fail(t, e, "cudaHostAlloc");
        t->h_pinned_cap[k] = want;
    }
    std::memcpy(t->h_pinned[k], src, (size_t)words * 4);
    e = cudaMemcpyAsync(dst, t->h_pinned[k], (size_t)words * 4, cudaMemcpyHostToDevice, t->stream);
    if (e != cudaSuccess) return cuda_fail(t, e, "host-to-device upload");
    e = cudaEventRecord(t->h_pinned_ev[k], t->stream);
    if (e != cudaSuccess) return cuda_fail(t, e, "cudaEventRecord");
    return TP_OK;
}

// Host half of appending one token to each of nodes[0..n): the checks, a new
// block for every node whose last block is full (*need of them), and the pool
// slot of each new token in t->tok_slots. Nothing changes on failure.
tp_status append_tokens_plan(tp_tree* t, const tp_node* nodes, int32_t n, int64_t* need_out) {
    SchedScratch& X = t->scratch;
    if (X.mark.size() < t->nodes.size()) {
        X.mark.resize(t->nodes.size(), 0);
        X.local.resize(t->nodes.size(), 0);
    }
    if (++X.epoch == 0) {
        std::fill(X.mark.begin(), X.mark.end(), 0u);
        X.epoch = 1;
    }
    const int32_t bt = t->cfg.block_tokens;
    int64_t need = 0;
    for (int32_t i = 0; i < n; ++i) {
        tp_status st = check_live(t, nodes[i], false);
        if (st != TP_OK) return st;
        const Node& nd = t->nodes[(size_t)nodes[i]];
        if (nd.state != 0) return fail(t, TP_ERR_FROZEN, "node " + std::to_string(nodes[i]) + " has been forked");
        if (X.mark[(size_t)nodes[i]] == X.epoch)
            return fail(t, TP_ERR_INVALID_ARG, "node " + std::to_string(nodes[i]) + " is listed twice");
        if (nd.n_tokens >= INT32_MAX / 2) return fail(t, TP_ERR_INVALID_ARG, "node too long");
        X.mark[(size_t)nodes[i]] = X.epoch;
        need += nd.n_tokens % bt == 0;
    }
    if (need > t->pool.free_count())
        return fail(t, TP_ERR_OOM, "pool exhausted: need " + std::to_string(need) + " blocks, " +
                                       std::to_string(t->pool.free_count()) + " free");
    std::vector<int32_t>& slots = t->tok_slots;
    slots.resize((size_t)n);
    for (int32_t i = 0; i < n; ++i) {
        Node& nd = t->nodes[(size_t)nodes[i]];
        if (nd.n_tokens % bt == 0) t->pool.alloc(1, nd.blocks);  // cannot fail: counted above
        slots[(size_t)i] = nd.blocks[(size_t)(nd.n_tokens / bt)] * bt + nd.n_tokens % bt;
    }
    *need_out = need;
    return TP_OK;
}

// Undoes append_tokens_plan's block allocations (before the commit).
void append_tokens_unplan(tp_tree* t, const tp_node* nodes, int32_t n) {
    const int32_t bt = t->cfg.block_tokens;
    for (int32_t i = 0; i < n; ++i) {
        Node& nd = t->nodes[(size_t)nodes[i]];
        if (nd.n_tokens % bt == 0) {
            t->pool.release({nd.blocks.back()});
            nd.blocks.pop_back();
        }
    }
}

void append_tokens_commit(tp_tree* t, const tp_node* nodes, int32_t n, int64_t need) {
    for (int32_t i = 0; i < n; ++i) ++t->nodes[(size_t)nodes[i]].n_tokens;
    ++t->version;
    if (need > 0) ++t->struct_version;
}

// One token step of the rollout's decode loop in one upload and one launch:
// append a token to each of nodes[0..n) with the stand-in activations of
// (seed, pos), Q of the rows into q; and, when the cached decode schedule is
// the one for exactly these nodes and the append stays inside their last
// blocks, the schedule patch the next tp_decode_ex(decode_flags) would apply.
// d_buf: device int32 scratch of at least 4 n words.
tp_status rollout_token_step(tp_tree* t, const tp_node* nodes, int32_t n, int32_t* d_buf, int64_t buf_words,
                             uint64_t seed, int32_t pos, uint16_t* q, uint32_t decode_flags) {
    if (n == 0) return TP_OK;
    int64_t need = 0;
    tp_status st = append_tokens_plan(t, nodes, n, &need);
    if (st != TP_OK) return st;
    const uint32_t key = decode_flags & ~TP_DECODE_NO_CACHE;
    const bool patch = !(decode_flags & TP_DECODE_NO_CACHE) && need == 0 && t->sched_valid &&
                       t->sched_flags == key && t->sched_version == t->version &&
                       t->sched_struct == t->struct_version && t->sched_leaves.size() == (size_t)n &&
                       std::equal(nodes, nodes + n, t->sched_leaves.begin()) &&
                       2 * (int64_t)n + (int64_t)t->sched.leaf_tail.size() <= buf_words;
    append_tokens_commit(t, nodes, n, need);
    const int32_t n_pairs = patch ? patch_schedule(t, t->sched, t->patch_words) : 0;
    std::vector<int32_t>& w = t->scratch.step_words;  // row nodes | pool slots | patch pairs
    w.assign(nodes, nodes + n);
    w.insert(w.end(), t->tok_slots.begin(), t->tok_slots.end());
    if (n_pairs > 0) w.insert(w.end(), t->patch_words.begin(), t->patch_words.begin() + 2 * (int64_t)n_pairs);
    st = (int64_t)w.size() <= buf_words ? stage_upload(t, d_buf, w.data(), (int64_t)w.size())
                                        : fail(t, TP_ERR_INVALID_ARG, "rollout step buffer too small");
    if (st == TP_OK) {
        StepArgs a;
        a.row_node = d_buf;
        a.slots = d_buf + n;
        a.pairs = d_buf + 2 * n;
        a.sched = t->d_sched;
        a.pool = (uint8_t*)t->cfg.pool;
        a.q = q;
        a.seed = seed;
        a.head_bytes = t->cfg.block_tokens * t->cfg.head_dim * 2;
        a.block_bytes = (int64_t)2 * t->cfg.num_kv_heads * a.head_bytes;
        a.hkv = t->cfg.num_kv_heads;
        a.q_width = t->cfg.num_q_heads * t->cfg.head_dim;
        a.pos = pos;
        a.n = n;
        a.n_pairs = n_pairs;
        a.err = t->d_err;
        a.pool_blocks = t->cfg.pool_blocks;
        a.sched_words = (int64_t)t->sched.words.size();
        LaunchTimer timer(t, KK_APPEND);
        cudaError_t e = launch_rollout_step(t->cfg.head_dim, a, t->stream);
        if (e != cudaSuccess) st = cuda_fail(t, e, "rollout step kernel");
    }
    if (st != TP_OK) {  // back to the state before the call; the cached schedule is rebuilt next time
        for (int32_t i = 0; i < n; ++i) --t->nodes[(size_t)nodes[i]].n_tokens;
        append_tokens_unplan(t, nodes, n);
        --t->version;
        if (need > 0) --t->struct_version;
        t->sched_valid = false;
        return st;
    }
    if (patch) t->sched_version = t->version;
    return TP_OK;
}

}  // namespace tp

namespace {

using tp::cuda_fail;
using tp::stage_upload;

thread_local std::string g_create_err;

bool aligned(const void* p, uintptr_t a) { return ((uintptr_t)p % a) == 0; }

// Grow a typed device buffer (counted in elements).
template <typename T>
tp_status ensure_device(tp_tree* t, T*& ptr, int64_t& cap, int64_t need, const char* what) {
    void* p = ptr;
    int64_t bytes = cap * (int64_t)sizeof(T);
    tp_status st = tp::ensure_device_bytes(t, &p, &bytes, need * (int64_t)sizeof(T), what);
    ptr = (T*)p;
    cap = bytes / (int64_t)sizeof(T);
    return st;
}

tp_status run_schedule(tp_tree* t, const tp::Schedule& S, const void* Q, void* O, float* LSE,
                       const int32_t* d_sched = nullptr);

// What a schedule's words index into (checked by the bounds-checked build).
tp::Extents extents_of(const tp_tree* t, const tp::Schedule& S) {
    tp::Extents x;
    x.pool_blocks = t->cfg.pool_blocks;
    x.n_tiles = S.n_tiles;
    x.n_occ = S.n_occ;
    x.n = S.n;
    x.n_slots = S.n_slots;
    x.n_merge = S.n_merge;
    x.hkv = t->cfg.num_kv_heads;
    x.group = t->cfg.num_q_heads / t->cfg.num_kv_heads;
    return x;
}

tp_status upload_schedule(tp_tree* t, const tp::Schedule& s) {
    const int64_t words = (int64_t)s.words.size();
    tp_status st = ensure_device(t, t->d_sched, t->d_sched_cap, words, "schedule buffer");
    if (st != TP_OK) return st;
    return stage_upload(t, t->d_sched, s.words.data(), words);
}

// Bring the cached device schedule up to date after appends that stayed
// inside the listed leaves' last blocks: only their last-tile words change.
tp_status patch_cached_schedule(tp_tree* t) {
    const int32_t n = tp::patch_schedule(t, t->sched, t->patch_words);
    if (n == 0) return TP_OK;
    tp_status st = ensure_device(t, t->d_patch, t->d_patch_cap, 2 * (int64_t)n, "schedule patch buffer");
    if (st != TP_OK) return st;
    st = stage_upload(t, t->d_patch, t->patch_words.data(), 2 * (int64_t)n);
    if (st != TP_OK) return st;
    cudaError_t e = tp::launch_patch(t->d_sched, t->d_patch, n, t->stream, (int64_t)t->sched.words.size(), t->d_err);
    tp::count_kernels(t, tp::KK_DECODE, 1);
    if (e != cudaSuccess) return cuda_fail(t, e, "schedule patch kernel");
    return TP_OK;
}

cudaEvent_t next_event(tp_tree* t) {
    if (t->ev_used == t->ev_pool.size()) {
        cudaEvent_t e = nullptr;
        if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
        t->ev_pool.push_back(e);
    }
    return t->ev_pool[t->ev_used++];
}

}  // namespace

namespace tp {
LaunchTimer::LaunchTimer(tp_tree* t, int kind) : t_(t), kind_(kind) {
    if (!t_->profiling) return;
    cudaEvent_t a = next_event(t_);
    b_ = next_event(t_);
    if (!a || !b_) {
        b_ = nullptr;
        return;
    }
    cudaEventRecord(a, t_->stream);
    index_ = t_->timed.size();
    t_->timed.push_back({kind_, a, b_, 1});
}
LaunchTimer::~LaunchTimer() {
    if (b_) cudaEventRecord(b_, t_->stream);
}
void LaunchTimer::kernels(int n) {
    if (b_) t_->timed[index_].kernels = n;
}
void count_kernels(tp_tree* t, int kind, int n) {
    if (t->profiling) t->untimed[kind] += n;
}
}  // namespace tp

extern "C" {

int64_t tp_pool_bytes(const tp_config* c) {
    if (!c || c->num_kv_heads < 1 || c->head_dim < 1 || c->block_tokens < 1 || c->pool_blocks < 1) return -1;
    return c->pool_blocks * 2 * (int64_t)c->num_kv_heads * c->block_tokens * c->head_dim * 2;
}

tp_status tp_tree_create(const tp_config* cfg, tp_tree** out) {
    if (!out) return TP_ERR_INVALID_ARG;
    *out = nullptr;
    auto bad = [](const char* m) {
        g_create_err = m;
        return TP_ERR_INVALID_ARG;
    };
    if (!cfg) return bad("cfg is NULL");
    if (cfg->num_q_heads < 1 || cfg->num_kv_heads < 1 || cfg->num_q_heads % cfg->num_kv_heads)
        return bad("num_q_heads must be a positive multiple of num_kv_heads");
    if (cfg->head_dim != 64 && cfg->head_dim != 128) return bad("head_dim must be 64 or 128");
    if (cfg->block_tokens != 32) return bad("block_tokens must be 32");
    if (cfg->pool_blocks < 1 || cfg->pool_blocks > tp::kMaxPoolBlocks) return bad("pool_blocks must be in [1, 2^24]");
    if (cfg->pool && !aligned(cfg->pool, 256)) return bad("pool must be 256-byte aligned");
    tp_tree* t = new (std::nothrow) tp_tree();
    if (!t) {
        g_create_err = "out of host memory";
        return TP_ERR_OOM;
    }
    t->cfg = *cfg;
    t->stream = (cudaStream_t)cfg->cuda_stream;
    t->pool.init(cfg->pool_blocks);
    if (cfg->pool) {
        cudaError_t e = cudaMalloc((void**)&t->d_err, 4 * sizeof(int32_t));
        if (e == cudaSuccess) e = cudaMemsetAsync(t->d_err, 0, 4 * sizeof(int32_t), t->stream);
        if (e != cudaSuccess) {
            g_create_err = std::string("device error flag: ") + cudaGetErrorString(e);
            cudaGetLastError();
            if (t->d_err) cudaFree(t->d_err);
            delete t;
            return TP_ERR_CUDA;
        }
    }
    *out = t;
    return TP_OK;
}

tp_status tp_tree_destroy(tp_tree* t) {
    if (!t) return TP_OK;
    if (t->cfg.pool) cudaStreamSynchronize(t->stream);
    if (t->d_err) cudaFree(t->d_err);
    if (t->d_sched) cudaFree(t->d_sched);
    if (t->d_part) cudaFree(t->d_part);
    if (t->d_gather_tiles) cudaFree(t->d_gather_tiles);
    if (t->d_patch) cudaFree(t->d_patch);
    if (t->d_tok_slots) cudaFree(t->d_tok_slots);
    for (cudaEvent_t e : t->ev_pool) cudaEventDestroy(e);
    if (t->ev_fork) cudaEventDestroy(t->ev_fork);
    if (t->ev_join) cudaEventDestroy(t->ev_join);
    if (t->side) cudaStreamDestroy(t->side);
    for (int k = 0; k < 2; ++k) {
        if (t->h_pinned[k]) cudaFreeHost(t->h_pinned[k]);
        if (t->h_pinned_ev[k]) cudaEventDestroy(t->h_pinned_ev[k]);
    }
    for (cudaStream_t s : {t->hp_h2d, t->hp_d2h, t->pf_copy})
        if (s) {
            cudaStreamSynchronize(s);
            cudaStreamDestroy(s);
        }
    for (int k = 0; k < 2; ++k) {
        for (cudaEvent_t e : {t->pf_up[k], t->pf_done[k]})
            if (e) cudaEventDestroy(e);
        if (t->d_pf[k]) cudaFree(t->d_pf[k]);
        if (t->h_pf[k]) cudaFreeHost(t->h_pf[k]);
    }
    for (int k = 0; k < 2; ++k) {
        for (cudaEvent_t e : {t->hp_up[k], t->hp_done[k], t->hp_down[k]})
            if (e) cudaEventDestroy(e);
        for (void* p : {t->hp_q[k], t->hp_o[k], t->hp_lse[k]})
            if (p) cudaFree(p);
    }
    delete t;
    return TP_OK;
}

tp_status tp_set_stream(tp_tree* t, void* stream) {
    if (!t) return TP_ERR_INVALID_ARG;
    t->stream = (cudaStream_t)stream;
    return TP_OK;
}

tp_status tp_add_root(tp_tree* t, tp_node* out) {
    if (!t || !out) return TP_ERR_INVALID_ARG;
    if (t->nodes.size() >= (size_t)INT32_MAX) return fail(t, TP_ERR_OOM, "node ids exhausted");
    t->nodes.emplace_back();
    *out = (tp_node)t->nodes.size() - 1;
    ++t->live_nodes;
    ++t->version;
    ++t->struct_version;
    return TP_OK;
}

tp_status tp_append_segment(tp_tree* t, tp_node node, int32_t n_tokens, const void* K, const void* V) {
    if (!t) return TP_ERR_INVALID_ARG;
    tp_status st = tp::check_live(t, node, false);
    if (st != TP_OK) return st;
    tp::Node& nd = t->nodes[(size_t)node];
    if (nd.state != 0) return fail(t, TP_ERR_FROZEN, "node " + std::to_string(node) + " has been forked");
    if (n_tokens < 0) return fail(t, TP_ERR_INVALID_ARG, "n_tokens < 0");
    if (n_tokens == 0) return TP_OK;
    if ((int64_t)nd.n_tokens + n_tokens > INT32_MAX / 2) return fail(t, TP_ERR_INVALID_ARG, "node too long");
    if (t->cfg.pool) {
        if (!K || !V || !aligned(K, 16) || !aligned(V, 16))
            return fail(t, TP_ERR_INVALID_ARG, "K and V must be non-NULL 16-byte aligned device pointers");
    } else if (K || V) {
        return fail(t, TP_ERR_INVALID_ARG, "metadata-only tree: K and V must be NULL");
    }
    const int32_t bt = t->cfg.block_tokens;
    const int64_t need = ((int64_t)nd.n_tokens + n_tokens + bt - 1) / bt - (int64_t)nd.blocks.size();
    const size_t old_blocks = nd.blocks.size();
    if (need > 0 && !t->pool.alloc(need, nd.blocks))
        return fail(t, TP_ERR_OOM, "pool exhausted: need " + std::to_string(need) + " blocks, " +
                                       std::to_string(t->pool.free_count()) + " free");
    if (t->cfg.pool) {
        const int32_t hkv = t->cfg.num_kv_heads, hd = t->cfg.head_dim;
        tp::AppendArgs a;
        a.pool = (uint8_t*)t->cfg.pool;
        a.head_bytes = bt * hd * 2;
        a.block_bytes = (int64_t)2 * hkv * a.head_bytes;
        a.hkv = hkv;
        a.err = t->d_err;
        a.pool_blocks = t->cfg.pool_blocks;
        const int64_t row_bytes = (int64_t)hkv * hd * 2;
        int64_t pos = nd.n_tokens;
        const int64_t end = (int64_t)nd.n_tokens + n_tokens;
        while (pos < end) {
            const int64_t bi = pos / bt;
            const int64_t stop = std::min<int64_t>(end, (bi + tp::kAppendMaxBlocks) * bt);
            a.first_row = (int32_t)(pos % bt);
            a.n_tokens = (int32_t)(stop - pos);
            const int64_t nb = (stop - 1) / bt - bi + 1;
            for (int64_t b = 0; b < nb; ++b) a.blocks[b] = nd.blocks[(size_t)(bi + b)];
            a.k = (const uint8_t*)K + (pos - nd.n_tokens) * row_bytes;
            a.v = (const uint8_t*)V + (pos - nd.n_tokens) * row_bytes;
            cudaError_t e;
            {
                tp::LaunchTimer timer(t, tp::KK_APPEND);
                e = tp::launch_append(hd, a, t->stream);
            }
            if (e != cudaSuccess) {
                std::vector<int32_t> fresh(nd.blocks.begin() + (long)old_blocks, nd.blocks.end());
                nd.blocks.resize(old_blocks);
                t->pool.release(fresh);
                return cuda_fail(t, e, "append kernel");
            }
            pos = stop;
        }
    }
    nd.n_tokens += n_tokens;
    ++t->version;
    if (need > 0) ++t->struct_version;
    return TP_OK;
}

tp_status tp_append_tokens(tp_tree* t, const tp_node* nodes, int32_t n, const void* K, const void* V) {
    if (!t) return TP_ERR_INVALID_ARG;
    if (n < 0) return fail(t, TP_ERR_INVALID_ARG, "n < 0");
    if (n == 0) return TP_OK;
    if (!nodes) return fail(t, TP_ERR_INVALID_ARG, "nodes is NULL");
    if (t->cfg.pool) {
        if (!K || !V || !aligned(K, 16) || !aligned(V, 16))
            return fail(t, TP_ERR_INVALID_ARG, "K and V must be non-NULL 16-byte aligned device pointers");
    } else if (K || V) {
        return fail(t, TP_ERR_INVALID_ARG, "metadata-only tree: K and V must be NULL");
    }
    int64_t need = 0;
    tp_status st = tp::append_tokens_plan(t, nodes, n, &need);
    if (st != TP_OK) return st;
    if (t->cfg.pool) {
        const int32_t bt = t->cfg.block_tokens;
        st = ensure_device(t, t->d_tok_slots, t->d_tok_slots_cap, n, "token slot buffer");
        if (st == TP_OK) st = stage_upload(t, t->d_tok_slots, t->tok_slots.data(), n);
        if (st == TP_OK) {
            tp::AppendTokensArgs a;
            a.k = K;
            a.v = V;
            a.slots = t->d_tok_slots;
            a.pool = (uint8_t*)t->cfg.pool;
            a.head_bytes = bt * t->cfg.head_dim * 2;
            a.block_bytes = (int64_t)2 * t->cfg.num_kv_heads * a.head_bytes;
            a.hkv = t->cfg.num_kv_heads;
            a.n = n;
            a.err = t->d_err;
            a.pool_blocks = t->cfg.pool_blocks;
            tp::LaunchTimer timer(t, tp::KK_APPEND);
            cudaError_t e = tp::launch_append_tokens(t->cfg.head_dim, a, t->stream);
            if (e != cudaSuccess) st = cuda_fail(t, e, "token append kernel");
        }
        if (st != TP_OK) {
            tp::append_tokens_unplan(t, nodes, n);
            return st;
        }
    }
    tp::append_tokens_commit(t, nodes, n, need);
    return TP_OK;
}

tp_status tp_synth_tokens(tp_tree* t, uint64_t seed, tp_node node, int32_t pos0, int32_t n_tokens, void* K, void* V,
                          void* Q) {
    if (!t) return TP_ERR_INVALID_ARG;
    if (!t->cfg.pool) return fail(t, TP_ERR_INVALID_ARG, "metadata-only tree launches no kernels");
    if (node < 0 || node >= (1 << 28)) return fail(t, TP_ERR_INVALID_ARG, "node key must be in [0, 2^28)");
    if (pos0 < 0 || n_tokens < 0 || (int64_t)pos0 + n_tokens > (1 << 20))
        return fail(t, TP_ERR_INVALID_ARG, "token positions must lie in [0, 2^20)");
    if ((K && !aligned(K, 8)) || (V && !aligned(V, 8)) || (Q && !aligned(Q, 8)))
        return fail(t, TP_ERR_INVALID_ARG, "K, V and Q must be 8-byte aligned device pointers");
    tp::SynthArgs a;
    a.k = (uint16_t*)K;
    a.v = (uint16_t*)V;
    a.q = (uint16_t*)Q;
    a.row_node = nullptr;
    a.seed = seed;
    a.rows = n_tokens;
    a.kv_width = t->cfg.num_kv_heads * t->cfg.head_dim;
    a.q_width = t->cfg.num_q_heads * t->cfg.head_dim;
    a.node0 = node;
    a.pos0 = pos0;
    tp::LaunchTimer timer(t, tp::KK_APPEND);
    cudaError_t e = tp::launch_synth(a, t->stream);
    if (e != cudaSuccess) return cuda_fail(t, e, "synth kernel");
    return TP_OK;
}

int64_t tp_advantage_workspace_bytes(int32_t n_nodes, int32_t n_out) {
    if (n_nodes < 0 || n_out < 0) return -1;
    return tp::advantage_ws_bytes(n_nodes, n_out);
}

tp_status tp_tree_advantage(const int32_t* parent, int32_t n_nodes, const int32_t* leaf, const float* reward,
                            int32_t n_out, float* adv, double* stats, void* workspace, int64_t workspace_bytes,
                            void* cuda_stream) {
    auto bad = [](const char* m) {
        g_create_err = m;
        return TP_ERR_INVALID_ARG;
    };
    if (n_nodes < 0 || n_out < 0) return bad("n_nodes and n_out must be >= 0");
    if (n_out > 0 && (!parent || !leaf || !reward || !adv)) return bad("parent, leaf, reward and adv must be non-NULL");
    if (!workspace || !aligned(workspace, 8) || workspace_bytes < tp::advantage_ws_bytes(n_nodes, n_out))
        return bad("workspace must be 8-byte aligned and hold tp_advantage_workspace_bytes() bytes");
    if (stats && !aligned(stats, 8)) return bad("stats must be 8-byte aligned");
    tp::AdvantageArgs a;
    a.parent = parent;
    a.leaf = leaf;
    a.reward = reward;
    a.adv = adv;
    a.stats = stats;
    a.ws = (uint8_t*)workspace;
    a.n_nodes = n_nodes;
    a.n_out = n_out;
    cudaError_t e = tp::launch_advantage(a, (cudaStream_t)cuda_stream);
    if (e != cudaSuccess) {
        g_create_err = std::string("advantage kernel: ") + cudaGetErrorString(e);
        return TP_ERR_CUDA;
    }
    return TP_OK;
}

tp_status tp_fork(tp_tree* t, tp_node node, int32_t k, tp_node* out_children) {
    if (!t) return TP_ERR_INVALID_ARG;
    tp_status st = tp::check_live(t, node, false);
    if (st != TP_OK) return st;
    if (k < 1) return fail(t, TP_ERR_INVALID_ARG, "fork needs k >= 1");
    if (!out_children) return fail(t, TP_ERR_INVALID_ARG, "out_children is NULL");
    if (t->nodes.size() + (size_t)k > (size_t)INT32_MAX) return fail(t, TP_ERR_OOM, "node ids exhausted");
    const int64_t before = t->nodes[(size_t)node].path_before + t->nodes[(size_t)node].n_tokens;
    for (int32_t c = 0; c < k; ++c) {
        tp::Node child;
        child.parent = node;
        child.path_before = before;
        t->nodes.push_back(std::move(child));
        out_children[c] = (tp_node)t->nodes.size() - 1;
    }
    tp::Node& nd = t->nodes[(size_t)node];
    nd.state = 1;
    nd.kids_live += k;
    t->live_nodes += k;
    ++t->version;
    ++t->struct_version;
    return TP_OK;
}

tp_status tp_prune(tp_tree* t, tp_node leaf) {
    if (!t) return TP_ERR_INVALID_ARG;
    tp_status st = tp::check_live(t, leaf, true);
    if (st != TP_OK) return st;
    int32_t x = leaf;
    while (true) {
        tp::Node& nd = t->nodes[(size_t)x];
        t->pool.release(nd.blocks);
        nd.blocks.clear();
        nd.blocks.shrink_to_fit();
        nd.state = 2;
        --t->live_nodes;
        x = nd.parent;
        if (x == -1) break;
        if (--t->nodes[(size_t)x].kids_live > 0) break;
    }
    ++t->version;
    ++t->struct_version;
    return TP_OK;
}

tp_status tp_decode_ex(tp_tree* t, const tp_node* leaves, int32_t n, const void* Q, void* O, float* LSE,
                       uint32_t flags) {
    const tp::CallRange range("tp_decode_ex");
    if (!t) return TP_ERR_INVALID_ARG;
    if (n < 0) return fail(t, TP_ERR_INVALID_ARG, "n < 0");
    if (n == 0) return TP_OK;
    if (!leaves) return fail(t, TP_ERR_INVALID_ARG, "leaves is NULL");
    if (!t->cfg.pool) return fail(t, TP_ERR_INVALID_ARG, "metadata-only tree cannot decode");
    if (!Q || !O || !LSE || !aligned(Q, 16) || !aligned(O, 16) || !aligned(LSE, 4))
        return fail(t, TP_ERR_INVALID_ARG, "Q/O must be 16-byte and LSE 4-byte aligned device pointers");
    // Schedule cache: reuse the last schedule for the same leaf list and
    // flags; after appends that only filled the leaves' last blocks further
    // (a decode loop appending one token per leaf), patch its tile words.
    const uint32_t key_flags = flags & ~TP_DECODE_NO_CACHE;
    const bool same_call = !(flags & TP_DECODE_NO_CACHE) && t->sched_valid && t->sched_flags == key_flags &&
                           t->sched_leaves.size() == (size_t)n &&
                           std::equal(leaves, leaves + n, t->sched_leaves.begin());
    tp::Schedule& S = t->sched;
    if (same_call && t->sched_version != t->version && t->sched_struct == t->struct_version) {
        tp_status st = patch_cached_schedule(t);
        if (st != TP_OK) {
            t->sched_valid = false;
            return st;
        }
        t->sched_version = t->version;
    } else if (!same_call || t->sched_version != t->version) {
        t->sched_valid = false;
        tp_status st = tp::build_schedule(t, leaves, n, flags, S);
        if (st != TP_OK) return st;
        st = upload_schedule(t, S);
        if (st != TP_OK) return st;
        t->sched_valid = true;
        t->sched_version = t->version;
        t->sched_struct = t->struct_version;
        t->sched_flags = key_flags;
        t->sched_leaves.assign(leaves, leaves + n);
    }
    return run_schedule(t, S, Q, O, LSE);
}

tp_status tp_prefill(tp_tree* t, const tp_node* nodes, const int32_t* n_queries, int32_t n, const void* Q, void* O,
                     float* LSE, uint32_t flags) {
    const tp::CallRange range("tp_prefill");
    if (!t) return TP_ERR_INVALID_ARG;
    if (n < 0) return fail(t, TP_ERR_INVALID_ARG, "n < 0");
    if (n == 0) return TP_OK;
    if (!nodes || !n_queries) return fail(t, TP_ERR_INVALID_ARG, "nodes or n_queries is NULL");
    if (!t->cfg.pool) return fail(t, TP_ERR_INVALID_ARG, "metadata-only tree cannot run attention");
    if (!Q || !O || !LSE || !aligned(Q, 16) || !aligned(O, 16) || !aligned(LSE, 4))
        return fail(t, TP_ERR_INVALID_ARG, "Q/O must be 16-byte and LSE 4-byte aligned device pointers");
    tp::Schedule& S = t->pf_sched;
    tp_status st = tp::build_prefill_schedule(t, nodes, n_queries, n, flags, S);
    if (st != TP_OK) return st;
    if (S.n == 0) return TP_OK;
    // device buffer b: uploaded on the copy stream once the kernels of the
    // call two back (its last reader) are done; the attention waits for it
    cudaError_t e = cudaSuccess;
    if (!t->pf_copy) {
        e = cudaStreamCreateWithFlags(&t->pf_copy, cudaStreamNonBlocking);
        for (int k = 0; k < 2 && e == cudaSuccess; ++k)
            for (cudaEvent_t* ev : {&t->pf_up[k], &t->pf_done[k]})
                if (e == cudaSuccess) e = cudaEventCreateWithFlags(ev, cudaEventDisableTiming);
        if (e != cudaSuccess) return cuda_fail(t, e, "prefill upload stream");
    }
    const int b = (int)(t->pf_calls & 1);
    const int64_t words = (int64_t)S.words.size();
    if (t->d_pf_cap[b] < words) {  // grow: the buffer's last reader must be done before it is freed
        e = cudaEventSynchronize(t->pf_done[b]);
        if (e != cudaSuccess) return cuda_fail(t, e, "cudaEventSynchronize");
        st = ensure_device(t, t->d_pf[b], t->d_pf_cap[b], words, "prefill schedule buffer");
        if (st != TP_OK) return st;
    }
    e = cudaEventSynchronize(t->pf_up[b]);  // the pinned buffer's previous upload has left it
    if (e != cudaSuccess) return cuda_fail(t, e, "cudaEventSynchronize");
    if (t->h_pf_cap[b] < words) {
        if (t->h_pf[b]) cudaFreeHost(t->h_pf[b]);
        t->h_pf[b] = nullptr;
        t->h_pf_cap[b] = 0;
        e = cudaHostAlloc((void**)&t->h_pf[b], (size_t)words * 4, cudaHostAllocDefault);
        if (e != cudaSuccess) return cuda_fail(t, e, "cudaHostAlloc");
        t->h_pf_cap[b] = words;
    }
    std::memcpy(t->h_pf[b], S.words.data(), (size_t)words * 4);
    e = cudaStreamWaitEvent(t->pf_copy, t->pf_done[b], 0);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(t->d_pf[b], t->h_pf[b], (size_t)words * 4, cudaMemcpyHostToDevice, t->pf_copy);
    if (e == cudaSuccess) e = cudaEventRecord(t->pf_up[b], t->pf_copy);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(t->stream, t->pf_up[b], 0);
    if (e != cudaSuccess) return cuda_fail(t, e, "prefill schedule upload");
    st = run_schedule(t, S, Q, O, LSE, t->d_pf[b]);
    if (st != TP_OK) return st;
    e = cudaEventRecord(t->pf_done[b], t->stream);
    if (e != cudaSuccess) return cuda_fail(t, e, "cudaEventRecord");
    ++t->pf_calls;
    return TP_OK;
}

}  // extern "C"

namespace {
// One host-buffer call: upload Q into staging slot b once the attention that
// last read that slot has finished, run the attention there once the upload
// has landed and the slot's previous results have been downloaded, then
// download O and LSE. Consecutive calls alternate slots, so a call's upload
// and download overlap the neighbouring calls' attention.
template <typename Run>
tp_status run_host(tp_tree* t, int64_t q_bytes, int64_t o_bytes, int64_t lse_bytes, const void* Qh, void* Oh,
                   float* Lh, Run run) {
    cudaError_t e = cudaSuccess;
    if (!t->hp_h2d) {
        e = cudaStreamCreateWithFlags(&t->hp_h2d, cudaStreamNonBlocking);
        if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&t->hp_d2h, cudaStreamNonBlocking);
        for (int k = 0; k < 2 && e == cudaSuccess; ++k)
            for (cudaEvent_t* ev : {&t->hp_up[k], &t->hp_done[k], &t->hp_down[k]})
                if (e == cudaSuccess) e = cudaEventCreateWithFlags(ev, cudaEventDisableTiming);
        if (e != cudaSuccess) return cuda_fail(t, e, "host-buffer streams");
    }
    const int b = (int)(t->hp_calls & 1);
    if (q_bytes > t->hp_q_cap[b] || o_bytes > t->hp_o_cap[b] || lse_bytes > t->hp_lse_cap[b]) {
        // a slot grows: no copy of the other calls may still use it
        e = cudaStreamSynchronize(t->hp_h2d);
        if (e == cudaSuccess) e = cudaStreamSynchronize(t->hp_d2h);
        if (e != cudaSuccess) return cuda_fail(t, e, "host-buffer streams");
    }
    tp_status st = tp::ensure_device_bytes(t, &t->hp_q[b], &t->hp_q_cap[b], q_bytes, "query staging");
    if (st == TP_OK) st = tp::ensure_device_bytes(t, &t->hp_o[b], &t->hp_o_cap[b], o_bytes, "output staging");
    if (st == TP_OK) st = tp::ensure_device_bytes(t, &t->hp_lse[b], &t->hp_lse_cap[b], lse_bytes, "LSE staging");
    if (st != TP_OK) return st;
    e = cudaStreamWaitEvent(t->hp_h2d, t->hp_done[b], 0);
    if (e == cudaSuccess) e = cudaMemcpyAsync(t->hp_q[b], Qh, (size_t)q_bytes, cudaMemcpyHostToDevice, t->hp_h2d);
    if (e == cudaSuccess) e = cudaEventRecord(t->hp_up[b], t->hp_h2d);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(t->stream, t->hp_up[b], 0);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(t->stream, t->hp_down[b], 0);
    if (e != cudaSuccess) return cuda_fail(t, e, "query upload");
    st = run(t->hp_q[b], t->hp_o[b], (float*)t->hp_lse[b]);
    if (st != TP_OK) return st;
    e = cudaEventRecord(t->hp_done[b], t->stream);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(t->hp_d2h, t->hp_done[b], 0);
    if (e == cudaSuccess) e = cudaMemcpyAsync(Oh, t->hp_o[b], (size_t)o_bytes, cudaMemcpyDeviceToHost, t->hp_d2h);
    if (e == cudaSuccess) e = cudaMemcpyAsync(Lh, t->hp_lse[b], (size_t)lse_bytes, cudaMemcpyDeviceToHost, t->hp_d2h);
    if (e == cudaSuccess) e = cudaEventRecord(t->hp_down[b], t->hp_d2h);
    if (e != cudaSuccess) return cuda_fail(t, e, "result download");
    ++t->hp_calls;
    return TP_OK;
}
}  // namespace

extern "C" {

tp_status tp_decode_host(tp_tree* t, const tp_node* leaves, int32_t n, const void* Q_host, void* O_host,
                         float* LSE_host, uint32_t flags) {
    const tp::CallRange range("tp_decode_host");
    if (!t) return TP_ERR_INVALID_ARG;
    if (n < 0) return fail(t, TP_ERR_INVALID_ARG, "n < 0");
    if (n == 0) return TP_OK;
    if (!leaves) return fail(t, TP_ERR_INVALID_ARG, "leaves is NULL");
    if (!t->cfg.pool) return fail(t, TP_ERR_INVALID_ARG, "metadata-only tree cannot decode");
    if (!Q_host || !O_host || !LSE_host) return fail(t, TP_ERR_INVALID_ARG, "Q/O/LSE host pointer is NULL");
    const int64_t row = (int64_t)t->cfg.num_q_heads * t->cfg.head_dim;
    return run_host(t, n * row * 2, n * row * 2, (int64_t)n * t->cfg.num_q_heads * 4, Q_host, O_host, LSE_host,
                    [&](const void* Q, void* O, float* LSE) { return tp_decode_ex(t, leaves, n, Q, O, LSE, flags); });
}

tp_status tp_prefill_host(tp_tree* t, const tp_node* nodes, const int32_t* n_queries, int32_t n, const void* Q_host,
                          void* O_host, float* LSE_host, uint32_t flags) {
    const tp::CallRange range("tp_prefill_host");
    if (!t) return TP_ERR_INVALID_ARG;
    if (n < 0) return fail(t, TP_ERR_INVALID_ARG, "n < 0");
    if (n == 0) return TP_OK;
    if (!nodes || !n_queries) return fail(t, TP_ERR_INVALID_ARG, "nodes or n_queries is NULL");
    if (!t->cfg.pool) return fail(t, TP_ERR_INVALID_ARG, "metadata-only tree cannot run attention");
    if (!Q_host || !O_host || !LSE_host) return fail(t, TP_ERR_INVALID_ARG, "Q/O/LSE host pointer is NULL");
    int64_t total = 0;
    for (int32_t i = 0; i < n; ++i) {
        if (n_queries[i] < 0) return fail(t, TP_ERR_INVALID_ARG, "n_queries[i] < 0");
        total += n_queries[i];
    }
    if (total == 0) return TP_OK;
    const int64_t row = (int64_t)t->cfg.num_q_heads * t->cfg.head_dim;
    return run_host(t, total * row * 2, total * row * 2, total * t->cfg.num_q_heads * 4, Q_host, O_host, LSE_host,
                    [&](const void* Q, void* O, float* LSE) {
                        return tp_prefill(t, nodes, n_queries, n, Q, O, LSE, flags);
                    });
}

tp_status tp_debug_prefill_schedule(tp_tree* t, const tp_node* nodes, const int32_t* n_queries, int32_t n,
                                    uint32_t flags, int32_t* buf, int64_t cap, int64_t* len) {
    if (!t || !len) return TP_ERR_INVALID_ARG;
    if (n < 0 || (n > 0 && (!nodes || !n_queries))) return fail(t, TP_ERR_INVALID_ARG, "bad node list");
    tp::Schedule S;
    tp_status st = tp::build_prefill_schedule(t, nodes, n_queries, n, flags, S);
    if (st != TP_OK) return st;
    *len = (int64_t)S.words.size();
    if (cap < *len) return cap == 0 ? TP_OK : fail(t, TP_ERR_INVALID_ARG, "buffer too small");
    if (!buf) return fail(t, TP_ERR_INVALID_ARG, "buf is NULL");
    std::memcpy(buf, S.words.data(), S.words.size() * 4);
    return TP_OK;
}

}  // extern "C"

namespace {
// Launch the attention and merge kernels of a schedule already on the
// device (at d_sched; the decode cache's t->d_sched when null).
tp_status run_schedule(tp_tree* t, const tp::Schedule& S, const void* Q, void* O, float* LSE, const int32_t* d_sched) {
    if (!d_sched) d_sched = t->d_sched;
    const int32_t hq = t->cfg.num_q_heads, hd = t->cfg.head_dim;
    const int64_t part_floats = (int64_t)S.n_slots * hq * (hd + 1);
    tp_status st = ensure_device(t, t->d_part, t->d_part_cap, std::max<int64_t>(part_floats, 1), "partial buffer");
    if (st != TP_OK) return st;

    tp::DecodeArgs a;
    if (S.prefill) {
        a.unit_pos = d_sched + S.off_unit_pos;
        a.vis = d_sched + S.off_vis;
        a.out = (uint16_t*)O;
        a.out_lse = LSE;
    }
    a.units = d_sched + S.off_units;
    a.tiles = d_sched + S.off_tiles;
    a.occ = d_sched + S.off_occ;
    a.q = (const uint16_t*)Q;
    a.pool = (const uint8_t*)t->cfg.pool;
    a.part_o = t->d_part;
    a.part_lse = t->d_part + (int64_t)S.n_slots * hq * hd;
    a.err = t->d_err;
    a.counters = t->d_err + 1;
    a.counter = nullptr;
    a.n_tc_units = S.n_tc;
    a.n_tensor_units = S.n_tensor;
    a.unit_begin = a.unit_end = 0;
    a.head_bytes = t->cfg.block_tokens * hd * 2;
    a.block_bytes = (int64_t)2 * t->cfg.num_kv_heads * a.head_bytes;
    a.n_units = S.n_units;
    a.hq = hq;
    a.hkv = t->cfg.num_kv_heads;
    a.group = hq / t->cfg.num_kv_heads;
    a.qk_scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)hd));
    a.kv_read_once = S.kv_read_once ? 1 : 0;
    a.ext = extents_of(t, S);
    cudaError_t e = cudaSuccess;
    if (S.n_tc > 0 && S.n_units > S.n_tc && !t->side) {  // concurrent tcgen05 units need a second stream
        e = cudaStreamCreateWithFlags(&t->side, cudaStreamNonBlocking);
        if (e == cudaSuccess) e = cudaEventCreateWithFlags(&t->ev_fork, cudaEventDisableTiming);
        if (e == cudaSuccess) e = cudaEventCreateWithFlags(&t->ev_join, cudaEventDisableTiming);
        if (e != cudaSuccess) return cuda_fail(t, e, "side stream");
    }
    if (a.n_units > 0) {
        tp::LaunchTimer timer(t, tp::KK_DECODE);
        e = tp::launch_decode(hd, a, t->stream, t->side, t->ev_fork, t->ev_join);
        timer.kernels((S.n_tc > 0) + (S.n_tensor > 0) + (S.n_units > S.n_tc + S.n_tensor));
    }
    if (e != cudaSuccess) return cuda_fail(t, e, "decode kernel");

    tp::MergeArgs m;
    m.merge_off = d_sched + S.off_merge_off;
    m.merge_slot = d_sched + S.off_merge_slot;
    m.merge_rec = S.off_merge_rec ? d_sched + S.off_merge_rec : nullptr;
    m.part_o = a.part_o;
    m.part_lse = a.part_lse;
    m.out = (uint16_t*)O;
    m.lse = LSE;
    m.counters = t->d_err + 1;
    m.err = t->d_err;
    m.n_merge = S.n_merge;
    m.n_slots = S.n_slots;
    m.n = S.n_merge > 0 ? S.n : 0;  // 0: every row was written by its only unit; only re-arm the counters
    m.hq = hq;
    {
        tp::LaunchTimer timer(t, tp::KK_MERGE);
        e = tp::launch_merge(hd, m, t->stream);
    }
    if (e != cudaSuccess) return cuda_fail(t, e, "merge kernel");
    return TP_OK;
}
}  // namespace

extern "C" {

tp_status tp_decode_noalloc(tp_tree* t, const tp_node* leaves, int32_t n, const void* Q, void* O, float* LSE,
                            uint32_t flags) {
    const tp::CallRange range("tp_decode_noalloc");
    if (!t) return TP_ERR_INVALID_ARG;
    if (n < 0) return fail(t, TP_ERR_INVALID_ARG, "n < 0");
    if (n == 0) return TP_OK;
    if (!leaves) return fail(t, TP_ERR_INVALID_ARG, "leaves is NULL");
    if (!t->cfg.pool) return fail(t, TP_ERR_INVALID_ARG, "metadata-only tree cannot decode");
    if (!Q || !O || !LSE || !aligned(Q, 16) || !aligned(O, 16) || !aligned(LSE, 4))
        return fail(t, TP_ERR_INVALID_ARG, "Q/O must be 16-byte and LSE 4-byte aligned device pointers");
    // The schedule is uploaded from a host vector that dies on return: a
    // captured copy node would read it again on every replay. Refuse capture.
    cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
    cudaError_t ce = cudaStreamIsCapturing(t->stream, &cap);
    if (ce != cudaSuccess) return cuda_fail(t, ce, "stream capture query");
    if (cap != cudaStreamCaptureStatusNone)
        return fail(t, TP_ERR_INVALID_ARG, "tp_decode_noalloc cannot run while its stream is being captured");
    tp::Schedule S;  // host-side only; the tree's schedule cache is left alone
    tp_status st = tp::build_schedule(t, leaves, n, flags & ~TP_DECODE_NO_CACHE, S);
    if (st != TP_OK) return st;
    const int32_t hq = t->cfg.num_q_heads, hd = t->cfg.head_dim;
    const int64_t sched_bytes = ((int64_t)S.words.size() * 4 + 255) / 256 * 256;
    const int64_t part_bytes = (int64_t)S.n_slots * hq * (hd + 1) * 4;
    if (sched_bytes + part_bytes > TP_NOALLOC_SCRATCH_BYTES)
        return fail(t, TP_ERR_OOM,
                    "tp_decode_noalloc needs " + std::to_string(sched_bytes + part_bytes) +
                        " bytes of static scratch; the library holds " + std::to_string(TP_NOALLOC_SCRATCH_BYTES) +
                        " (decode fewer leaves per call, or use tp_decode_ex)");
    void* base = nullptr;
    cudaError_t e = tp::noalloc_scratch(&base);
    if (e != cudaSuccess) return cuda_fail(t, e, "static scratch address");
    int32_t* d_sched = (int32_t*)base;
    float* d_part = (float*)((uint8_t*)base + sched_bytes);
    e = cudaMemcpyAsync(d_sched, S.words.data(), S.words.size() * 4, cudaMemcpyHostToDevice, t->stream);
    if (e != cudaSuccess) return cuda_fail(t, e, "schedule upload");
    e = cudaMemsetAsync(t->d_err + 1, 0, 3 * sizeof(int32_t), t->stream);  // unit counters start at zero
    if (e != cudaSuccess) return cuda_fail(t, e, "counter reset");

    tp::DecodeArgs a;
    a.units = d_sched + S.off_units;
    a.tiles = d_sched + S.off_tiles;
    a.occ = d_sched + S.off_occ;
    a.q = (const uint16_t*)Q;
    a.pool = (const uint8_t*)t->cfg.pool;
    a.part_o = d_part;
    a.part_lse = d_part + (int64_t)S.n_slots * hq * hd;
    a.err = t->d_err;
    a.counters = t->d_err + 1;
    a.counter = nullptr;
    a.n_tc_units = S.n_tc;
    a.n_tensor_units = S.n_tensor;
    a.unit_begin = a.unit_end = 0;
    a.head_bytes = t->cfg.block_tokens * hd * 2;
    a.block_bytes = (int64_t)2 * t->cfg.num_kv_heads * a.head_bytes;
    a.n_units = S.n_units;
    a.hq = hq;
    a.hkv = t->cfg.num_kv_heads;
    a.group = hq / t->cfg.num_kv_heads;
    a.qk_scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)hd));
    a.kv_read_once = S.kv_read_once ? 1 : 0;
    a.ext = extents_of(t, S);
    e = tp::launch_decode(hd, a, t->stream);
    if (e != cudaSuccess) return cuda_fail(t, e, "decode kernel");
    tp::MergeArgs m;
    m.merge_off = d_sched + S.off_merge_off;
    m.merge_slot = d_sched + S.off_merge_slot;
    m.merge_rec = S.off_merge_rec ? d_sched + S.off_merge_rec : nullptr;
    m.part_o = a.part_o;
    m.part_lse = a.part_lse;
    m.out = (uint16_t*)O;
    m.lse = LSE;
    m.counters = t->d_err + 1;
    m.err = t->d_err;
    m.n_merge = S.n_merge;
    m.n_slots = S.n_slots;
    m.n = n;
    m.hq = hq;
    e = tp::launch_merge(hd, m, t->stream);
    if (e != cudaSuccess) return cuda_fail(t, e, "merge kernel");
    return TP_OK;
}

tp_status tp_decode(tp_tree* t, const tp_node* leaves, int32_t n, const void* Q, void* O, float* LSE) {
    return tp_decode_ex(t, leaves, n, Q, O, LSE, 0u);
}

tp_status tp_profile_start(tp_tree* t) {
    if (!t) return TP_ERR_INVALID_ARG;
    if (!t->cfg.pool) return fail(t, TP_ERR_INVALID_ARG, "metadata-only tree launches no kernels");
    cudaError_t e = cudaStreamSynchronize(t->stream);  // recycled events must be idle
    if (e != cudaSuccess) return cuda_fail(t, e, "cudaStreamSynchronize");
    t->timed.clear();
    t->ev_used = 0;
    for (int64_t& k : t->untimed) k = 0;
    t->profiling = true;
    return TP_OK;
}

tp_status tp_profile_stop(tp_tree* t, tp_kernel_times* out) {
    if (!t || !out) return TP_ERR_INVALID_ARG;
    t->profiling = false;
    std::memset(out, 0, sizeof *out);
    if (!t->cfg.pool) return TP_OK;
    cudaError_t e = cudaStreamSynchronize(t->stream);
    if (e != cudaSuccess) return cuda_fail(t, e, "cudaStreamSynchronize");
    for (const auto& x : t->timed) {
        float ms = 0.f;
        e = cudaEventElapsedTime(&ms, x.a, x.b);
        if (e != cudaSuccess) return cuda_fail(t, e, "cudaEventElapsedTime");
        out->launches[x.kind] += x.kernels;
        out->milliseconds[x.kind] += ms;
    }
    for (int k = 0; k < TP_KERNEL_KINDS; ++k) {
        out->launches[k] += t->untimed[k];
        t->untimed[k] = 0;
    }
    t->timed.clear();
    t->ev_used = 0;
    return TP_OK;
}

tp_status tp_debug_wait_probe(tp_tree* t, int64_t limit_ns) {
    if (!t) return TP_ERR_INVALID_ARG;
    if (!t->cfg.pool) return fail(t, TP_ERR_INVALID_ARG, "metadata-only tree launches no kernels");
    if (limit_ns < 1000 || limit_ns > 1000000000) return fail(t, TP_ERR_INVALID_ARG, "limit_ns must lie in [1e3, 1e9]");
    cudaError_t e = tp::launch_wait_probe(t->d_err, (uint64_t)limit_ns, t->stream);
    if (e != cudaSuccess) return cuda_fail(t, e, "wait probe kernel");
    return TP_OK;
}

tp_status tp_sync(tp_tree* t) {
    if (!t) return TP_ERR_INVALID_ARG;
    if (!t->cfg.pool) return TP_OK;
    cudaError_t e = cudaStreamSynchronize(t->stream);
    if (e == cudaSuccess && t->hp_h2d) e = cudaStreamSynchronize(t->hp_h2d);
    if (e == cudaSuccess && t->hp_d2h) e = cudaStreamSynchronize(t->hp_d2h);
    if (e != cudaSuccess) return cuda_fail(t, e, "cudaStreamSynchronize");
    int32_t flag = 0;
    e = cudaMemcpy(&flag, t->d_err, sizeof flag, cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(t, e, "error flag read");
    if (flag) {
        cudaMemset(t->d_err, 0, sizeof(int32_t));
        std::string what;
        if (flag & tp::kErrBounds) what = "an index failed its bounds check (the access was skipped)";
        if (flag & ~tp::kErrBounds) what += std::string(what.empty() ? "" : "; ") + "a kernel gave up a bounded wait";
        return fail(t, TP_ERR_DEVICE, what + " (flag " + std::to_string(flag) + ")");
    }
    return TP_OK;
}

const char* tp_last_error(tp_tree* t) { return t ? t->err.c_str() : g_create_err.c_str(); }

tp_status tp_get_node_info(tp_tree* t, tp_node node, tp_node_info* out) {
    if (!t || !out) return TP_ERR_INVALID_ARG;
    if (node < 0 || node >= (tp_node)t->nodes.size()) return fail(t, TP_ERR_BAD_NODE, "unknown node id");
    const tp::Node& nd = t->nodes[(size_t)node];
    out->parent = nd.parent;
    out->state = nd.state;
    out->n_tokens = nd.n_tokens;
    out->n_live_children = nd.kids_live;
    out->path_tokens = nd.path_before + nd.n_tokens;
    return TP_OK;
}

tp_status tp_get_stats(tp_tree* t, tp_stats* out) {
    if (!t || !out) return TP_ERR_INVALID_ARG;
    out->pool_blocks = t->pool.size();
    out->free_blocks = t->pool.free_count();
    out->live_nodes = t->live_nodes;
    out->total_nodes = (int64_t)t->nodes.size();
    return TP_OK;
}

tp_status tp_debug_path(tp_tree* t, tp_node leaf, int64_t* slots, int64_t cap, int64_t* n) {
    if (!t || !n) return TP_ERR_INVALID_ARG;
    tp_status st = tp::check_live(t, leaf, true);
    if (st != TP_OK) return st;
    const tp::Node& nd = t->nodes[(size_t)leaf];
    const int64_t len = nd.path_before + nd.n_tokens;
    *n = len;
    if (cap < len || (len && !slots)) return fail(t, TP_ERR_INVALID_ARG, "slots buffer too small");
    std::vector<int32_t> tiles;
    tp::path_tiles(t, leaf, tiles);
    const int32_t bt = t->cfg.block_tokens;
    int64_t k = 0;
    for (int32_t w : tiles) {
        const int64_t blk = w >> tp::kTileValidBits;
        const int32_t valid = (w & ((1 << tp::kTileValidBits) - 1)) + 1;
        for (int32_t r = 0; r < valid; ++r) slots[k++] = blk * bt + r;
    }
    return TP_OK;
}

tp_status tp_debug_gather(tp_tree* t, tp_node leaf, void* K_out, void* V_out, int64_t cap_tokens, int64_t* n) {
    if (!t || !n) return TP_ERR_INVALID_ARG;
    tp_status st = tp::check_live(t, leaf, true);
    if (st != TP_OK) return st;
    if (!t->cfg.pool) return fail(t, TP_ERR_INVALID_ARG, "metadata-only tree has no device pool");
    const tp::Node& nd = t->nodes[(size_t)leaf];
    const int64_t len = nd.path_before + nd.n_tokens;
    *n = len;
    if (cap_tokens < len) return fail(t, TP_ERR_INVALID_ARG, "output buffers too small");
    if (len == 0) return TP_OK;
    if (!K_out || !V_out || !aligned(K_out, 16) || !aligned(V_out, 16))
        return fail(t, TP_ERR_INVALID_ARG, "K_out/V_out must be 16-byte aligned device pointers");
    std::vector<int32_t> tiles;
    tp::path_tiles(t, leaf, tiles);
    st = ensure_device(t, t->d_gather_tiles, t->d_gather_cap, (int64_t)tiles.size(), "gather tiles");
    if (st != TP_OK) return st;
    cudaError_t e = cudaMemcpyAsync(t->d_gather_tiles, tiles.data(), tiles.size() * 4, cudaMemcpyHostToDevice, t->stream);
    if (e != cudaSuccess) return cuda_fail(t, e, "gather tile upload");
    tp::GatherArgs a;
    a.tiles = t->d_gather_tiles;
    a.pool = (const uint8_t*)t->cfg.pool;
    a.k_out = K_out;
    a.v_out = V_out;
    a.head_bytes = t->cfg.block_tokens * t->cfg.head_dim * 2;
    a.block_bytes = (int64_t)2 * t->cfg.num_kv_heads * a.head_bytes;
    a.hkv = t->cfg.num_kv_heads;
    a.n_tiles = (int32_t)tiles.size();
    a.block_tokens = t->cfg.block_tokens;
    a.err = t->d_err;
    a.pool_blocks = t->cfg.pool_blocks;
    {
        tp::LaunchTimer timer(t, tp::KK_GATHER);
        e = tp::launch_gather(t->cfg.head_dim, a, len, t->stream);
    }
    if (e != cudaSuccess) return cuda_fail(t, e, "gather kernel");
    e = cudaStreamSynchronize(t->stream);  // the host tile list must outlive the copy
    if (e != cudaSuccess) return cuda_fail(t, e, "gather sync");
    return TP_OK;
}

tp_status tp_debug_check_schedule(tp_tree* t, const int32_t* w, int64_t n_words, int64_t* violations) {
    if (!t || !violations) return TP_ERR_INVALID_ARG;
    if (!w || n_words < tp::kSchedHeaderWords || w[0] != tp::kSchedMagic)
        return fail(t, TP_ERR_INVALID_ARG, "not a schedule (short buffer or bad magic)");
    const int32_t n_units = w[1], n_tiles = w[2], n_occ = w[3], n = w[4], n_slots = w[5], n_merge = w[6];
    const int32_t n_tensor = w[8], n_tc = w[9];
    const bool prefill = w[10] == 1;
    if (n_units < 0 || n_tiles < 0 || n_occ < 0 || n < 0 || n_slots < 0 || n_merge < 0 || n_tensor < 0 || n_tc < 0 ||
        (int64_t)n_tc + n_tensor > n_units)
        return fail(t, TP_ERR_INVALID_ARG, "bad schedule header");
    const int64_t off_units = tp::kSchedHeaderWords, off_tiles = off_units + (int64_t)n_units * tp::kUnitWords;
    const int64_t off_occ = off_tiles + n_tiles, off_moff = off_occ + n_occ, off_mslot = off_moff + n + 1;
    const int64_t off_mrec = off_mslot + n_merge + (prefill ? (int64_t)n_units + n : 0);
    const bool has_rec = w[11] == tp::kMergeRecWords;
    if (w[11] != (prefill ? 0 : tp::kMergeRecWords))
        return fail(t, TP_ERR_INVALID_ARG, "bad schedule header (merge records)");
    const int64_t end = off_mrec + (has_rec ? (int64_t)n * tp::kMergeRecWords : 0);
    if (n_words < end) return fail(t, TP_ERR_INVALID_ARG, "schedule shorter than its header says");
    tp::Extents x;
    x.pool_blocks = t->cfg.pool_blocks;
    x.n_tiles = n_tiles;
    x.n_occ = n_occ;
    x.n = n;
    x.n_slots = n_slots;
    x.n_merge = n_merge;
    x.hkv = t->cfg.num_kv_heads;
    x.group = t->cfg.num_q_heads / t->cfg.num_kv_heads;
    int64_t bad[5] = {0, 0, 0, 0, 0};  // units, tile words, occurrence entries, merge ranges, merge slots
    for (int32_t k = 0; k < n_units; ++k) {
        const int32_t* u = w + off_units + (int64_t)k * tp::kUnitWords;
        // launch order: tcgen05 units, then mma.sync, then CUDA-core units
        const int32_t kind = k < n_tc ? tp::KIND_TC : k < n_tc + n_tensor ? tp::KIND_TENSOR : tp::KIND_CUDA_CORE;
        bad[0] += !(u[tp::U_KIND] == kind &&
                    tp::unit_ok(u[tp::U_TILE_OFF], u[tp::U_N_TILES], u[tp::U_OCC_OFF], u[tp::U_ROW0], u[tp::U_N_ROWS],
                                u[tp::U_SLOT_BASE], u[tp::U_KVH], tp::unit_rows_limit(kind), prefill, x));
    }
    for (int64_t k = 0; k < n_tiles; ++k) bad[1] += !tp::tile_word_ok(w[off_tiles + k], x.pool_blocks);
    for (int64_t k = 0; k < n_occ; ++k) bad[2] += !tp::in_range(w[off_occ + k], n);
    for (int32_t i = 0; i < n; ++i) bad[3] += !tp::merge_range_ok(w[off_moff + i], w[off_moff + i + 1], n_merge);
    for (int64_t k = 0; k < n_merge; ++k) bad[4] += !tp::in_range(w[off_mslot + k], n_slots);
    // merge records: the count of the CSR range (or -1 past 15) and its slots
    for (int32_t i = 0; has_rec && i < n; ++i) {
        const int32_t* r = w + off_mrec + (int64_t)i * tp::kMergeRecWords;
        const int64_t beg = w[off_moff + i], cnt = (int64_t)w[off_moff + i + 1] - beg;
        const bool range_ok = tp::merge_range_ok(w[off_moff + i], w[off_moff + i + 1], n_merge);
        if (r[0] == -1 ? cnt < tp::kMergeRecWords - 1 : (r[0] < 0 || r[0] >= tp::kMergeRecWords || r[0] != cnt)) {
            ++bad[3];
            continue;
        }
        for (int32_t k = 0; k < r[0]; ++k)
            bad[4] += !tp::in_range(r[1 + k], n_slots) || !range_ok || r[1 + k] != w[off_mslot + beg + k];
    }
    std::memcpy(violations, bad, sizeof bad);
    return TP_OK;
}

tp_status tp_debug_schedule(tp_tree* t, const tp_node* leaves, int32_t n, uint32_t flags, int32_t* buf, int64_t cap,
                            int64_t* len) {
    if (!t || !len) return TP_ERR_INVALID_ARG;
    if (n < 0 || (n > 0 && !leaves)) return fail(t, TP_ERR_INVALID_ARG, "bad leaf list");
    tp::Schedule S;
    tp_status st = tp::build_schedule(t, leaves, n, flags, S);
    if (st != TP_OK) return st;
    *len = (int64_t)S.words.size();
    if (cap < *len) return cap == 0 ? TP_OK : fail(t, TP_ERR_INVALID_ARG, "buffer too small");
    if (!buf) return fail(t, TP_ERR_INVALID_ARG, "buf is NULL");
    std::memcpy(buf, S.words.data(), S.words.size() * 4);
    return TP_OK;
}

}  // extern "C"
