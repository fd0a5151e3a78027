// rollout.cpp -- segment-level tree sampling (Sec. 2.2, Algorithm 1) driven
// through the tree API, with a synthetic stand-in for the language model, and
// the probability-based branching assignment (Sec. 4.6).
//
// One loop pass: every queued path generates one segment (Inference), each
// segment either finishes its trajectory (an output), fails (early stop:
// the path is pruned at once) or continues; the continuing paths of each
// query are forked so that the query has min(b0 * N^j, w - outputs) paths at
// depth j (branching budget transfer); a query left with no path and fewer
// than w outputs re-spawns one path from a random segment boundary of one
// of its finished candidates (depth-first-search fallback).
//
// Stand-in model. Every decision is a SplitMix64 draw addressed by the node
// id and token index (splitmix.h), so a run is a pure function of its
// parameters: segment length (a token is EOS with probability p_eos), token
// log-probabilities kappa * ln(1 - u) with a per-segment scale kappa in
// [0, 2), "boxed answer" and "repetition" flags per segment, and the reward
// of a boxed trajectory. K, V and Q of every token are bf16 draws of the
// same generator. With decode on, each generated token is appended to its
// path (tp_append_tokens) and the paths still generating run decode
// attention over their root-to-leaf paths (tp_decode_ex), as an inference
// engine's attention does once per token.
#include <algorithm>
#include <cmath>
#include <cstring>
#include <vector>

#include "forest.h"
#include "splitmix.h"

namespace tp {

tp_status branch_split(const double* logp, int32_t n, int32_t budget, int32_t policy, double temperature,
                       int32_t* out, std::vector<double>& frac, std::vector<int32_t>& order) {
    if (n < 0 || budget < n) return TP_ERR_INVALID_ARG;
    if (n == 0) return TP_OK;
    if (policy == TP_BRANCH_EVEN) {
        for (int32_t i = 0; i < n; ++i) out[i] = budget / n + (i < budget % n ? 1 : 0);
        return TP_OK;
    }
    if ((policy != TP_BRANCH_LOGP_HIGH && policy != TP_BRANCH_LOGP_LOW) || !logp || !(temperature > 0.0))
        return TP_ERR_INVALID_ARG;
    const double sign = policy == TP_BRANCH_LOGP_HIGH ? 1.0 : -1.0;
    const int32_t extra = budget - n;  // every path keeps one branch
    frac.resize((size_t)n);
    double m = -INFINITY;
    for (int32_t i = 0; i < n; ++i) {
        if (!std::isfinite(logp[i])) return TP_ERR_INVALID_ARG;
        frac[(size_t)i] = sign * logp[i] / temperature;
        m = std::max(m, frac[(size_t)i]);
    }
    double z = 0.0;
    for (int32_t i = 0; i < n; ++i) {
        frac[(size_t)i] = std::exp(frac[(size_t)i] - m);
        z += frac[(size_t)i];
    }
    // largest-remainder rounding of the quotas extra * softmax_i
    int64_t used = 0;
    for (int32_t i = 0; i < n; ++i) {
        const double quota = (double)extra * (frac[(size_t)i] / z);
        const double whole = std::floor(quota);
        out[i] = 1 + (int32_t)whole;
        used += (int64_t)whole;
        frac[(size_t)i] = quota - whole;
    }
    const int64_t left = std::min<int64_t>(std::max<int64_t>(extra - used, 0), n);
    order.resize((size_t)n);
    for (int32_t i = 0; i < n; ++i) order[(size_t)i] = i;
    std::stable_sort(order.begin(), order.end(),
                     [&](int32_t a, int32_t b) { return frac[(size_t)a] > frac[(size_t)b]; });
    for (int64_t k = 0; k < left; ++k) ++out[order[(size_t)k]];
    return TP_OK;
}

}  // namespace tp

namespace {

using tp::fail;

enum : int64_t { EV_ROOT = 1, EV_FORK, EV_SEGMENT, EV_OUTPUT, EV_PRUNE, EV_FALLBACK, EV_DONE };

struct Path {
    int32_t q, node;
};

struct Segment {
    int32_t len, status;
    double logp;
};

struct OutputRec {
    int32_t node, depth;
    bool cand, alive;
};

struct QueryState {
    int32_t b0 = 1, fallbacks = 0, n_out = 0;
    std::vector<OutputRec> outs;
    bool done = false;
};

struct DevBuf {
    void* p = nullptr;
    int64_t cap = 0;
};

class Rollout {
   public:
    Rollout(tp_tree* t, const tp_rollout_params& p, int64_t* ev, int64_t cap, const tp_rollout_probe* probe)
        : t_(t), p_(p), ev_(ev), cap_(cap), probe_(probe) {}
    ~Rollout() {
        if (t_->cfg.pool) cudaStreamSynchronize(t_->stream);
        for (DevBuf* b : {&k_, &v_, &q_, &o_, &lse_, &rows_})
            if (b->p) cudaFree(b->p);
    }
    tp_status run(tp_rollout_stats* stats);

   private:
    tp_tree* t_;
    const tp_rollout_params& p_;
    int64_t* ev_;
    int64_t cap_;
    const tp_rollout_probe* probe_;
    tp_rollout_stats st_{};
    std::vector<int32_t> depth_;  // per node id: segments on the root-to-node path
    std::vector<QueryState> qs_;
    std::vector<Path> queue_;
    std::vector<Segment> seg_;
    DevBuf k_, v_, q_, o_, lse_, rows_;
    std::vector<int32_t> gen_, counts_;
    std::vector<double> frac_, logp_;
    std::vector<int32_t> order_, split_;

    double u(uint32_t tag, uint32_t a, uint32_t b, uint32_t c = 0) const {
        return tp::draw_uniform(p_.seed, tag, a, b, c);
    }
    void emit(int64_t kind, int32_t q, int32_t node, int64_t a = 0, int64_t b = 0, int64_t c = 0, int64_t d = 0) {
        if (ev_ && st_.events < cap_) {
            int64_t* e = ev_ + st_.events * 8;
            e[0] = kind, e[1] = q, e[2] = node, e[3] = a, e[4] = b, e[5] = c, e[6] = d, e[7] = 0;
        }
        ++st_.events;
    }
    void note_pool() {
        st_.peak_blocks = std::max<int64_t>(st_.peak_blocks, t_->pool.size() - t_->pool.free_count());
    }
    tp_status grow(DevBuf& b, int64_t bytes, const char* what) {
        return tp::ensure_device_bytes(t_, &b.p, &b.cap, bytes, what);
    }
    tp_status fork(int32_t q, int32_t node, int32_t k, std::vector<Path>& out) {
        const size_t at = out.size();
        std::vector<tp_node> kids((size_t)k);
        tp_status s = tp_fork(t_, node, k, kids.data());
        if (s != TP_OK) return s;
        depth_.resize(t_->nodes.size(), 0);
        for (tp_node c : kids) {
            depth_[(size_t)c] = depth_[(size_t)node] + 1;
            out.push_back({q, c});
        }
        emit(EV_FORK, q, node, out[at].node, k);
        return TP_OK;
    }
    tp_status prune(int32_t q, int32_t leaf) {
        emit(EV_PRUNE, q, leaf);
        return tp_prune(t_, leaf);
    }
    // Append n tokens of stand-in K/V (tokens 0..n-1 of `node`) in one call.
    tp_status append_synth(int32_t node, int32_t n) {
        if (!t_->cfg.pool) return tp_append_segment(t_, node, n, nullptr, nullptr);
        tp::SynthArgs a{};
        a.k = (uint16_t*)k_.p;
        a.v = (uint16_t*)v_.p;
        a.seed = p_.seed;
        a.rows = n;
        a.kv_width = t_->cfg.num_kv_heads * t_->cfg.head_dim;
        a.q_width = t_->cfg.num_q_heads * t_->cfg.head_dim;
        a.node0 = node;
        a.pos0 = t_->nodes[(size_t)node].n_tokens;
        cudaError_t e;
        {
            tp::LaunchTimer timer(t_, tp::KK_APPEND);
            e = tp::launch_synth(a, t_->stream);
        }
        if (e != cudaSuccess) return tp::cuda_fail(t_, e, "synth kernel");
        return tp_append_segment(t_, node, n, k_.p, v_.p);
    }
    Segment draw_segment(int32_t node) const;
    tp_status inference();
    tp_status decode_tokens();
};

Segment Rollout::draw_segment(int32_t node) const {
    Segment s{p_.seg_tokens, 0, 0.0};
    for (int32_t t = 0; t < p_.seg_tokens; ++t)
        if (u(tp::kTagEos, (uint32_t)node, (uint32_t)t) < p_.p_eos) {
            s.len = t + 1;
            s.status |= TP_SEG_EOS;
            break;
        }
    const double kappa = 2.0 * u(tp::kTagSegment, (uint32_t)node, tp::kSegScale);
    double acc = 0.0;
    for (int32_t t = 0; t < s.len; ++t) acc += kappa * std::log(1.0 - u(tp::kTagTokenLogp, (uint32_t)node, (uint32_t)t));
    s.logp = acc / s.len;
    if (u(tp::kTagSegment, (uint32_t)node, tp::kSegBoxed) < p_.p_boxed) s.status |= TP_SEG_BOXED;
    if (u(tp::kTagSegment, (uint32_t)node, tp::kSegFail) < p_.p_fail) s.status |= TP_SEG_FAILED;
    if (depth_[(size_t)node] >= p_.max_depth) s.status |= TP_SEG_MAX_DEPTH;
    return s;
}

// Token-synchronous generation: token t of every path whose segment is longer
// than t is appended, then those paths decode.
tp_status Rollout::decode_tokens() {
    const int32_t qw = t_->cfg.num_q_heads * t_->cfg.head_dim;
    int32_t max_len = 0;
    for (const Segment& s : seg_) max_len = std::max(max_len, s.len);
    for (int32_t t = 0; t < max_len; ++t) {
        gen_.clear();
        for (size_t i = 0; i < queue_.size(); ++i)
            if (seg_[i].len > t) gen_.push_back(queue_[i].node);
        const int32_t n = (int32_t)gen_.size();
        // the token's stand-in activations straight into the pool, Q into q_,
        // and the cached decode schedule patched: one upload, one launch
        tp_status s = tp::rollout_token_step(t_, gen_.data(), n, (int32_t*)rows_.p, rows_.cap / 4, p_.seed, t,
                                             (uint16_t*)q_.p, p_.decode_flags);
        if (s != TP_OK) return s;
        note_pool();
        s = tp_decode_ex(t_, gen_.data(), n, q_.p, o_.p, (float*)lse_.p, p_.decode_flags);
        if (s != TP_OK) return s;
        if (probe_ && probe_->call == st_.decode_calls) {
            const int32_t rows = std::min(n, probe_->cap);
            if (probe_->o) {
                cudaError_t e = cudaMemcpyAsync(probe_->o, o_.p, (size_t)rows * qw * 2, cudaMemcpyDeviceToDevice, t_->stream);
                if (e == cudaSuccess && probe_->lse)
                    e = cudaMemcpyAsync(probe_->lse, lse_.p, (size_t)rows * t_->cfg.num_q_heads * 4,
                                        cudaMemcpyDeviceToDevice, t_->stream);
                if (e != cudaSuccess) return tp::cuda_fail(t_, e, "probe copy");
            }
            for (int32_t i = 0; i < rows; ++i) {
                if (probe_->rows) probe_->rows[2 * i] = gen_[(size_t)i], probe_->rows[2 * i + 1] = t;
            }
            if (probe_->n_rows) *probe_->n_rows = rows;
        }
        ++st_.decode_calls;
        st_.decode_rows += n;
    }
    return TP_OK;
}

tp_status Rollout::inference() {
    seg_.clear();
    for (const Path& p : queue_) seg_.push_back(draw_segment(p.node));
    if (p_.decode) {
        tp_status s = decode_tokens();
        if (s != TP_OK) return s;
    } else {
        for (size_t i = 0; i < queue_.size(); ++i) {
            tp_status s = append_synth(queue_[i].node, seg_[i].len);
            if (s != TP_OK) return s;
            note_pool();
        }
    }
    for (size_t i = 0; i < queue_.size(); ++i) {
        const Segment& s = seg_[i];
        emit(EV_SEGMENT, queue_[i].q, queue_[i].node, depth_[(size_t)queue_[i].node], s.len, s.status,
             [&] { int64_t b; std::memcpy(&b, &s.logp, 8); return b; }());
        ++st_.segments;
        st_.tokens += s.len;
    }
    return TP_OK;
}

tp_status Rollout::run(tp_rollout_stats* stats) {
    const tp_rollout_params& p = p_;
    const int32_t nq = p.n_queries;
    const int32_t kvw = t_->cfg.num_kv_heads * t_->cfg.head_dim, qw = t_->cfg.num_q_heads * t_->cfg.head_dim;
    int64_t max_prompt = 0;
    for (int32_t q = 0; q < nq; ++q) max_prompt = std::max<int64_t>(max_prompt, p.prompt_tokens[q]);
    if (t_->cfg.pool) {
        const int64_t rows_max = (int64_t)nq * p.width;  // paths in flight never exceed w per query
        const int64_t stage_rows = std::max<int64_t>({rows_max, max_prompt, (int64_t)p.seg_tokens});
        tp_status s = grow(k_, stage_rows * kvw * 2, "rollout K staging");
        if (s == TP_OK) s = grow(v_, stage_rows * kvw * 2, "rollout V staging");
        if (s == TP_OK && p.decode) s = grow(q_, rows_max * qw * 2, "rollout Q");
        if (s == TP_OK && p.decode) s = grow(o_, rows_max * qw * 2, "rollout O");
        if (s == TP_OK && p.decode) s = grow(lse_, rows_max * t_->cfg.num_q_heads * 4, "rollout LSE");
        if (s == TP_OK && p.decode) s = grow(rows_, rows_max * 16, "rollout token-step words");
        if (s != TP_OK) return s;
    }
    qs_.assign((size_t)nq, QueryState());
    const int64_t nodes_before = (int64_t)t_->nodes.size();

    // prompts: one root per query, then the initial fork (depth 0 budget b0)
    std::vector<Path> roots;
    for (int32_t q = 0; q < nq; ++q) {
        tp_node r;
        tp_status s = tp_add_root(t_, &r);
        if (s != TP_OK) return s;
        depth_.resize(t_->nodes.size(), 0);
        QueryState& Q = qs_[(size_t)q];
        Q.b0 = p.init_branches > 0 ? p.init_branches : 2 + (int32_t)(7.0 * u(tp::kTagQuery, (uint32_t)q, tp::kQueryInit));
        emit(EV_ROOT, q, r, p.prompt_tokens[q], Q.b0);
        s = append_synth(r, p.prompt_tokens[q]);
        if (s != TP_OK) return s;
        st_.prompt_tokens += p.prompt_tokens[q];
        note_pool();
        roots.push_back({q, r});
    }
    std::vector<Path> next;
    for (const Path& r : roots) {
        tp_status s = fork(r.q, r.node, std::min(qs_[(size_t)r.q].b0, p.width), next);
        if (s != TP_OK) return s;
    }
    queue_.swap(next);

    std::vector<Path> cont;
    while (!queue_.empty()) {
        ++st_.iterations;
        tp_status s = inference();
        if (s != TP_OK) return s;
        // finished and failed segments leave the queue as outputs
        cont.clear();
        logp_.clear();
        for (size_t i = 0; i < queue_.size(); ++i) {
            const Path& pa = queue_[i];
            const Segment& sg = seg_[i];
            QueryState& Q = qs_[(size_t)pa.q];
            const int32_t d = depth_[(size_t)pa.node];
            if (sg.status & TP_SEG_FAILED) {
                emit(EV_OUTPUT, pa.q, pa.node, d, 0, 0);
                Q.outs.push_back({pa.node, d, false, false});
                ++Q.n_out;
                s = prune(pa.q, pa.node);
            } else if (sg.status & (TP_SEG_EOS | TP_SEG_BOXED | TP_SEG_MAX_DEPTH)) {
                const bool cand = (sg.status & (TP_SEG_EOS | TP_SEG_BOXED)) != 0;
                const int64_t reward =
                    (sg.status & TP_SEG_BOXED) && u(tp::kTagSegment, (uint32_t)pa.node, tp::kSegCorrect) < p.p_correct;
                emit(EV_OUTPUT, pa.q, pa.node, d, cand, reward);
                const bool keep = cand && p.fallback;
                Q.outs.push_back({pa.node, d, cand, keep});
                ++Q.n_out;
                if (!keep) s = prune(pa.q, pa.node);
            } else {
                cont.push_back(pa);
                logp_.push_back(sg.logp);
            }
            if (s != TP_OK) return s;
        }
        st_.outputs = 0;
        for (const QueryState& Q : qs_) st_.outputs += Q.n_out;

        // Branching: per query (ascending), its continuing paths in queue order
        next.clear();
        counts_.assign((size_t)nq, 0);
        for (const Path& pa : cont) ++counts_[(size_t)pa.q];
        for (int32_t q = 0; q < nq; ++q) {
            const int32_t a = counts_[(size_t)q];
            if (a == 0) continue;
            QueryState& Q = qs_[(size_t)q];
            std::vector<double> lp;
            std::vector<int32_t> nodes;
            for (size_t i = 0; i < cont.size(); ++i)
                if (cont[i].q == q) {
                    nodes.push_back(cont[i].node);
                    lp.push_back(logp_[i]);
                }
            const int32_t j = depth_[(size_t)nodes[0]];
            int64_t budget = Q.b0;
            for (int32_t k = 0; k < j && budget < p.width; ++k) budget *= p.arity;
            budget = std::min<int64_t>(budget, p.width - Q.n_out);
            budget = std::max<int64_t>(budget, a);
            split_.resize((size_t)a);
            s = tp::branch_split(lp.data(), a, (int32_t)budget, p.policy, p.temperature, split_.data(), frac_, order_);
            if (s != TP_OK) return fail(t_, s, "branch assignment failed");
            for (int32_t i = 0; i < a; ++i) {
                s = fork(q, nodes[(size_t)i], split_[(size_t)i], next);
                if (s != TP_OK) return s;
            }
        }
        // Fallback: a query with no path and fewer than w outputs re-spawns
        // one path from a random boundary of a random finished candidate
        counts_.assign((size_t)nq, 0);
        for (const Path& pa : next) ++counts_[(size_t)pa.q];
        for (int32_t q = 0; q < nq && p.fallback; ++q) {
            QueryState& Q = qs_[(size_t)q];
            if (Q.done || counts_[(size_t)q] > 0 || Q.n_out >= p.width) continue;
            std::vector<int32_t> cands;
            for (size_t i = 0; i < Q.outs.size(); ++i)
                if (Q.outs[i].alive) cands.push_back((int32_t)i);
            if (cands.empty()) continue;
            const int32_t pick =
                cands[(size_t)(cands.size() * u(tp::kTagQuery, (uint32_t)q, tp::kQueryPick, (uint32_t)Q.fallbacks))];
            const OutputRec& c = Q.outs[(size_t)pick];
            const int32_t jb = (int32_t)(c.depth * u(tp::kTagQuery, (uint32_t)q, tp::kQueryDepth, (uint32_t)Q.fallbacks));
            int32_t at = c.node;
            while (depth_[(size_t)at] > jb) at = t_->nodes[(size_t)at].parent;
            ++Q.fallbacks;
            ++st_.fallbacks;
            emit(EV_FALLBACK, q, c.node, at, jb);
            s = fork(q, at, 1, next);
            if (s != TP_OK) return s;
            ++counts_[(size_t)q];
        }
        // queries with nothing left to sample release their kept candidates
        for (int32_t q = 0; q < nq; ++q) {
            QueryState& Q = qs_[(size_t)q];
            if (Q.done || counts_[(size_t)q] > 0) continue;
            for (OutputRec& o : Q.outs)
                if (o.alive) {
                    o.alive = false;
                    s = prune(q, o.node);
                    if (s != TP_OK) return s;
                }
            Q.done = true;
            emit(EV_DONE, q, -1, Q.n_out);
        }
        queue_.swap(next);
    }
    st_.nodes = (int64_t)t_->nodes.size() - nodes_before;
    if (stats) *stats = st_;
    return TP_OK;
}

}  // namespace

extern "C" {

tp_status tp_branch_assign(const double* logp, int32_t n, int32_t budget, int32_t policy, double temperature,
                           int32_t* out) {
    if (n > 0 && !out) return TP_ERR_INVALID_ARG;
    std::vector<double> frac;
    std::vector<int32_t> order;
    return tp::branch_split(logp, n, budget, policy, temperature, out, frac, order);
}

tp_status tp_rollout(tp_tree* t, const tp_rollout_params* p, int64_t* events, int64_t cap_events,
                     const tp_rollout_probe* probe, tp_rollout_stats* stats) {
    if (!t) return TP_ERR_INVALID_ARG;
    if (!p) return fail(t, TP_ERR_INVALID_ARG, "params is NULL");
    if (p->n_queries < 0 || (p->n_queries > 0 && !p->prompt_tokens))
        return fail(t, TP_ERR_INVALID_ARG, "n_queries < 0 or prompt_tokens is NULL");
    for (int32_t q = 0; q < p->n_queries; ++q)
        if (p->prompt_tokens[q] < 1 || p->prompt_tokens[q] > (1 << 20))
            return fail(t, TP_ERR_INVALID_ARG, "prompt lengths must lie in [1, 2^20]");
    if (p->width < 1 || p->max_depth < 1 || p->arity < 1 || p->init_branches < 0)
        return fail(t, TP_ERR_INVALID_ARG, "width, max_depth and arity must be >= 1, init_branches >= 0");
    if (p->seg_tokens < 1 || p->seg_tokens > (1 << 20)) return fail(t, TP_ERR_INVALID_ARG, "seg_tokens must lie in [1, 2^20]");
    if (p->policy != TP_BRANCH_EVEN && p->policy != TP_BRANCH_LOGP_HIGH && p->policy != TP_BRANCH_LOGP_LOW)
        return fail(t, TP_ERR_INVALID_ARG, "unknown branching policy");
    if (p->policy != TP_BRANCH_EVEN && !(p->temperature > 0.0))
        return fail(t, TP_ERR_INVALID_ARG, "temperature must be > 0");
    if (p->decode && !t->cfg.pool) return fail(t, TP_ERR_INVALID_ARG, "decode needs a device pool");
    if (events && cap_events < 0) return fail(t, TP_ERR_INVALID_ARG, "cap_events < 0");
    if (probe && probe->cap < 0) return fail(t, TP_ERR_INVALID_ARG, "probe cap < 0");
    if ((int64_t)t->nodes.size() + (int64_t)p->n_queries * p->width * (p->max_depth + 2) >= (1 << 28))
        return fail(t, TP_ERR_INVALID_ARG, "node ids would exceed the generator's 2^28 key range");
    Rollout r(t, *p, events, events ? cap_events : 0, probe);
    return r.run(stats);
}

}  // extern "C"
