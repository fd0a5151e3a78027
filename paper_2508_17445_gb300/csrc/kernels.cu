// kernels.cu -- sm_103a kernels of libtreepo.
//
//   append_kernel   copy a segment's K/V into pool blocks (16-byte chunks,
//                   XOR-swizzled inside each token row, see below)
//   decode_kernel   split-KV flash-decode: one CTA per unit = (chunk of path
//                   blocks, kv head, <= 64 stacked query rows). K/V blocks
//                   stream through a shared-memory ring filled by TMA bulk
//                   copies (cp.async.bulk + mbarrier transaction counts).
//                   Units with < 16 rows (one leaf's GQA group, or two) run
//                   on CUDA cores with warp-shuffle reductions; units whose
//                   stacked rows form a real contraction run Q.K^T and P.V on
//                   tensor cores (mma.sync m16n8k16 bf16 -> fp32).
//   merge_kernel    per (leaf occurrence, q-head): log-sum-exp merge of the
//                   partials of every unit on the path -> O (bf16), LSE (fp32)
//   gather_kernel   inspection: copy a path's K/V out through the block tables
//
// Attention per row (q-head h of one leaf): s_j = q.k_j / sqrt(d),
// LSE = ln sum_j exp(s_j), O = sum_j exp(s_j - LSE) v_j -- standard decode
// attention over the root-to-leaf path, the trajectory s_1 (+) ... (+) s_j of
// TreePO (Sec. 2.3). Scores are kept in the log2 domain (q.k * log2(e)/sqrt(d))
// so exponentials are exp2; partial LSEs are log2, the final LSE is natural.
//
// Pool layout. Block b holds [K|V][kv head] tiles of 32 tokens x d bf16; a
// tile is d/64 halves, each 32 rows of 128 bytes (64 elements) whose 16-byte
// chunk c sits at position c ^ (row & 7) (see kv_off). A bulk copy of a tile
// half lands in shared memory as 128-byte-swizzle atoms, the canonical layout
// of tcgen05 operands, and ldmatrix row gathers (8 rows, same chunk) and
// CUDA-core row reads both hit 8 distinct bank groups.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <algorithm>
#include <mutex>

#include "forest.h"
#include "splitmix.h"

namespace tp {
namespace {

constexpr int kConsumerWarps = 4;                          // attention warps per CTA
constexpr int kStreamerWarp = kConsumerWarps;              // issues the K/V bulk copies
constexpr int kFetcherWarp = kConsumerWarps + 1;           // claims units, stages their data
constexpr int kDecodeThreads = (kConsumerWarps + 2) * 32;
constexpr int kBlockTokens = 32;   // tokens per pool block (= tile)
constexpr int kStageTokens = 64;   // two tiles per pipeline stage
constexpr int kStages = 2;         // stages in each CTA's shared-memory ring
constexpr uint64_t kWaitLimitNs = 2000000000ull;  // bounded mbarrier waits: 2 s

// ------------------------------------------------------------ PTX helpers --
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{ .reg .pred p; mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2; selp.u32 %0, 1, 0, p; }"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

__device__ __forceinline__ float fast_exp2(float x) {  // ex2.approx: exp2(-inf) = +0
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// Non-blocking probe of an mbarrier phase.
__device__ __forceinline__ bool mbar_test(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{ .reg .pred p; mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2; selp.u32 %0, 1, 0, p; }"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

__device__ __forceinline__ uint64_t global_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// Wait for an mbarrier phase with a time limit; false if the limit ran out.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, uint64_t limit_ns = kWaitLimitNs) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = global_ns();
    for (uint32_t i = 1;; ++i) {
        if (mbar_try_wait(bar, parity)) return true;
        if ((i & 63) == 0 && global_ns() - t0 > limit_ns) return false;
    }
}

__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
    asm volatile(
        "cp.async.bulk.shared::cta.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
        "l"(src), "r"(bytes), "r"(bar)
        : "memory");
}

// L2 residency: a decode call streams GBs of K/V through the 129 MB L2 once,
// while its fp32 partials (tens of MB) are written by the attention kernels
// and read back by the merge. K/V copies read once go in as evict-first, the
// partials as evict-last, and the merge reads them as evict-first (dead
// after), so they are served from L2 instead of a round trip through HBM.
__device__ __forceinline__ uint64_t l2_evict_first() {
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
    return p;
}

__device__ __forceinline__ uint64_t l2_evict_last() {
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
    return p;
}

__device__ __forceinline__ void bulk_g2s_hint(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar,
                                              uint64_t pol) {
    asm volatile(
        "cp.async.bulk.shared::cta.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;" ::"r"(
            dst),
        "l"(src), "r"(bytes), "r"(bar), "l"(pol)
        : "memory");
}

__device__ __forceinline__ void st_f2_hint(float* p, float x, float y, uint64_t pol) {
    asm volatile("st.global.L2::cache_hint.v2.f32 [%0], {%1, %2}, %3;" ::"l"(p), "f"(x), "f"(y), "l"(pol) : "memory");
}

__device__ __forceinline__ void st_f4_hint(float* p, float4 v, uint64_t pol) {
    asm volatile("st.global.L2::cache_hint.v4.f32 [%0], {%1, %2, %3, %4}, %5;" ::"l"(p), "f"(v.x), "f"(v.y), "f"(v.z),
                 "f"(v.w), "l"(pol)
                 : "memory");
}

__device__ __forceinline__ float4 ld_f4_hint(const float* p, uint64_t pol) {
    float4 v;
    asm volatile("ld.global.L2::cache_hint.v4.f32 {%0, %1, %2, %3}, [%4], %5;"
                 : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
                 : "l"(p), "l"(pol));
    return v;
}

// Drop a 128-byte L2 line without writing it back (its contents become
// undefined): for partial rows the merge has consumed.
__device__ __forceinline__ void l2_discard(const void* p) {
    if ((reinterpret_cast<uintptr_t>(p) & 127) == 0)  // whole lines only (the partial rows are 256-byte aligned)
        asm volatile("discard.global.L2 [%0], 128;" ::"l"(p) : "memory");
}

__device__ __forceinline__ float2 ld_f2_hint(const float* p, uint64_t pol) {
    float2 v;
    asm volatile("ld.global.L2::cache_hint.v2.f32 {%0, %1}, [%2], %3;" : "=f"(v.x), "=f"(v.y) : "l"(p), "l"(pol));
    return v;
}

// 16-byte global -> shared copy that bypasses registers (cp.async)
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_all;" ::: "memory"); }

__device__ __forceinline__ void fence_proxy_async() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}

__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}

__device__ __forceinline__ void mma_bf16(float (&c)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
    __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&v);
}

// 32-byte global store (sm_100 and later); dst must be 32-byte aligned
__device__ __forceinline__ void st_global_v8(void* dst, const uint32_t* w) {
    asm volatile("st.global.v8.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};" ::"l"(dst), "r"(w[0]), "r"(w[1]),
                 "r"(w[2]), "r"(w[3]), "r"(w[4]), "r"(w[5]), "r"(w[6]), "r"(w[7])
                 : "memory");
}

// the same with an L2 cache policy
__device__ __forceinline__ void st_global_v8_hint(void* dst, const uint32_t* w, uint64_t pol) {
    asm volatile("st.global.L2::cache_hint.v8.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8}, %9;" ::"l"(dst), "r"(w[0]),
                 "r"(w[1]), "r"(w[2]), "r"(w[3]), "r"(w[4]), "r"(w[5]), "r"(w[6]), "r"(w[7]), "l"(pol)
                 : "memory");
}

// max of three (one instruction on sm_100 and later)
__device__ __forceinline__ float fmax3(float a, float b, float c) {
    float r;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
    return r;
}

// Packed fp32 pairs (sm_100 and later): one instruction, two lanes, each
// rounded exactly like its scalar counterpart.
__device__ __forceinline__ uint64_t f2_pack(float lo, float hi) {
    uint64_t r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
    return r;
}
__device__ __forceinline__ void f2_unpack(uint64_t v, float& lo, float& hi) {
    asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ uint64_t f2_fma(uint64_t a, uint64_t b, uint64_t c) {
    uint64_t r;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(a), "l"(b), "l"(c));
    return r;
}
__device__ __forceinline__ uint64_t f2_add(uint64_t a, uint64_t b) {
    uint64_t r;
    asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
    return r;
}

// bf16 pair in a 32-bit word -> two fp32 (exact: bf16 is the top half of fp32)
__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

// Byte offset of 16-byte chunk `chunk` of token row `row` in a K or V tile of
// `rows` token rows: the tile is split into 64-element halves of head_dim,
// each half a run of 128-byte rows with chunk position (chunk & 7) ^ (row & 7)
// -- the 128-byte-swizzle atoms (8 rows x 128 B) that tcgen05 operand
// descriptors address, and bank-conflict free for ldmatrix row gathers and
// for one-row reads.
template <int ROWS>
__device__ __forceinline__ int kv_off(int row, int chunk) {
    return (chunk >> 3) * (ROWS * 128) + row * 128 + (((chunk & 7) ^ (row & 7)) << 4);
}

// Bounds-checked build: true when an index check passed; otherwise records
// the failure in the device error word (the caller skips the access). In the
// default build it is `true` and the check compiles away.
__device__ __forceinline__ bool check(bool ok, int32_t* err) {
    if (kBoundsCheck && !ok) {
        atomicOr(err, kErrBounds);
        return false;
    }
    return true;
}

// ------------------------------------------------------------------ append --
template <int HD>
__global__ void append_kernel(const AppendArgs a) {
    constexpr int CH = HD / 8;  // 16-byte chunks per token row
    const int64_t per_kv = (int64_t)a.n_tokens * a.hkv * CH;
    const int64_t total = 2 * per_kv;
    for (int64_t idx = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; idx < total;
         idx += (int64_t)gridDim.x * blockDim.x) {
        const int kv = idx >= per_kv;
        const int64_t r = kv ? idx - per_kv : idx;
        const int c = (int)(r % CH);
        const int h = (int)((r / CH) % a.hkv);
        const int i = (int)(r / ((int64_t)CH * a.hkv));
        const uint4 val = reinterpret_cast<const uint4*>(kv ? a.v : a.k)[r];
        const int pos = a.first_row + i;
        const int blk = a.blocks[pos / kBlockTokens];
        const int row = pos % kBlockTokens;
        if (!check(in_range(blk, a.pool_blocks), a.err)) continue;
        uint8_t* dst = a.pool + (int64_t)blk * a.block_bytes + (int64_t)(kv * a.hkv + h) * a.head_bytes +
                       kv_off<kBlockTokens>(row, c);
        *reinterpret_cast<uint4*>(dst) = val;
    }
}

// ----------------------------------------------------------- token append --
// Decode-loop append: one token for each of n nodes, each to its own slot.
template <int HD>
__global__ void append_tokens_kernel(const AppendTokensArgs a) {
    constexpr int CH = HD / 8;
    const int64_t per_kv = (int64_t)a.n * a.hkv * CH;
    for (int64_t idx = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; idx < 2 * per_kv;
         idx += (int64_t)gridDim.x * blockDim.x) {
        const int kv = idx >= per_kv;
        const int64_t r = kv ? idx - per_kv : idx;
        const int c = (int)(r % CH);
        const int h = (int)((r / CH) % a.hkv);
        const int i = (int)(r / ((int64_t)CH * a.hkv));
        const int32_t slot = a.slots[i];
        if (!check(in_range(slot, a.pool_blocks * kBlockTokens), a.err)) continue;
        const uint4 val = reinterpret_cast<const uint4*>(kv ? a.v : a.k)[r];
        uint8_t* dst = a.pool + (int64_t)(slot / kBlockTokens) * a.block_bytes +
                       (int64_t)(kv * a.hkv + h) * a.head_bytes + kv_off<kBlockTokens>(slot % kBlockTokens, c);
        *reinterpret_cast<uint4*>(dst) = val;
    }
}

// ------------------------------------------------------ stand-in activations --
// A 64-bit draw -> 4 consecutive bf16 values (low 16 bits first), as two
// 32-bit words of bf16 pairs.
__device__ __forceinline__ uint2 synth_words(uint64_t h) {
    const uint32_t lo = synth_bf16_bits((uint32_t)h & 0xffffu) | (uint32_t)synth_bf16_bits((uint32_t)(h >> 16) & 0xffffu) << 16;
    const uint32_t hi = synth_bf16_bits((uint32_t)(h >> 32) & 0xffffu) | (uint32_t)synth_bf16_bits((uint32_t)(h >> 48)) << 16;
    return make_uint2(lo, hi);
}

// One thread per 64-bit draw = 4 consecutive bf16 values of one row.
__global__ void synth_kernel(const SynthArgs a) {
    const int kv_words = a.kv_width / 4, q_words = a.q_width / 4;
    const int words = (a.k ? kv_words : 0) + (a.v ? kv_words : 0) + (a.q ? q_words : 0);
    const int64_t total = a.rows * words;
    for (int64_t idx = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; idx < total;
         idx += (int64_t)gridDim.x * blockDim.x) {
        const int64_t i = idx / words;
        int w = (int)(idx % words);
        uint16_t* out;
        uint32_t tag;
        int width;
        if (a.k && w < kv_words) {
            out = a.k, tag = kTagK, width = a.kv_width;
        } else {
            if (a.k) w -= kv_words;
            if (a.v && w < kv_words) {
                out = a.v, tag = kTagV, width = a.kv_width;
            } else {
                if (a.v) w -= kv_words;
                out = a.q, tag = kTagQ, width = a.q_width;
            }
        }
        const uint32_t node = (uint32_t)(a.row_node ? a.row_node[i] : a.node0);
        const uint32_t pos = (uint32_t)(a.row_node ? a.pos0 : a.pos0 + i);
        const uint64_t h = splitmix64(a.seed, draw_counter(tag, node, pos, (uint32_t)w));
        *reinterpret_cast<uint2*>(out + i * width + 4 * w) = synth_words(h);
    }
}

// One token step of the rollout's decode loop: row i's new token (node
// row_node[i], position pos) gets the stand-in activations synth_kernel
// would draw for it, K and V written straight into its pool slot (the bytes
// append_tokens_kernel would write), Q into q; then the schedule words the
// append changed are patched. One thread per 16-byte K/V chunk (two draws),
// per Q draw, per patch.
template <int HD>
__global__ void rollout_step_kernel(const StepArgs a) {
    constexpr int CH = HD / 8;
    const int64_t kv_items = (int64_t)a.n * 2 * a.hkv * CH;
    const int q_words = a.q_width / 4;
    const int64_t q_items = (int64_t)a.n * q_words;
    const int64_t total = kv_items + q_items + a.n_pairs;
    for (int64_t idx = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; idx < total;
         idx += (int64_t)gridDim.x * blockDim.x) {
        if (idx < kv_items) {
            const int c = (int)(idx % CH);
            const int h = (int)((idx / CH) % a.hkv);
            const int kv = (int)((idx / ((int64_t)CH * a.hkv)) & 1);
            const int i = (int)(idx / ((int64_t)CH * a.hkv * 2));
            const uint32_t node = (uint32_t)a.row_node[i], tag = kv ? kTagV : kTagK;
            const uint32_t w0 = (uint32_t)(h * (HD / 4) + 2 * c);  // the chunk's two draws of the row
            const uint2 x0 = synth_words(splitmix64(a.seed, draw_counter(tag, node, (uint32_t)a.pos, w0)));
            const uint2 x1 = synth_words(splitmix64(a.seed, draw_counter(tag, node, (uint32_t)a.pos, w0 + 1)));
            const int32_t slot = a.slots[i];
            if (!check(in_range(slot, a.pool_blocks * kBlockTokens), a.err)) continue;
            uint8_t* dst = a.pool + (int64_t)(slot / kBlockTokens) * a.block_bytes +
                           (int64_t)(kv * a.hkv + h) * a.head_bytes + kv_off<kBlockTokens>(slot % kBlockTokens, c);
            *reinterpret_cast<uint4*>(dst) = make_uint4(x0.x, x0.y, x1.x, x1.y);
        } else if (idx < kv_items + q_items) {
            const int64_t r = idx - kv_items;
            const int i = (int)(r / q_words), w = (int)(r % q_words);
            const uint32_t node = (uint32_t)a.row_node[i];
            *reinterpret_cast<uint2*>(a.q + (int64_t)i * a.q_width + 4 * w) =
                synth_words(splitmix64(a.seed, draw_counter(kTagQ, node, (uint32_t)a.pos, (uint32_t)w)));
        } else {
            const int64_t k = idx - kv_items - q_items;
            if (!check(in_range(a.pairs[2 * k], a.sched_words), a.err)) continue;
            a.sched[a.pairs[2 * k]] = a.pairs[2 * k + 1];
        }
    }
}

// -------------------------------------------------------- tree advantage --
// Eq. tree_ae over a node table, in fp64 and in four launches spread over
// the SMs (GB300 runs fp64 at a small fraction of its fp32 rate per SM, so
// one CTA doing every output's divisions was fp64-bound):
//   init   every node's (count, sum) and reward range cleared;
//   walk   every output adds its reward to each strict ancestor's (count,
//          sum) and folds it into its root's reward range;
//   means  every node's sum_x / count_x, once (fp64 divisions are slow,
//          and the ancestors of many outputs coincide);
//   abar   A_i = mean over those ancestors x of (R_i - sum_x / count_x), for
//          outputs whose query's rewards are not all equal, with the sums of
//          A_i and of accepted outputs; the last CTA to finish takes the mean
//          and (population) std over the accepted outputs and writes
//          adv_i = A_i / std (0 for rejected outputs, or when std is 0).
// Workspace: cnt[n] | kmin[n] | kmax[n] | sum[n] (fp64) | abar[n_out] |
// root[n_out] | depth[n_out] | totals (fp64 s, c) | bad flag | CTA ticket.
constexpr int kAdvThreads = 256;      // init and the final pass
constexpr int kAdvWalkThreads = 32;   // one warp per CTA: outputs spread over many SMs
constexpr int kAdvAbarThreads = 128;  // the last CTA also runs the final pass over every output

struct AdvWs {
    int32_t* cnt;
    uint32_t* kmin;
    uint32_t* kmax;
    double* sum;
    double* abar;
    int32_t* root_of;
    int32_t* depth_of;
    double* tot;      // [2]: sum of A_i, accepted outputs
    int32_t* flags;   // [2]: malformed table, CTAs of the abar launch done
};

__host__ __device__ __forceinline__ int64_t adv_tail_offset(int64_t n_nodes, int64_t n_out) {
    return ((12 * n_nodes + 7) / 8) * 8 + 8 * n_nodes + 8 * n_out + 8 * n_out;
}

__device__ __forceinline__ AdvWs adv_ws(const AdvantageArgs& a) {
    AdvWs w;
    w.cnt = reinterpret_cast<int32_t*>(a.ws);
    w.kmin = reinterpret_cast<uint32_t*>(w.cnt + a.n_nodes);
    w.kmax = w.kmin + a.n_nodes;
    w.sum = reinterpret_cast<double*>(a.ws + ((12ll * a.n_nodes + 7) / 8) * 8);
    w.abar = w.sum + a.n_nodes;
    w.root_of = reinterpret_cast<int32_t*>(w.abar + a.n_out);
    w.depth_of = w.root_of + a.n_out;
    w.tot = reinterpret_cast<double*>(a.ws + adv_tail_offset(a.n_nodes, a.n_out));
    w.flags = reinterpret_cast<int32_t*>(w.tot + 2);
    return w;
}

__device__ __forceinline__ uint32_t reward_key(float r) {  // order-preserving float -> uint
    const uint32_t u = __float_as_uint(r);
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

template <int THREADS>
__device__ double block_sum(double v, double* red) {
    for (int off = 16; off; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
    if (THREADS == 32) return v;
    __syncthreads();
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
    __syncthreads();
    double s = 0.0;
    for (int k = 0; k < THREADS / 32; ++k) s += red[k];  // same order in every thread
    __syncthreads();
    return s;
}

__global__ void __launch_bounds__(kAdvThreads) advantage_init_kernel(const AdvantageArgs a) {
    const AdvWs w = adv_ws(a);
    for (int64_t x = (int64_t)blockIdx.x * kAdvThreads + threadIdx.x; x < a.n_nodes;
         x += (int64_t)gridDim.x * kAdvThreads) {
        w.cnt[x] = 0;
        w.sum[x] = 0.0;
        w.kmin[x] = 0xffffffffu;
        w.kmax[x] = 0u;
    }
    if (blockIdx.x == 0 && threadIdx.x == 0) {
        w.tot[0] = w.tot[1] = 0.0;
        w.flags[0] = w.flags[1] = 0;
    }
}

__global__ void __launch_bounds__(kAdvWalkThreads) advantage_walk_kernel(const AdvantageArgs a) {
    const AdvWs w = adv_ws(a);
    const int i = blockIdx.x * kAdvWalkThreads + threadIdx.x;
    if (i >= a.n_out) return;
    const int32_t lf = a.leaf[i];
    w.root_of[i] = -1;
    w.depth_of[i] = 0;
    if (lf < 0 || lf >= a.n_nodes) {
        w.flags[0] = 1;
        return;
    }
    const float r = a.reward[i];
    int32_t root = lf, depth = 0;
    for (int32_t x = a.parent[lf]; x != -1; x = a.parent[x]) {
        if (x < -1 || x >= a.n_nodes || depth >= a.n_nodes) {  // malformed table: stop
            w.flags[0] = 1;
            return;
        }
        atomicAdd(&w.cnt[x], 1);
        atomicAdd(&w.sum[x], (double)r);
        root = x;
        ++depth;
    }
    atomicMin(&w.kmin[root], reward_key(r));
    atomicMax(&w.kmax[root], reward_key(r));
    w.root_of[i] = root;
    w.depth_of[i] = depth;
}

__global__ void __launch_bounds__(kAdvThreads) advantage_means_kernel(const AdvantageArgs a) {
    const AdvWs w = adv_ws(a);
    for (int64_t x = (int64_t)blockIdx.x * kAdvThreads + threadIdx.x; x < a.n_nodes;
         x += (int64_t)gridDim.x * kAdvThreads)
        if (w.cnt[x] > 0) w.sum[x] /= (double)w.cnt[x];  // the sub-group mean of G_x
}

__global__ void __launch_bounds__(kAdvAbarThreads) advantage_abar_kernel(const AdvantageArgs a) {
    __shared__ double red[kAdvAbarThreads / 32];
    __shared__ bool last;
    const AdvWs w = adv_ws(a);
    const int i = blockIdx.x * kAdvAbarThreads + threadIdx.x;
    double s = 0.0, c = 0.0;
    if (i < a.n_out) {
        const int32_t root = w.root_of[i], depth = w.depth_of[i];
        if (root < 0 || depth == 0 || w.kmin[root] == w.kmax[root]) {
            w.abar[i] = 0.0;
            w.depth_of[i] = 0;  // rejected
        } else {
            const double r = (double)a.reward[i];
            double acc = 0.0;
            for (int32_t x = a.parent[a.leaf[i]]; x != -1; x = a.parent[x]) acc += r - w.sum[x];  // sum = mean here
            s = acc / (double)depth;
            c = 1.0;
            w.abar[i] = s;
        }
    }
    __threadfence();  // every thread's A_i (and rejections) before the CTA's ticket
    s = block_sum<kAdvAbarThreads>(s, red);
    c = block_sum<kAdvAbarThreads>(c, red);
    if (threadIdx.x == 0) {
        atomicAdd(&w.tot[0], s);
        atomicAdd(&w.tot[1], c);
        __threadfence();  // the totals before the ticket
        last = atomicAdd(&w.flags[1], 1) == (int)gridDim.x - 1;
    }
    __syncthreads();
    if (!last) return;
    // the last CTA: mean, std and the normalised advantages of every output
    // (the other CTAs' writes read through L2, past this SM's L1)
    __threadfence();
    const double n_acc = __ldcg(&w.tot[1]);
    const double mean = n_acc > 0.0 ? __ldcg(&w.tot[0]) / n_acc : 0.0;
    double v = 0.0;
    for (int k = threadIdx.x; k < a.n_out; k += kAdvAbarThreads)
        if (__ldcg(&w.depth_of[k]) > 0) {
            const double d = __ldcg(&w.abar[k]) - mean;
            v += d * d;
        }
    const double var = n_acc > 0.0 ? block_sum<kAdvAbarThreads>(v, red) / n_acc : 0.0;
    const double sd = sqrt(var), inv_sd = sd > 0.0 ? 1.0 / sd : 0.0;
    for (int k = threadIdx.x; k < a.n_out; k += kAdvAbarThreads)
        a.adv[k] = (__ldcg(&w.depth_of[k]) > 0 && sd > 0.0) ? (float)(__ldcg(&w.abar[k]) * inv_sd) : 0.f;
    if (threadIdx.x == 0 && a.stats) {
        a.stats[0] = n_acc;
        a.stats[1] = mean;
        a.stats[2] = sd;
        a.stats[3] = __ldcg(&w.flags[0]) ? 1.0 : 0.0;
    }
}

// ------------------------------------------------------- schedule patch --
__global__ void patch_kernel(int32_t* sched, const int32_t* pairs, int32_t n, int64_t sched_words, int32_t* err) {
    const int k = blockIdx.x * blockDim.x + threadIdx.x;
    if (k < n && check(in_range(pairs[2 * k], sched_words), err)) sched[pairs[2 * k]] = pairs[2 * k + 1];
}

// ------------------------------------------------------------------ gather --
template <int HD>
__global__ void gather_kernel(const GatherArgs a, int64_t n_tokens) {
    constexpr int CH = HD / 8;
    const int64_t per_kv = n_tokens * a.hkv * CH;
    for (int64_t idx = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; idx < 2 * per_kv;
         idx += (int64_t)gridDim.x * blockDim.x) {
        const int kv = idx >= per_kv;
        const int64_t r = kv ? idx - per_kv : idx;
        const int c = (int)(r % CH);
        const int h = (int)((r / CH) % a.hkv);
        const int64_t tok = r / ((int64_t)CH * a.hkv);
        // walk the tile list: tiles are full blocks except possibly the last
        // block of each node, so locate the token by a linear scan
        int64_t base = 0;
        int32_t w = 0;
        for (int k = 0; k < a.n_tiles; ++k) {
            w = a.tiles[k];
            const int valid = (w & ((1 << kTileValidBits) - 1)) + 1;
            if (tok < base + valid) break;
            base += valid;
        }
        const int row = (int)(tok - base);
        const int64_t blk = w >> kTileValidBits;
        if (!check(tile_word_ok(w, a.pool_blocks), a.err)) continue;
        const uint8_t* src = a.pool + blk * a.block_bytes + (int64_t)(kv * a.hkv + h) * a.head_bytes +
                             kv_off<kBlockTokens>(row, c);
        reinterpret_cast<uint4*>(kv ? a.v_out : a.k_out)[r] = *reinterpret_cast<const uint4*>(src);
    }
}

// ------------------------------------------------------------------ decode --
// Persistent, warp-specialised kernel. Each CTA (two per SM) runs
// kConsumerWarps consumer warps and two producer warps until the global unit
// counter runs past the unit list (units are sorted longest first, so the
// counter hands them out in LPT order):
//   fetcher   claims the next unit, publishes its descriptor and tile words
//             in one of two shared-memory unit slots and stages a tensor
//             unit's query rows with TMA -- up to two units ahead;
//   streamer  (one lane) streams the published units' tile pairs into a ring
//             of shared-memory stages with TMA bulk copies, with nothing but
//             stage waits between one unit and the next, so HBM keeps
//             streaming while the consumers finish a unit (split combine,
//             partial stores);
//   consumers run the attention math on each stage.
// Every wait is an mbarrier wait bounded in time; a wait that runs out sets
// the device error flag and the kernel carries on to a bounded exit.
struct UnitDesc {
    int tile_off, n_tiles, occ_off, row0, n_rows, slot_base, kvh, kind;
    int pos0;  // prefill: path position of the unit's first token
};

template <int HD>
struct Smem {
    static constexpr int kRowBytes = HD * 2;
    static constexpr int kHalfBytes = kStageTokens * kRowBytes;  // K or V of one stage
    static constexpr int kStageBytes = 2 * kHalfBytes;
    static constexpr int kRingBytes = kStages * kStageBytes;
    // split combine: the (kConsumerWarps - 1) warps that hand over their
    // state, 16 rows x kParkPitch floats each (o in columns [0, HD), m and l
    // in HD and HD + 1; the pitch makes the float2 accesses of a half warp
    // hit 32 distinct banks); the CUDA-core combine (4 x 8 rows x HD + 64
    // floats) fits in the same region
    static constexpr int kParkPitch = HD + 8;
    static constexpr int kParkFloats = (kConsumerWarps - 1) * 16 * kParkPitch;
    // the query rows of one tensor unit (64 rows x HD bf16), staged by TMA one
    // row per copy at a 16-byte-padded pitch so ldmatrix rows fall in
    // distinct bank groups
    static constexpr int kQPitch = HD * 2 + 16;
    static constexpr int kQBytes = kConsumerWarps * 16 * kQPitch;
    static constexpr int kBytes = kRingBytes + kParkFloats * 4 + kQBytes;
    // the CUDA-core kind stages no query rows and combines through a smaller
    // park (per warp: 8 maxima, 8 sums, 8 rows of HD), followed by its score
    // scratch ([warp][64 tokens][8 rows]); at ~90 KB two CTAs share an SM
    static constexpr int kCcParkFloats = kConsumerWarps * 8 * (2 + HD);
    static constexpr int kCcScratchFloats = kConsumerWarps * kStageTokens * 8;
    static constexpr int kCcBytes = kRingBytes + (kCcParkFloats + kCcScratchFloats) * 4;
};

template <int HD, int KIND>
constexpr int decode_smem() {
    return KIND == KIND_CUDA_CORE ? Smem<HD>::kCcBytes : Smem<HD>::kBytes;
}

// Shared control block of one CTA.
struct Ctl {
    uint64_t full[kStages];   // stage filled (producer arrival + TMA bytes)
    uint64_t empty[kStages];  // stage consumed (one arrival per consumer warp)
    uint64_t ufull[2];        // unit slot published
    uint64_t uempty[2];       // unit slot read by every consumer warp
    uint64_t csync;           // consumer-only barrier (split combine)
    uint64_t qfull;           // the current tensor unit's query rows landed
    uint64_t qempty;          // every consumer warp holds its query fragments
    int valid[kStages][2];    // valid tokens of the stage's two tiles (0: no tile)
    int unit[2];              // published unit index (-1: no more units)
    int desc[2][kUnitWords + 1];  // published unit descriptor (+ path position)
    int tiles[2][kMaxUnitTiles];  // published unit's tile words
    int abort;
};

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

template <typename CtlT>
__device__ __forceinline__ void note_timeout(const DecodeArgs& a, CtlT& c, int code) {
    atomicOr(a.err, code);
    *reinterpret_cast<volatile int*>(&c.abort) = 1;
}

// Producer: issue the bulk copies of one tile pair (tile words w[0..1],
// w = -1 for a missing second tile) into stage `st`, and record the pair's
// valid token counts for the consumers.
template <int HD, typename CtlT>
__device__ __forceinline__ void issue_pair(const DecodeArgs& a, CtlT& c, int kvh, uint8_t* ring, const int32_t (&w)[2],
                                           int st) {
    constexpr int RB = HD * 2;
    uint8_t* sk = ring + st * Smem<HD>::kStageBytes;
    uint8_t* sv = sk + Smem<HD>::kHalfBytes;
    const uint32_t bar = smem_u32(&c.full[st]);
    int valid[2] = {0, 0};
    uint32_t bytes = 0;
    for (int j = 0; j < 2; ++j)
        if (w[j] >= 0 && check(tile_word_ok(w[j], a.ext.pool_blocks), a.err)) {  // a bad word: a missing tile
            valid[j] = (w[j] & ((1 << kTileValidBits) - 1)) + 1;
            bytes += 2u * (uint32_t)(valid[j] * RB);
        }
    c.valid[st][0] = valid[0];
    c.valid[st][1] = valid[1];
    mbar_arrive_expect_tx(bar, bytes);  // release: the valid counts are visible to the stage's waiters
    // a tile is HD/64 halves of 32 rows x 128 B; the stage holds each half
    // for 64 rows, so tile j's half h lands at h * 64 * 128 + j * 32 * 128
    for (int j = 0; j < 2; ++j) {
        if (!valid[j]) continue;
        const int64_t blk = w[j] >> kTileValidBits;
        const uint8_t* src = a.pool + blk * a.block_bytes + (int64_t)kvh * a.head_bytes;
#pragma unroll
        for (int h = 0; h < HD / 64; ++h) {
            const int so = h * kBlockTokens * 128, dofs = h * kStageTokens * 128 + j * kBlockTokens * 128;
            if (!a.kv_read_once) {  // blocks re-read by other units (prefill, no-share control): keep them in L2
                bulk_g2s(smem_u32(sk + dofs), src + so, valid[j] * 128, bar);
                bulk_g2s(smem_u32(sv + dofs), src + (int64_t)a.hkv * a.head_bytes + so, valid[j] * 128, bar);
            } else {
                const uint64_t pol = l2_evict_first();
                bulk_g2s_hint(smem_u32(sk + dofs), src + so, valid[j] * 128, bar, pol);
                bulk_g2s_hint(smem_u32(sv + dofs), src + (int64_t)a.hkv * a.head_bytes + so, valid[j] * 128, bar, pol);
            }
        }
    }
}

// Consumer side of the stage ring (one instance per consumer warp).
struct RingReader {
    Ctl* c;
    uint8_t* ring;
    int stage;
    uint32_t phase;
    uint32_t sync_phase;
    uint32_t q_phase;

    template <int HD>
    __device__ __forceinline__ const uint8_t* acquire(const DecodeArgs& a, int& v0, int& v1) {
        if (!mbar_wait(smem_u32(&c->full[stage]), phase)) note_timeout(a, *c, 1);
        v0 = c->valid[stage][0];
        v1 = c->valid[stage][1];
        return ring + stage * Smem<HD>::kStageBytes;
    }
    __device__ __forceinline__ void release(int lane) {
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&c->empty[stage]));
        if (++stage == kStages) {
            stage = 0;
            phase ^= 1;
        }
    }
    // barrier of the consumer warps only (the producer never takes part)
    __device__ __forceinline__ void consumers_sync(const DecodeArgs& a, int lane) {
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&c->csync));
        if (!mbar_wait(smem_u32(&c->csync), sync_phase)) note_timeout(a, *c, 4);
        sync_phase ^= 1;
    }
};

// ---- CUDA-core path: <= 16 rows, 8 rows per warp ------------------------
// Lane layout: LPT = HD/8 lanes share one token (8 dims each, one 16-byte
// chunk), TPS = 32/LPT tokens per warp step. Dot products over the LPT lanes
// of a token are finished by a transposing butterfly: each level halves the
// number of rows a lane carries, so 8 rows cost 7 shuffles instead of 8x4.
template <int HD>
struct CudaCorePath {
    static constexpr int LPT = HD / 8;
    static constexpr int TPS = 32 / LPT;
    static constexpr int NR = 8;

    // acc[0..7] -> lane keeps one row's full sum; returns it.
    __device__ __forceinline__ static float transpose_reduce(float (&acc)[NR], int lane) {
        if (LPT == 16) {
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const bool up = lane & 8;
                const float send = up ? acc[i] : acc[i + 4];
                const float keep = up ? acc[i + 4] : acc[i];
                acc[i] = keep + __shfl_xor_sync(0xffffffffu, send, 8);
            }
#pragma unroll
            for (int i = 0; i < 2; ++i) {
                const bool up = lane & 4;
                const float send = up ? acc[i] : acc[i + 2];
                const float keep = up ? acc[i + 2] : acc[i];
                acc[i] = keep + __shfl_xor_sync(0xffffffffu, send, 4);
            }
            {
                const bool up = lane & 2;
                const float send = up ? acc[0] : acc[1];
                const float keep = up ? acc[1] : acc[0];
                acc[0] = keep + __shfl_xor_sync(0xffffffffu, send, 2);
            }
            return acc[0] + __shfl_xor_sync(0xffffffffu, acc[0], 1);  // row (lane >> 1) & 7
        } else {
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const bool up = lane & 4;
                const float send = up ? acc[i] : acc[i + 4];
                const float keep = up ? acc[i + 4] : acc[i];
                acc[i] = keep + __shfl_xor_sync(0xffffffffu, send, 4);
            }
#pragma unroll
            for (int i = 0; i < 2; ++i) {
                const bool up = lane & 2;
                const float send = up ? acc[i] : acc[i + 2];
                const float keep = up ? acc[i + 2] : acc[i];
                acc[i] = keep + __shfl_xor_sync(0xffffffffu, send, 2);
            }
            const bool up = lane & 1;
            const float send = up ? acc[0] : acc[1];
            const float keep = up ? acc[1] : acc[0];
            return keep + __shfl_xor_sync(0xffffffffu, send, 1);  // row lane & 7
        }
    }
    __device__ __forceinline__ static int reduce_row(int lane) { return LPT == 16 ? (lane >> 1) & 7 : lane & 7; }
    __device__ __forceinline__ static bool reduce_writer(int lane) { return LPT == 16 ? (lane & 1) == 0 : true; }

    __device__ static void unit(const DecodeArgs& a, const UnitDesc& u, RingReader& rr, float* park,
                                float* scratch) {
        const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
        const int n_rg = (u.n_rows + NR - 1) / NR;  // 1 or 2 row groups
        const int n_sp = kConsumerWarps / n_rg;     // token splits
        const int rg = warp % n_rg, sp = warp / n_rg;
        const int TW = kStageTokens / n_sp;  // tokens of a stage this warp handles
        const int dg = lane % LPT, ts = lane / LPT;

        // q rows of this warp, 8 dims per lane, pre-scaled to the log2 domain;
        // packed in row pairs (rows 2i, 2i + 1) for the f32x2 dot products
        float qf[NR][8];
#pragma unroll
        for (int r = 0; r < NR; ++r) {
            const int rr_ = rg * NR + r;
            if (rr_ < u.n_rows) {
                const int item_row = u.row0 + rr_;
                int occ = a.occ[u.occ_off + item_row / a.group];
                if (!check(in_range(occ, a.ext.n), a.err)) occ = 0;
                const int qh = u.kvh * a.group + item_row % a.group;
                const uint4 w = *reinterpret_cast<const uint4*>(a.q + ((int64_t)occ * a.hq + qh) * HD + dg * 8);
                const uint32_t ww[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    qf[r][2 * k] = bf_lo(ww[k]) * a.qk_scale_log2;
                    qf[r][2 * k + 1] = bf_hi(ww[k]) * a.qk_scale_log2;
                }
            } else {
#pragma unroll
                for (int k = 0; k < 8; ++k) qf[r][k] = 0.f;
            }
        }
        uint64_t q2[NR / 2][8];
#pragma unroll
        for (int i = 0; i < NR / 2; ++i)
#pragma unroll
            for (int k = 0; k < 8; ++k) q2[i][k] = f2_pack(qf[2 * i][k], qf[2 * i + 1][k]);
        // o of each row in dimension pairs (k, k + 1)
        uint64_t o2[NR][4];
#pragma unroll
        for (int r = 0; r < NR; ++r)
#pragma unroll
            for (int k = 0; k < 4; ++k) o2[r][k] = 0ull;
        // running max / sum of row (lane >> 2), replicated over its quad
        float m_run = -INFINITY, l_run = 0.f;
        float* sc = scratch + warp * (kStageTokens * NR);  // [token][row]

        const int n_pairs = (u.n_tiles + 1) / 2;
        for (int pr = 0; pr < n_pairs; ++pr) {
            int v0, v1;
            const uint8_t* sk = rr.acquire<HD>(a, v0, v1);
            const uint8_t* sv = sk + Smem<HD>::kHalfBytes;
            const int tbase = sp * TW;
            // ---- scores: s[t][row] for this warp's TW tokens
            for (int s0 = 0; s0 < TW; s0 += TPS) {
                const int t = tbase + s0 + ts;  // token within the stage
                const uint4 kw = *reinterpret_cast<const uint4*>(sk + kv_off<kStageTokens>(t, dg));
                const uint32_t kk[4] = {kw.x, kw.y, kw.z, kw.w};
                // two rows per f32x2 FMA; each row's sum in the same order
                // (and rounding) as a scalar fmaf chain over k
                uint64_t acc2[NR / 2];
#pragma unroll
                for (int i = 0; i < NR / 2; ++i) acc2[i] = 0ull;
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    const float k0 = bf_lo(kk[k]), k1 = bf_hi(kk[k]);
                    const uint64_t kb0 = f2_pack(k0, k0), kb1 = f2_pack(k1, k1);
#pragma unroll
                    for (int i = 0; i < NR / 2; ++i) acc2[i] = f2_fma(q2[i][2 * k], kb0, acc2[i]);
#pragma unroll
                    for (int i = 0; i < NR / 2; ++i) acc2[i] = f2_fma(q2[i][2 * k + 1], kb1, acc2[i]);
                }
                float acc[NR];
#pragma unroll
                for (int i = 0; i < NR / 2; ++i) f2_unpack(acc2[i], acc[2 * i], acc[2 * i + 1]);
                float s = transpose_reduce(acc, lane);
                const int valid = (t & 31) < ((t < kBlockTokens) ? v0 : v1);
                if (!valid) s = -INFINITY;
                if (reduce_writer(lane)) sc[(s0 + ts) * NR + reduce_row(lane)] = s;
            }
            __syncwarp();
            // ---- online softmax: quad r owns row r, tokens strided by 4
            float alpha;
            {
                const int r = lane >> 2, q4 = lane & 3;
                float mx = -INFINITY;
                for (int t = q4; t < TW; t += 4) mx = fmaxf(mx, sc[t * NR + r]);
                mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
                mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
                const float m_new = fmaxf(m_run, mx);
                const float m_use = (m_new == -INFINITY) ? 0.f : m_new;  // all masked so far
                alpha = fast_exp2(m_run - m_use);
                float sum = 0.f;
                for (int t = q4; t < TW; t += 4) {
                    const float p = fast_exp2(sc[t * NR + r] - m_use);
                    sc[t * NR + r] = p;
                    sum += p;
                }
                sum += __shfl_xor_sync(0xffffffffu, sum, 1);
                sum += __shfl_xor_sync(0xffffffffu, sum, 2);
                l_run = l_run * alpha + sum;
                m_run = m_new;
            }
            __syncwarp();
            // ---- rescale and accumulate P.V
            if (!__all_sync(0xffffffffu, alpha == 1.f)) {
                const uint64_t nz = f2_pack(-0.f, -0.f);  // x * al + (-0) = x * al exactly
#pragma unroll
                for (int r = 0; r < NR; ++r) {
                    const float al = __shfl_sync(0xffffffffu, alpha, r * 4);
                    const uint64_t al2 = f2_pack(al, al);
#pragma unroll
                    for (int k = 0; k < 4; ++k) o2[r][k] = f2_fma(o2[r][k], al2, nz);
                }
            }
            for (int s0 = 0; s0 < TW; s0 += TPS) {
                const int t = tbase + s0 + ts;
                const uint4 vw = *reinterpret_cast<const uint4*>(sv + kv_off<kStageTokens>(t, dg));
                const uint32_t vv[4] = {vw.x, vw.y, vw.z, vw.w};
                uint64_t v2[4];  // dimension pairs (2k, 2k + 1)
#pragma unroll
                for (int k = 0; k < 4; ++k) v2[k] = f2_pack(bf_lo(vv[k]), bf_hi(vv[k]));
                const float4 p0 = *reinterpret_cast<const float4*>(&sc[(s0 + ts) * NR]);
                const float4 p1 = *reinterpret_cast<const float4*>(&sc[(s0 + ts) * NR + 4]);
                const float p[NR] = {p0.x, p0.y, p0.z, p0.w, p1.x, p1.y, p1.z, p1.w};
#pragma unroll
                for (int r = 0; r < NR; ++r) {
                    const uint64_t pb = f2_pack(p[r], p[r]);
#pragma unroll
                    for (int k = 0; k < 4; ++k) o2[r][k] = f2_fma(pb, v2[k], o2[r][k]);
                }
            }
            __syncwarp();  // sc is rewritten by the next stage's scores
            rr.release(lane);
        }
        float o[NR][8];
#pragma unroll
        for (int r = 0; r < NR; ++r)
#pragma unroll
            for (int k = 0; k < 4; ++k) f2_unpack(o2[r][k], o[r][2 * k], o[r][2 * k + 1]);
        // ---- fold the TPS token slots of each lane column
#pragma unroll
        for (int off = LPT; off < 32; off <<= 1)
#pragma unroll
            for (int r = 0; r < NR; ++r)
#pragma unroll
                for (int k = 0; k < 8; ++k) o[r][k] += __shfl_xor_sync(0xffffffffu, o[r][k], off);
        // ---- combine the token splits of each row group through shared memory
        float* cm = park;                 // [warp][NR] max
        float* cl = cm + 4 * NR;          // [warp][NR] sum
        float* co = cl + 4 * NR;          // [warp][NR][HD]
        rr.consumers_sync(a, lane);       // the previous unit's combine is done with the park
        if ((lane & 3) == 0) {
            cm[warp * NR + (lane >> 2)] = m_run;
            cl[warp * NR + (lane >> 2)] = l_run;
        }
        if (ts == 0) {
#pragma unroll
            for (int r = 0; r < NR; ++r) {
                float4* dst = reinterpret_cast<float4*>(co + (warp * NR + r) * HD + dg * 8);
                dst[0] = make_float4(o[r][0], o[r][1], o[r][2], o[r][3]);
                dst[1] = make_float4(o[r][4], o[r][5], o[r][6], o[r][7]);
            }
        }
        rr.consumers_sync(a, lane);
        if (sp != 0) return;
        // this warp writes rows rg*8 .. rg*8+7; lanes: row = lane / 4, 4 lanes per row
        const int r = lane >> 2, q4 = lane & 3;
        const int rr_ = rg * NR + r;
        float M = -INFINITY;
        for (int s = 0; s < n_sp; ++s) M = fmaxf(M, cm[(s * n_rg + rg) * NR + r]);
        float L = 0.f;
        float w[kConsumerWarps];
        for (int s = 0; s < n_sp; ++s) {
            const float ms = cm[(s * n_rg + rg) * NR + r];
            w[s] = (ms == -INFINITY) ? 0.f : fast_exp2(ms - M);
            L += w[s] * cl[(s * n_rg + rg) * NR + r];
        }
        if (rr_ < u.n_rows) {
            const int item_row = u.row0 + rr_;
            const int slot = u.slot_base + item_row / a.group;
            const int qh = u.kvh * a.group + item_row % a.group;
            float* dst = a.part_o + ((int64_t)slot * a.hq + qh) * HD;
            const float inv = 1.f / L;
            const uint64_t pol = l2_evict_last();
            for (int d = q4 * 4; d < HD; d += 16) {
                float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
                for (int s = 0; s < n_sp; ++s) {
                    const float4 x = *reinterpret_cast<const float4*>(co + ((s * n_rg + rg) * NR + r) * HD + d);
                    acc.x += w[s] * x.x;
                    acc.y += w[s] * x.y;
                    acc.z += w[s] * x.z;
                    acc.w += w[s] * x.w;
                }
                st_f4_hint(dst + d, make_float4(acc.x * inv, acc.y * inv, acc.z * inv, acc.w * inv), pol);
            }
            if (q4 == 0) a.part_lse[(int64_t)slot * a.hq + qh] = M + __log2f(L);
        }
    }
};

// ---- tensor-core path: 16-row MMA tiles, one per warp -------------------
// CAUSAL (prefill): row r sees only the first vis[occurrence of r] tokens of
// its path; the unit's tiles start at path position u.pos0.
template <int HD>
struct TensorPath {
    static constexpr int KS = HD / 16;  // k-steps of Q.K^T
    static constexpr int NT = HD / 8;   // n-tiles of the output

    template <bool CAUSAL>
    __device__ static void unit(const DecodeArgs& a, const UnitDesc& u, RingReader& rr, float* park,
                                const uint8_t* qbuf) {
        const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
        const int n_mt = (u.n_rows + 15) / 16;  // 1..4
        const int n_sp = (n_mt == 1) ? 4 : (n_mt == 2) ? 2 : 1;
        const int mt = warp % n_mt, sp = warp / n_mt;
        const bool active = sp < n_sp;
        const int TW = kStageTokens / n_sp;  // 16, 32 or 64 tokens per stage
        const int g4 = lane >> 2, c4 = lane & 3;

        // Q fragments from the unit's staged query rows (row r of the unit at
        // qbuf + r * HD * 2); rows past n_rows are zero
        uint32_t qa[KS][4];
        if (!mbar_wait(smem_u32(&rr.c->qfull), rr.q_phase)) note_timeout(a, *rr.c, 1);
        rr.q_phase ^= 1;
        if (active) {
            const int mi = lane >> 3, ri = lane & 7;
            const uint32_t qb = smem_u32(qbuf) + (mt * 16 + (mi & 1) * 8 + ri) * Smem<HD>::kQPitch + (mi >> 1) * 16;
            const bool lo_ok = mt * 16 + g4 < u.n_rows, hi_ok = mt * 16 + g4 + 8 < u.n_rows;
#pragma unroll
            for (int ks = 0; ks < KS; ++ks) {
                ldsm_x4(qb + ks * 32, qa[ks][0], qa[ks][1], qa[ks][2], qa[ks][3]);
                if (!lo_ok) qa[ks][0] = qa[ks][2] = 0u;
                if (!hi_ok) qa[ks][1] = qa[ks][3] = 0u;
            }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&rr.c->qempty));
        float o[NT][4];
#pragma unroll
        for (int j = 0; j < NT; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;
        float m_run[2] = {-INFINITY, -INFINITY}, l_run[2] = {0.f, 0.f};  // rows g4, g4 + 8 (lane partial l)
        int vis[2] = {0, 0}, pos = u.pos0;  // CAUSAL: visible tokens of rows g4, g4 + 8; pair position
        if constexpr (CAUSAL) {
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const int r = mt * 16 + g4 + 8 * h;
                if (r >= u.n_rows) {
                    vis[h] = 0x7fffffff;
                    continue;
                }
                const int occ = a.occ[u.occ_off + (u.row0 + r) / a.group];
                vis[h] = check(in_range(occ, a.ext.n), a.err) ? a.vis[occ] : 0;
            }
        }

        const int n_pairs = (u.n_tiles + 1) / 2;
        for (int pr = 0; pr < n_pairs; ++pr) {
            int v0, v1;
            const uint8_t* stage = rr.acquire<HD>(a, v0, v1);
            const int pos_t0 = pos, pos_t1 = pos + v0;  // path positions of the pair's two tiles
            pos += v0 + v1;
            if (active) {
                const uint32_t sk = smem_u32(stage);
                const uint32_t sv = sk + Smem<HD>::kHalfBytes;
                const int tbase = sp * TW;
                for (int kb = 0; kb < TW; kb += 16) {
                    // S = Q K^T for 16 tokens: two n8 tiles
                    float s[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
                    const int mi = lane >> 3, ri = lane & 7;
#pragma unroll
                    for (int ks = 0; ks < KS; ++ks) {
                        const int tok = tbase + kb + (mi >> 1) * 8 + ri;
                        const int ch = ks * 2 + (mi & 1);
                        uint32_t b0, b1, b2, b3;
                        ldsm_x4(sk + kv_off<kStageTokens>(tok, ch), b0, b1, b2, b3);
                        mma_bf16(s[0], qa[ks], b0, b1);
                        mma_bf16(s[1], qa[ks], b2, b3);
                    }
                    // scale, mask, online softmax over these 16 tokens
                    float mx[2] = {-INFINITY, -INFINITY};
#pragma unroll
                    for (int j = 0; j < 2; ++j)
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            const int tok = tbase + kb + j * 8 + 2 * c4 + (e & 1);
                            const int lim = (tok < kBlockTokens) ? v0 : v1;
                            bool keep = (tok & 31) < lim;
                            if constexpr (CAUSAL)
                                keep = keep && ((tok < kBlockTokens ? pos_t0 : pos_t1) + (tok & 31)) < vis[e >> 1];
                            const float x = keep ? s[j][e] * a.qk_scale_log2 : -INFINITY;
                            s[j][e] = x;
                            mx[e >> 1] = fmaxf(mx[e >> 1], x);
                        }
                    float alpha[2], m_use[2];
#pragma unroll
                    for (int h = 0; h < 2; ++h) {
                        mx[h] = fmaxf(mx[h], __shfl_xor_sync(0xffffffffu, mx[h], 1));
                        mx[h] = fmaxf(mx[h], __shfl_xor_sync(0xffffffffu, mx[h], 2));
                        const float m_new = fmaxf(m_run[h], mx[h]);
                        m_use[h] = (m_new == -INFINITY) ? 0.f : m_new;
                        alpha[h] = fast_exp2(m_run[h] - m_use[h]);
                        m_run[h] = m_new;
                        l_run[h] *= alpha[h];
                    }
                    // A fragment of P: (row g, tok 2c..) (row g+8, tok 2c..) (row g, tok 2c+8..) (row g+8, ..)
                    uint32_t pa[4];
#pragma unroll
                    for (int j = 0; j < 2; ++j) {
                        const float p0 = fast_exp2(s[j][0] - m_use[0]), p1 = fast_exp2(s[j][1] - m_use[0]);
                        const float p2 = fast_exp2(s[j][2] - m_use[1]), p3 = fast_exp2(s[j][3] - m_use[1]);
                        l_run[0] += p0 + p1;
                        l_run[1] += p2 + p3;
                        pa[2 * j] = pack_bf16(p0, p1);
                        pa[2 * j + 1] = pack_bf16(p2, p3);
                    }
#pragma unroll
                    for (int j = 0; j < NT; ++j) {
                        o[j][0] *= alpha[0];
                        o[j][1] *= alpha[0];
                        o[j][2] *= alpha[1];
                        o[j][3] *= alpha[1];
                    }
                    // O += P V: V^T fragments via ldmatrix.trans, two n8 tiles per load
#pragma unroll
                    for (int dp = 0; dp < HD / 16; ++dp) {
                        const int tok = tbase + kb + (mi & 1) * 8 + ri;
                        const int ch = dp * 2 + (mi >> 1);
                        uint32_t b0, b1, b2, b3;
                        ldsm_x4_t(sv + kv_off<kStageTokens>(tok, ch), b0, b1, b2, b3);
                        mma_bf16(o[2 * dp], pa, b0, b1);
                        mma_bf16(o[2 * dp + 1], pa, b2, b3);
                    }
                }
            }
            rr.release(lane);
        }
        // full row sums over the quad
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            l_run[h] += __shfl_xor_sync(0xffffffffu, l_run[h], 1);
            l_run[h] += __shfl_xor_sync(0xffffffffu, l_run[h], 2);
        }
        if (n_sp > 1) {
            // token splits of one M-tile meet in shared memory: [warp][16 rows][pitch]
            constexpr int PP = Smem<HD>::kParkPitch;
            constexpr int PW = 16 * PP;
            rr.consumers_sync(a, lane);  // the previous unit's combine is done with the park
            if (active && sp > 0) {
                float* p = park + ((sp - 1) * n_mt + mt) * PW;
#pragma unroll
                for (int j = 0; j < NT; ++j)
#pragma unroll
                    for (int h = 0; h < 2; ++h)
                        *reinterpret_cast<float2*>(&p[(g4 + 8 * h) * PP + j * 8 + 2 * c4]) =
                            make_float2(o[j][2 * h], o[j][2 * h + 1]);
                if (c4 == 0)
#pragma unroll
                    for (int h = 0; h < 2; ++h)
                        *reinterpret_cast<float2*>(&p[(g4 + 8 * h) * PP + HD]) = make_float2(m_run[h], l_run[h]);
            }
            rr.consumers_sync(a, lane);
            if (active && sp == 0) {
                for (int s = 1; s < n_sp; ++s) {
                    const float* p = park + ((s - 1) * n_mt + mt) * PW;
#pragma unroll
                    for (int h = 0; h < 2; ++h) {
                        const int row = g4 + 8 * h;
                        const float2 ml = *reinterpret_cast<const float2*>(&p[row * PP + HD]);
                        const float ms = ml.x, ls = ml.y;
                        const float M = fmaxf(m_run[h], ms);
                        const float Mu = (M == -INFINITY) ? 0.f : M;
                        const float wa = fast_exp2(m_run[h] - Mu), wb = fast_exp2(ms - Mu);
#pragma unroll
                        for (int j = 0; j < NT; ++j) {
                            const float2 x = *reinterpret_cast<const float2*>(&p[row * PP + j * 8 + 2 * c4]);
                            o[j][2 * h] = o[j][2 * h] * wa + wb * x.x;
                            o[j][2 * h + 1] = o[j][2 * h + 1] * wa + wb * x.y;
                        }
                        l_run[h] = l_run[h] * wa + ls * wb;
                        m_run[h] = M;
                    }
                }
            }
        }
        if (!active || sp != 0) return;
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int r = mt * 16 + g4 + 8 * h;
            if (r >= u.n_rows) continue;
            const int item_row = u.row0 + r;
            const int qh = u.kvh * a.group + item_row % a.group;
            const float inv = 1.f / l_run[h];
            if (CAUSAL && u.slot_base < 0) {  // the row's only unit: final O and LSE
                const int occ = a.occ[u.occ_off + item_row / a.group];
                if (!check(in_range(occ, a.ext.n), a.err)) continue;
                uint16_t* dst = a.out + ((int64_t)occ * a.hq + qh) * HD;
#pragma unroll
                for (int j = 0; j < NT; ++j)
                    *reinterpret_cast<uint32_t*>(dst + j * 8 + 2 * c4) = pack_bf16(o[j][2 * h] * inv, o[j][2 * h + 1] * inv);
                if (c4 == 0) a.out_lse[(int64_t)occ * a.hq + qh] = (m_run[h] + __log2f(l_run[h])) * 0.69314718055994531f;
                continue;
            }
            const int slot = u.slot_base + item_row / a.group;
            float* dst = a.part_o + ((int64_t)slot * a.hq + qh) * HD;
            const uint64_t pol = l2_evict_last();
#pragma unroll
            for (int j = 0; j < NT; ++j) st_f2_hint(dst + j * 8 + 2 * c4, o[j][2 * h] * inv, o[j][2 * h + 1] * inv, pol);
            if (c4 == 0) a.part_lse[(int64_t)slot * a.hq + qh] = m_run[h] + __log2f(l_run[h]);
        }
    }
};

// Fetcher warp: claim units, publish descriptor + tile words, stage a tensor
// unit's query rows (one bulk copy per leaf occurrence group, lanes in
// parallel).
template <int HD, int KIND>
__device__ void fetch_units(const DecodeArgs& a, Ctl& c, uint8_t* qbuf) {
    const int lane = threadIdx.x & 31;
    volatile int* abort = &c.abort;
    for (int k = 0;; ++k) {
        const int q = k & 1;
        // the slot is free once the consumers and the streamer are done with unit k-2
        if (!mbar_wait(smem_u32(&c.uempty[q]), ((k >> 1) & 1) ^ 1)) note_timeout(a, c, 2);
        int u = -1;
        if (lane == 0) {
            u = *abort ? -1 : a.unit_begin + atomicAdd(a.counter, 1);
            if (u >= a.unit_end) u = -1;
        }
        u = __shfl_sync(0xffffffffu, u, 0);
        const int word = (u >= 0 && lane < kUnitWords) ? a.units[(int64_t)u * kUnitWords + lane] : 0;
        UnitDesc d;
        d.tile_off = __shfl_sync(0xffffffffu, word, U_TILE_OFF);
        d.n_tiles = __shfl_sync(0xffffffffu, word, U_N_TILES);
        d.occ_off = __shfl_sync(0xffffffffu, word, U_OCC_OFF);
        d.row0 = __shfl_sync(0xffffffffu, word, U_ROW0);
        d.n_rows = __shfl_sync(0xffffffffu, word, U_N_ROWS);
        d.slot_base = __shfl_sync(0xffffffffu, word, U_SLOT_BASE);
        d.kvh = __shfl_sync(0xffffffffu, word, U_KVH);
        d.kind = __shfl_sync(0xffffffffu, word, U_KIND);
        if (kBoundsCheck && u >= 0 &&
            !(d.kind == (KIND == KIND_CUDA_CORE ? KIND_CUDA_CORE : KIND_TENSOR) &&
              unit_ok(d.tile_off, d.n_tiles, d.occ_off, d.row0, d.n_rows, d.slot_base, d.kvh,
                      unit_rows_limit(d.kind), KIND == KIND_PREFILL, a.ext))) {
            if (lane == 0) atomicOr(a.err, kErrBounds);  // a bad unit record: this CTA takes no more units
            u = -1;
        }
        if (u >= 0)
            for (int t = lane; t < d.n_tiles; t += 32) c.tiles[q][t] = a.tiles[d.tile_off + t];
        if (lane == 0) {
            volatile int* dw = c.desc[q];
            dw[U_TILE_OFF] = d.tile_off;
            dw[U_N_TILES] = d.n_tiles;
            dw[U_OCC_OFF] = d.occ_off;
            dw[U_ROW0] = d.row0;
            dw[U_N_ROWS] = d.n_rows;
            dw[U_SLOT_BASE] = d.slot_base;
            dw[U_KVH] = d.kvh;
            dw[U_KIND] = d.kind;
            dw[kUnitWords] = (u >= 0 && a.unit_pos) ? a.unit_pos[u] : 0;
            *reinterpret_cast<volatile int*>(&c.unit[q]) = u;
        }
        __threadfence_block();  // every lane's tile-word stores, before lane 0 publishes
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&c.ufull[q]));  // release: slot visible to its readers
        if (u < 0) return;
        if constexpr (KIND == KIND_TENSOR || KIND == KIND_PREFILL) {
            // query rows of the unit: item row row0 + r is q-head
            // kvh * g + (row0 + r) % g of occurrence occ[(row0 + r) / g]
            if (!mbar_wait(smem_u32(&c.qempty), (k & 1) ^ 1)) note_timeout(a, c, 2);
            if (lane == 0) mbar_arrive_expect_tx(smem_u32(&c.qfull), (uint32_t)d.n_rows * HD * 2);
            __syncwarp();
            const int g = a.group;
            for (int r = lane; r < d.n_rows; r += 32) {  // one 2*HD-byte copy per row
                const int item_row = d.row0 + r;
                int occ = a.occ[d.occ_off + item_row / g];
                if (!check(in_range(occ, a.ext.n), a.err)) occ = 0;
                const uint16_t* src = a.q + ((int64_t)occ * a.hq + d.kvh * g + item_row % g) * HD;
                bulk_g2s(smem_u32(qbuf + r * Smem<HD>::kQPitch), src, HD * 2, smem_u32(&c.qfull));
            }
        }
    }
}

// Streamer (one lane): stream the tile pairs of each published unit.
template <int HD>
__device__ void stream_units(const DecodeArgs& a, Ctl& c, uint8_t* ring) {
    int stage = 0;
    uint32_t phase = 0;
    for (int k = 0;; ++k) {
        const int q = k & 1;
        if (!mbar_wait(smem_u32(&c.ufull[q]), (k >> 1) & 1)) {
            note_timeout(a, c, 2);
            return;
        }
        const int u = *reinterpret_cast<volatile int*>(&c.unit[q]);
        if (u < 0) return;
        const int n_tiles = *reinterpret_cast<volatile int*>(&c.desc[q][U_N_TILES]);
        const int kvh = *reinterpret_cast<volatile int*>(&c.desc[q][U_KVH]);
        const volatile int* tw = c.tiles[q];
        const int n_pairs = (n_tiles + 1) / 2;
        for (int pr = 0; pr < n_pairs; ++pr) {
            const int32_t w[2] = {tw[2 * pr], 2 * pr + 1 < n_tiles ? tw[2 * pr + 1] : -1};
            if (!mbar_wait(smem_u32(&c.empty[stage]), phase ^ 1)) note_timeout(a, c, 2);
            fence_proxy_async();
            issue_pair<HD>(a, c, kvh, ring, w, stage);
            if (++stage == kStages) {
                stage = 0;
                phase ^= 1;
            }
        }
        mbar_arrive(smem_u32(&c.uempty[q]));  // done with the slot's tile words
    }
}

template <int HD, int KIND>
__device__ void consume(const DecodeArgs& a, Ctl& c, uint8_t* ring, float* park, const uint8_t* qbuf,
                        float* scratch) {
    const int lane = threadIdx.x & 31;
    RingReader rr{&c, ring, 0, 0, 0, 0};
    for (int k = 0;; ++k) {
        const int q = k & 1;
        if (!mbar_wait(smem_u32(&c.ufull[q]), (k >> 1) & 1)) {
            note_timeout(a, c, 8);
            return;
        }
        const int u = *reinterpret_cast<volatile int*>(&c.unit[q]);
        UnitDesc d;
        {
            const volatile int* dw = c.desc[q];
            d.tile_off = dw[U_TILE_OFF];
            d.n_tiles = dw[U_N_TILES];
            d.occ_off = dw[U_OCC_OFF];
            d.row0 = dw[U_ROW0];
            d.n_rows = dw[U_N_ROWS];
            d.slot_base = dw[U_SLOT_BASE];
            d.kvh = dw[U_KVH];
            d.kind = dw[U_KIND];
            d.pos0 = dw[kUnitWords];
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&c.uempty[q]));
        if (u < 0) return;
        if constexpr (KIND == KIND_TENSOR)
            TensorPath<HD>::template unit<false>(a, d, rr, park, qbuf);
        else if constexpr (KIND == KIND_PREFILL)
            TensorPath<HD>::template unit<true>(a, d, rr, park, qbuf);
        else
            CudaCorePath<HD>::unit(a, d, rr, park, scratch);
    }
}

// One persistent launch per unit kind (tensor units come first in the list),
// so each path gets its own register allocation.
template <int HD, int KIND>
__global__ void __launch_bounds__(kDecodeThreads, 2) decode_kernel(const DecodeArgs a) {
    extern __shared__ __align__(128) uint8_t smem[];
    __shared__ __align__(16) Ctl ctl;
    uint8_t* ring = smem;
    float* park = reinterpret_cast<float*>(smem + Smem<HD>::kRingBytes);
    uint8_t* qbuf = smem + Smem<HD>::kRingBytes + Smem<HD>::kParkFloats * 4;  // tensor kinds only
    float* cc_scratch = park + Smem<HD>::kCcParkFloats;                         // CUDA-core kind only
    const int tid = threadIdx.x, warp = tid >> 5;
    // zero the ring once: rows past a partial block are never copied and must
    // hold finite values (their probabilities are exactly 0)
    {
        uint4* r4 = reinterpret_cast<uint4*>(ring);
        for (int i = tid; i < Smem<HD>::kRingBytes / 16; i += kDecodeThreads) r4[i] = make_uint4(0, 0, 0, 0);
    }
    if (tid == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(smem_u32(&ctl.full[s]), 1);
            mbar_init(smem_u32(&ctl.empty[s]), kConsumerWarps);
        }
        for (int q = 0; q < 2; ++q) {
            mbar_init(smem_u32(&ctl.ufull[q]), 1);
            mbar_init(smem_u32(&ctl.uempty[q]), kConsumerWarps + 1);  // consumers + streamer
        }
        mbar_init(smem_u32(&ctl.csync), kConsumerWarps);
        mbar_init(smem_u32(&ctl.qfull), 1);
        mbar_init(smem_u32(&ctl.qempty), kConsumerWarps);
        ctl.abort = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    fence_proxy_async();
    __syncthreads();
    if (warp == kStreamerWarp) {
        if ((tid & 31) == 0) stream_units<HD>(a, ctl, ring);
        return;
    }
    if (warp == kFetcherWarp) {
        fetch_units<HD, KIND>(a, ctl, qbuf);
        return;
    }
    consume<HD, KIND>(a, ctl, ring, park, qbuf, cc_scratch);
}


// ---------------------------------------------------------- tcgen05 path --
// Units of 17..128 stacked query rows: Q.K^T and P.V run as tcgen05.mma
// (M = 128 rows, bf16 -> fp32) issued by one thread, accumulators in tensor
// memory. Warps: 0-3 softmax + epilogue (warp w owns TMEM lanes 32w..32w+31,
// i.e. query rows 32w..32w+31: one row per thread, no shuffles), 4 the K/V
// streamer, 5 the unit fetcher (also stages the unit's query rows in the
// swizzled operand layout), 6 the MMA issuer.
//   S = Q K^T    A = query rows (smem, K-major), B = K stage (smem, K-major),
//                D = S buffer (TMEM, 64 columns, double-buffered)
//   O += P V     A = P (TMEM, bf16 pairs written over the S buffer),
//                B = V stage (smem, MN-major), D = O (TMEM, HD columns)
// S of the next stage is issued before P.V of the current one, so the
// tensor core overlaps the softmax. O is rescaled only when a row's running
// max grows by more than 2^8 (p <= 256 stays exact in fp32 and ~bf16);
// otherwise the stale max is kept, which leaves O / l unchanged.
constexpr int kTcConsumerWarps = 4;
constexpr int kTcStreamerWarp = 4, kTcFetcherWarp = 5, kTcIssuerWarp = 6;
constexpr int kTcThreads = 7 * 32;
constexpr int kTcRows = 128;          // MMA M (unit rows padded to it)
constexpr uint32_t kTmemCols = 256;   // S0 [0,64) S1 [64,128) O [128, 128 + HD)
constexpr float kRescaleLog2 = 8.f;

template <int HD>
struct TcSmem {
    static constexpr int kStageBytes = 2 * (HD / 64) * kStageTokens * 128;  // K then V of 64 tokens
    static constexpr int kRingBytes = kStages * kStageBytes;
    static constexpr int kQBytes = (HD / 64) * kTcRows * 128;
    static constexpr int kBytes = kRingBytes + kQBytes + 1024;  // + slack to align to 1024
};

static_assert(kStages == 2, "the S buffers and the ring slots share their index");

struct CtlTc {
    // Each tcgen05.commit costs the issuing thread about as long as an MMA,
    // so one commit serves every waiter of the same completion: s_full[s]
    // also frees ring slot s's K half (the S buffer and the ring slot of a
    // stage share its index, kStages = 2), and vempty[s] also tells the
    // softmax that the P.V of the stage in slot s has finished.
    uint64_t kfull[kStages];   // K half of the stage landed (streamer + TMA bytes)
    uint64_t vfull[kStages];   // V half landed
    uint64_t vempty[kStages];  // V half read by P.V (issuer's commit)
    uint64_t ufull[2], uempty[2];
    uint64_t qfull;           // query rows staged (fetcher)
    uint64_t qempty;          // the unit's last Q.K^T done (issuer's commit)
    uint64_t s_full[2];       // S buffer holds scores, K half read (issuer's commit)
    uint64_t p_full[2];       // S buffer holds P (one arrival per consumer warp)
    uint64_t o_full;          // the unit's last P.V done (issuer's commit)
    uint64_t o_free;          // the epilogue has read O (one arrival per consumer warp)
    int valid[kStages][2];
    int unit[2];
    int desc[2][kUnitWords + 1];  // + path position of the unit's first token (prefill)
    int tiles[2][kMaxUnitTiles];
    uint32_t tmem;
    int abort;
};

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

__device__ __forceinline__ void tc_commit(uint32_t bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar) : "memory");
}

// sm_100 shared-memory matrix descriptor: 128-byte swizzle, version 1.
__device__ __forceinline__ uint64_t smem_desc(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
    return (uint64_t)((saddr >> 4) & 0x3FFF) | ((uint64_t)((lbo >> 4) & 0x3FFF) << 16) |
           ((uint64_t)((sbo >> 4) & 0x3FFF) << 32) | ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}

// Instruction descriptor, kind::f16: D fp32, A and B bf16, M = 128.
template <int N, bool B_MN_MAJOR>
__device__ __forceinline__ constexpr uint32_t mma_idesc() {
    return (1u << 4) | (1u << 7) | (1u << 10) | ((B_MN_MAJOR ? 1u : 0u) << 16) | ((uint32_t)(N >> 3) << 17) |
           ((uint32_t)(kTcRows >> 4) << 24);
}

__device__ __forceinline__ void mma_ss(uint32_t d, uint64_t a, uint64_t b, uint32_t idesc, uint32_t acc) {
    asm volatile(
        "{ .reg .pred p; setp.ne.b32 p, %4, 0; tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p; }" ::"r"(d),
        "l"(a), "l"(b), "r"(idesc), "r"(acc));
}

__device__ __forceinline__ void mma_ts(uint32_t d, uint32_t a_tmem, uint64_t b, uint32_t idesc, uint32_t acc) {
    asm volatile(
        "{ .reg .pred p; setp.ne.b32 p, %4, 0; tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p; }" ::"r"(d),
        "r"(a_tmem), "l"(b), "r"(idesc), "r"(acc));
}

// 32 consecutive TMEM columns of this thread's lane
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,"
        "%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
          "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]),
          "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
          "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// the same load without the wait, so two can be in flight
__device__ __forceinline__ void tmem_ld32_nowait(uint32_t taddr, uint32_t (&r)[32]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,"
        "%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
          "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]),
          "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
          "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
}

__device__ __forceinline__ void tmem_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }

__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&r)[32]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,"
        "%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
        "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]),
        "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(r[16]), "r"(r[17]), "r"(r[18]),
        "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]),
        "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
        : "memory");
    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ UnitDesc read_desc(const int* slot) {
    const volatile int* dw = slot;
    UnitDesc d;
    d.tile_off = dw[U_TILE_OFF];
    d.n_tiles = dw[U_N_TILES];
    d.occ_off = dw[U_OCC_OFF];
    d.row0 = dw[U_ROW0];
    d.n_rows = dw[U_N_ROWS];
    d.slot_base = dw[U_SLOT_BASE];
    d.kvh = dw[U_KVH];
    d.kind = dw[U_KIND];
    d.pos0 = dw[kUnitWords];
    return d;
}

// Fetcher warp: claim units, publish descriptor + tile words, stage query rows
// in the 128-byte-swizzle K-major layout the MMA reads. Rows past n_rows are
// left as they are: a row of A only reaches the same row of S, P and O, and
// those rows are never written out.
template <int HD>
__device__ void tc_fetch(const DecodeArgs& a, CtlTc& c, uint8_t* qbuf) {
    const int lane = threadIdx.x & 31;
    volatile int* abort = &c.abort;
    for (int k = 0;; ++k) {
        const int q = k & 1;
        if (!mbar_wait(smem_u32(&c.uempty[q]), ((k >> 1) & 1) ^ 1)) note_timeout(a, c, 2);
        int u = -1;
        if (lane == 0) {
            u = *abort ? -1 : a.unit_begin + atomicAdd(a.counter, 1);
            if (u >= a.unit_end) u = -1;
        }
        u = __shfl_sync(0xffffffffu, u, 0);
        const int word = (u >= 0 && lane < kUnitWords) ? a.units[(int64_t)u * kUnitWords + lane] : 0;
        const int n_tiles = __shfl_sync(0xffffffffu, word, U_N_TILES);
        const int tile_off = __shfl_sync(0xffffffffu, word, U_TILE_OFF);
        if constexpr (kBoundsCheck) {
            const int w_occ = __shfl_sync(0xffffffffu, word, U_OCC_OFF), w_row0 = __shfl_sync(0xffffffffu, word, U_ROW0);
            const int w_rows = __shfl_sync(0xffffffffu, word, U_N_ROWS);
            const int w_slot = __shfl_sync(0xffffffffu, word, U_SLOT_BASE), w_kvh = __shfl_sync(0xffffffffu, word, U_KVH);
            const int w_kind = __shfl_sync(0xffffffffu, word, U_KIND);
            if (u >= 0 && !(w_kind == KIND_TC && unit_ok(tile_off, n_tiles, w_occ, w_row0, w_rows, w_slot, w_kvh,
                                                         kTcRowsPerUnit, a.vis != nullptr, a.ext))) {
                if (lane == 0) atomicOr(a.err, kErrBounds);  // a bad unit record: this CTA takes no more units
                u = -1;
            }
        }
        if (u >= 0)
            for (int t = lane; t < n_tiles; t += 32) c.tiles[q][t] = a.tiles[tile_off + t];
        if (lane < kUnitWords) reinterpret_cast<volatile int*>(c.desc[q])[lane] = word;
        if (lane == kUnitWords)
            reinterpret_cast<volatile int*>(c.desc[q])[lane] = (u >= 0 && a.unit_pos) ? a.unit_pos[u] : 0;
        if (lane == 0) *reinterpret_cast<volatile int*>(&c.unit[q]) = u;
        __threadfence_block();
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&c.ufull[q]));
        if (u < 0) return;
        const int occ_off = __shfl_sync(0xffffffffu, word, U_OCC_OFF);
        const int row0 = __shfl_sync(0xffffffffu, word, U_ROW0);
        const int n_rows = __shfl_sync(0xffffffffu, word, U_N_ROWS);
        const int kvh = __shfl_sync(0xffffffffu, word, U_KVH);
        // the previous unit's Q.K^T MMAs have read the buffer
        if (!mbar_wait(smem_u32(&c.qempty), (k & 1) ^ 1)) note_timeout(a, c, 2);
        constexpr int CH = HD / 8;  // 16-byte chunks per row
        const int g = a.group;
        // lane = query row (rows lane, lane + 32, ...): its source row is
        // found once -- prefill schedules list query rows in order
        // (occurrence = query index), decode looks the occurrence up, all
        // lookups in flight together -- then its CH chunks go out as 16-byte
        // async copies straight into the swizzled layout, offsets known at
        // compile time, every copy of the tile in flight at once
        constexpr int kRowsPerLane = kTcRows / 32;
        const bool in_order = a.vis != nullptr;
        int64_t src_off[kRowsPerLane];
#pragma unroll
        for (int i = 0; i < kRowsPerLane; ++i) {
            const int r = lane + 32 * i;
            const int item_row = row0 + r, p = item_row / g, hh = item_row - p * g;
            int occ = r >= n_rows ? 0 : in_order ? occ_off + p : a.occ[occ_off + p];
            if (!check(in_range(occ, a.ext.n), a.err)) occ = 0;
            src_off[i] = ((int64_t)occ * a.hq + kvh * g + hh) * HD;
        }
        const uint32_t q_base = smem_u32(qbuf);
#pragma unroll
        for (int i = 0; i < kRowsPerLane; ++i) {
            const int r = lane + 32 * i;
            if (r >= n_rows) break;
            const uint16_t* src = a.q + src_off[i];
            const uint32_t dst = q_base + r * 128, x = r & 7;
#pragma unroll
            for (int ch = 0; ch < CH; ++ch)
                cp_async16(dst + (ch >> 3) * (kTcRows * 128) + (((ch & 7) ^ x) << 4), src + ch * 8);
        }
        cp_async_wait_all();
        fence_proxy_async();  // the copies -> visible to the tensor core
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&c.qfull));
    }
}

// Bulk copies of one half (K or V) of a tile pair into a stage; w = -1 for a
// missing second tile.
template <int HD>
__device__ __forceinline__ void issue_half(const DecodeArgs& a, int kvh, int kv, uint8_t* dst, const int32_t (&w)[2],
                                           uint32_t bar, bool once) {
    uint32_t bytes = 0;
    int valid[2] = {0, 0};
    for (int j = 0; j < 2; ++j)
        if (w[j] >= 0 && check(tile_word_ok(w[j], a.ext.pool_blocks), a.err)) {  // a bad word: a missing tile
            valid[j] = (w[j] & ((1 << kTileValidBits) - 1)) + 1;
            bytes += (uint32_t)(valid[j] * HD * 2);
        }
    mbar_arrive_expect_tx(bar, bytes);
    for (int j = 0; j < 2; ++j) {
        if (!valid[j]) continue;
        const uint8_t* src = a.pool + (int64_t)(w[j] >> kTileValidBits) * a.block_bytes +
                             (int64_t)(kv * a.hkv + kvh) * a.head_bytes;
#pragma unroll
        for (int h = 0; h < HD / 64; ++h) {
            const uint32_t d = smem_u32(dst + h * kStageTokens * 128 + j * kBlockTokens * 128);
            if (once)
                bulk_g2s_hint(d, src + h * kBlockTokens * 128, valid[j] * 128, bar, l2_evict_first());
            else
                bulk_g2s(d, src + h * kBlockTokens * 128, valid[j] * 128, bar);
        }
    }
}

// Streamer lane: K and V halves of each published unit's tile pairs, each
// half refilled as soon as its own slot frees (K is freed by Q.K^T, V only by
// P.V, so K runs ahead while V waits for the softmax).
template <int HD>
__device__ void tc_stream(const DecodeArgs& a, CtlTc& c, uint8_t* ring) {
    int ks = 0, vs = 0;
    uint32_t kph = 0, vph = 0;
    for (int k = 0;; ++k) {
        const int q = k & 1;
        if (!mbar_wait(smem_u32(&c.ufull[q]), (k >> 1) & 1)) {
            note_timeout(a, c, 2);
            return;
        }
        if (*reinterpret_cast<volatile int*>(&c.unit[q]) < 0) return;
        const int n_tiles = *reinterpret_cast<volatile int*>(&c.desc[q][U_N_TILES]);
        const int kvh = *reinterpret_cast<volatile int*>(&c.desc[q][U_KVH]);
        // the unit's rows are its item's only row block (fewer than a full
        // tile from row 0): no other unit reads this chunk
        const bool once = a.kv_read_once && *reinterpret_cast<volatile int*>(&c.desc[q][U_ROW0]) == 0 &&
                          *reinterpret_cast<volatile int*>(&c.desc[q][U_N_ROWS]) < kTcRows;
        const volatile int* tw = c.tiles[q];
        const int n_pairs = (n_tiles + 1) / 2;
        int kj = 0, vj = 0;
        uint64_t idle_since = 0;
        uint32_t spins = 0;
        while (vj < n_pairs) {
            bool progress = false;
            if (kj < n_pairs && mbar_test(smem_u32(&c.s_full[ks]), kph ^ 1)) {  // K slot read by Q.K^T
                const int32_t w[2] = {tw[2 * kj], 2 * kj + 1 < n_tiles ? tw[2 * kj + 1] : -1};
                fence_proxy_async();
                issue_half<HD>(a, kvh, 0, ring + ks * TcSmem<HD>::kStageBytes, w, smem_u32(&c.kfull[ks]), once);
                if (++ks == kStages) {
                    ks = 0;
                    kph ^= 1;
                }
                ++kj;
                progress = true;
            }
            if (vj < kj && mbar_test(smem_u32(&c.vempty[vs]), vph ^ 1)) {
                const int32_t w[2] = {tw[2 * vj], 2 * vj + 1 < n_tiles ? tw[2 * vj + 1] : -1};
                fence_proxy_async();
                issue_half<HD>(a, kvh, 1, ring + vs * TcSmem<HD>::kStageBytes + (HD / 64) * kStageTokens * 128, w,
                               smem_u32(&c.vfull[vs]), once);
                if (++vs == kStages) {
                    vs = 0;
                    vph ^= 1;
                }
                ++vj;
                progress = true;
            }
            if (progress) {
                spins = 0;
                idle_since = 0;
            } else if ((++spins & 1023) == 0) {
                const uint64_t now = global_ns();
                if (idle_since == 0) {
                    idle_since = now;
                } else if (now - idle_since > kWaitLimitNs) {
                    note_timeout(a, c, 2);
                    return;
                }
            }
        }
        mbar_arrive(smem_u32(&c.uempty[q]));
    }
}

// MMA issuer lane.
template <int HD>
__device__ void tc_issue(const DecodeArgs& a, CtlTc& c, const uint8_t* ring, const uint8_t* qbuf) {
    constexpr uint32_t kIdescS = mma_idesc<kStageTokens, false>();
    constexpr uint32_t kIdescPV = mma_idesc<HD, true>();
    const uint32_t tmem = c.tmem;
    const uint32_t q_addr = smem_u32(qbuf), ring_addr = smem_u32(ring);
    int s_stage = 0, v_stage = 0;
    uint32_t s_phase = 0, v_phase = 0;
    uint32_t gs = 0;  // stages issued by this CTA so far (S buffer = gs & 1)
    for (int k = 0;; ++k) {
        const int q = k & 1;
        if (!mbar_wait(smem_u32(&c.ufull[q]), (k >> 1) & 1)) {
            note_timeout(a, c, 2);
            return;
        }
        if (*reinterpret_cast<volatile int*>(&c.unit[q]) < 0) return;
        const int n_tiles = *reinterpret_cast<volatile int*>(&c.desc[q][U_N_TILES]);
        const int n_pairs = (n_tiles + 1) / 2;
        if (!mbar_wait(smem_u32(&c.qfull), k & 1)) note_timeout(a, c, 2);
        tc_fence_after();
        // Event loop: issue Q.K^T of the next stage as soon as its K/V has
        // landed (and its S buffer is free, i.e. P.V two stages back is
        // issued), and P.V of the oldest stage as soon as its P is written;
        // neither waits on the other.
        int next_s = 0, next_pv = 0;
        bool q_released = false;
        uint64_t idle_since = 0;
        uint32_t spins = 0;
        while (next_pv < n_pairs) {
            bool progress = false;
            if (next_s < n_pairs && next_s <= next_pv + 1 && mbar_test(smem_u32(&c.kfull[s_stage]), s_phase)) {
                tc_fence_after();
                const uint32_t g_stage = gs + next_s;
                const uint32_t kb = ring_addr + s_stage * TcSmem<HD>::kStageBytes;
                const uint32_t d = tmem + (g_stage & 1) * kStageTokens;
#pragma unroll
                for (int ks = 0; ks < HD / 16; ++ks) {
                    const uint32_t off = (ks >> 2) * (kStageTokens * 128) + (ks & 3) * 32;
                    const uint32_t qoff = (ks >> 2) * (kTcRows * 128) + (ks & 3) * 32;
                    mma_ss(d, smem_desc(q_addr + qoff, 16, 1024), smem_desc(kb + off, 16, 1024), kIdescS, ks > 0);
                }
                tc_commit(smem_u32(&c.s_full[g_stage & 1]));  // = ring slot s_stage
                if (++s_stage == kStages) {
                    s_stage = 0;
                    s_phase ^= 1;
                }
                ++next_s;
                progress = true;
            }
            if (next_s == n_pairs && !q_released) {
                tc_commit(smem_u32(&c.qempty));  // every Q.K^T of the unit issued
                q_released = true;
            }
            const uint32_t gp = gs + next_pv;
            if (next_pv < next_s && mbar_test(smem_u32(&c.p_full[gp & 1]), (gp >> 1) & 1) &&
                mbar_test(smem_u32(&c.vfull[v_stage]), v_phase)) {
                tc_fence_after();
                if (next_pv == 0) {  // the previous unit's epilogue has read O
                    if (!mbar_wait(smem_u32(&c.o_free), (k & 1) ^ 1)) note_timeout(a, c, 2);
                    tc_fence_after();
                }
                const uint32_t vb = ring_addr + v_stage * TcSmem<HD>::kStageBytes + (HD / 64) * kStageTokens * 128;
                const uint32_t p_tmem = tmem + (gp & 1) * kStageTokens;
#pragma unroll
                for (int kk = 0; kk < kStageTokens / 16; ++kk)
                    mma_ts(tmem + 2 * kStageTokens, p_tmem + kk * 8,
                           smem_desc(vb + kk * 2048, kStageTokens * 128, 1024), kIdescPV,
                           (next_pv > 0 || kk > 0) ? 1u : 0u);
                tc_commit(smem_u32(&c.vempty[v_stage]));
                if (next_pv + 1 == n_pairs) tc_commit(smem_u32(&c.o_full));
                if (++v_stage == kStages) {
                    v_stage = 0;
                    v_phase ^= 1;
                }
                ++next_pv;
                progress = true;
            }
            if (progress) {
                spins = 0;
                idle_since = 0;
            } else if ((++spins & 1023) == 0) {  // bounded: give up after the wait limit
                const uint64_t now = global_ns();
                if (idle_since == 0) {
                    idle_since = now;
                } else if (now - idle_since > kWaitLimitNs) {
                    note_timeout(a, c, 2);
                    return;
                }
            }
        }
        gs += n_pairs;
        mbar_arrive(smem_u32(&c.uempty[q]));
    }
}

// Softmax + epilogue warps: thread = query row (warp * 32 + lane). CAUSAL
// (prefill): the row sees only the first vis tokens of its path.
template <int HD, bool CAUSAL>
__device__ void tc_consume(const DecodeArgs& a, CtlTc& c) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int row = warp * 32 + lane;
    const uint32_t lane_addr = c.tmem + ((uint32_t)(warp * 32) << 16);
    const uint32_t o_addr = lane_addr + 2 * kStageTokens;
    uint32_t gs = 0;
    for (int k = 0;; ++k) {
        const int q = k & 1;
        if (!mbar_wait(smem_u32(&c.ufull[q]), (k >> 1) & 1)) {
            note_timeout(a, c, 8);
            return;
        }
        if (*reinterpret_cast<volatile int*>(&c.unit[q]) < 0) return;
        const UnitDesc d = read_desc(c.desc[q]);
        const volatile int* tw = c.tiles[q];
        const int n_pairs = (d.n_tiles + 1) / 2;
        float m_used = -INFINITY, l = 0.f;
        int vis = 0x7fffffff, pos = d.pos0;
        if (CAUSAL && row < d.n_rows) {
            const int occ = a.occ[d.occ_off + (d.row0 + row) / a.group];
            vis = check(in_range(occ, a.ext.n), a.err) ? a.vis[occ] : 0;
        }
        for (int j = 0; j < n_pairs; ++j) {
            const uint32_t g_stage = gs + j, sb = g_stage & 1;
            int v0 = (tw[2 * j] & ((1 << kTileValidBits) - 1)) + 1;
            int v1 = 2 * j + 1 < d.n_tiles ? (tw[2 * j + 1] & ((1 << kTileValidBits) - 1)) + 1 : 0;
            if (kBoundsCheck) {  // a tile the streamer refused holds no token
                if (!tile_word_ok(tw[2 * j], a.ext.pool_blocks)) v0 = 0;
                if (v1 && !tile_word_ok(tw[2 * j + 1], a.ext.pool_blocks)) v1 = 0;
            }
            // CAUSAL: tokens of tile h visible to this row: lim_h = min(valid, vis - position)
            int lim0 = v0, lim1 = v1;
            if (CAUSAL) {
                lim0 = max(0, min(v0, vis - pos));
                lim1 = max(0, min(v1, vis - (pos + v0)));
                pos += v0 + v1;
            }
            if (!mbar_wait(smem_u32(&c.s_full[sb]), (g_stage >> 1) & 1)) note_timeout(a, c, 1);
            tc_fence_after();
            if (warp * 32 >= d.n_rows) {  // padding rows only: their P is never read back
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_u32(&c.p_full[sb]));
                continue;
            }
            const uint32_t s_addr = lane_addr + sb * kStageTokens;
            // the stage's 64 scores of this row, read once (two loads in flight)
            uint32_t r[2][32];
            tmem_ld32_nowait(s_addr, r[0]);
            tmem_ld32_nowait(s_addr + 32, r[1]);
            tmem_wait_ld();
            // row max over the tokens the row may see, on the raw scores (the
            // scale is positive); a stage every row of the warp sees whole
            // takes the unmasked path
            const bool whole = __all_sync(0xffffffffu, lim0 == 32 && lim1 == 32);
            float mx = -INFINITY;
            if (whole) {  // four independent chains of three-input maxima
                float m0 = -INFINITY, m1 = -INFINITY, m2 = -INFINITY, m3 = -INFINITY;
#pragma unroll
                for (int t = 0; t < 32; t += 4) {
                    m0 = fmax3(m0, __uint_as_float(r[0][t]), __uint_as_float(r[0][t + 1]));
                    m1 = fmax3(m1, __uint_as_float(r[0][t + 2]), __uint_as_float(r[0][t + 3]));
                    m2 = fmax3(m2, __uint_as_float(r[1][t]), __uint_as_float(r[1][t + 1]));
                    m3 = fmax3(m3, __uint_as_float(r[1][t + 2]), __uint_as_float(r[1][t + 3]));
                }
                mx = fmaxf(fmax3(m0, m1, m2), m3);
            } else {
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int lim = h ? lim1 : lim0;
#pragma unroll
                    for (int t = 0; t < 32; ++t)
                        if (t < lim) mx = fmaxf(mx, __uint_as_float(r[h][t]));
                }
            }
            mx *= a.qk_scale_log2;
            const float m_new = fmaxf(m_used, mx);
            const bool need = m_new > m_used + kRescaleLog2;
            if (__any_sync(0xffffffffu, need)) {
                const float alpha = need ? fast_exp2(m_used - m_new) : 1.f;
                if (j > 0) {  // O holds earlier stages: wait for the last P.V, then scale it
                    const uint32_t prev = g_stage - 1;  // its P.V used ring slot prev & 1
                    if (!mbar_wait(smem_u32(&c.vempty[prev & 1]), (prev >> 1) & 1)) note_timeout(a, c, 1);
                    tc_fence_after();
#pragma unroll 1
                    for (int cc = 0; cc < HD / 32; ++cc) {
                        uint32_t ov[32];
                        tmem_ld32(o_addr + cc * 32, ov);
#pragma unroll
                        for (int t = 0; t < 32; ++t) ov[t] = __float_as_uint(__uint_as_float(ov[t]) * alpha);
                        tmem_st32(o_addr + cc * 32, ov);
                    }
                }
                if (need) {
                    l *= alpha;
                    m_used = m_new;
                }
            }
            // P = exp2(s * scale - m_used) as bf16 pairs over the S columns
            uint32_t pw[32];
            float sum = 0.f;
            const float sc = a.qk_scale_log2, neg_m = -m_used;
            if (whole) {  // scale and shift two scores per instruction; two pair sums
                const uint64_t sc2 = f2_pack(sc, sc), nm2 = f2_pack(neg_m, neg_m);
                uint64_t acc[2] = {0, 0};
#pragma unroll
                for (int h = 0; h < 2; ++h)
#pragma unroll
                    for (int t = 0; t < 32; t += 2) {
                        float x0, x1;
                        f2_unpack(f2_fma(f2_pack(__uint_as_float(r[h][t]), __uint_as_float(r[h][t + 1])), sc2, nm2),
                                  x0, x1);
                        const float p0 = fast_exp2(x0), p1 = fast_exp2(x1);
                        acc[(t >> 1) & 1] = f2_add(acc[(t >> 1) & 1], f2_pack(p0, p1));
                        pw[h * 16 + t / 2] = pack_bf16(p0, p1);
                    }
                float s0, s1, s2, s3;
                f2_unpack(acc[0], s0, s1);
                f2_unpack(acc[1], s2, s3);
                sum = (s0 + s2) + (s1 + s3);
            } else {
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int lim = h ? lim1 : lim0;
#pragma unroll
                    for (int t = 0; t < 32; t += 2) {
                        const float p0 = t < lim ? fast_exp2(fmaf(__uint_as_float(r[h][t]), sc, neg_m)) : 0.f;
                        const float p1 = t + 1 < lim ? fast_exp2(fmaf(__uint_as_float(r[h][t + 1]), sc, neg_m)) : 0.f;
                        sum += p0 + p1;
                        pw[h * 16 + t / 2] = pack_bf16(p0, p1);
                    }
                }
            }
            l += sum;
            tmem_st32(s_addr, pw);
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&c.p_full[sb]));
        }
        gs += n_pairs;
        // epilogue: O / l and the log2 LSE of this row
        if (!mbar_wait(smem_u32(&c.o_full), k & 1)) note_timeout(a, c, 1);
        tc_fence_after();
        if (warp * 32 >= d.n_rows) {  // padding rows only
            __syncwarp();
            if (lane == 0) {
                mbar_arrive(smem_u32(&c.o_free));
                mbar_arrive(smem_u32(&c.uempty[q]));
            }
            continue;
        }
        bool live = row < d.n_rows;
        const bool final_out = CAUSAL && d.slot_base < 0;  // the row's only unit: final O and LSE
        float* dst = nullptr;
        uint16_t* dst16 = nullptr;
        if (live) {
            const int item_row = d.row0 + row;
            const int qh = d.kvh * a.group + item_row % a.group;
            if (final_out) {
                const int occ = a.occ[d.occ_off + item_row / a.group];
                live = check(in_range(occ, a.ext.n), a.err);
                dst16 = a.out + ((int64_t)occ * a.hq + qh) * HD;
                if (live) a.out_lse[(int64_t)occ * a.hq + qh] = (m_used + __log2f(l)) * 0.69314718055994531f;
            } else {
                const int slot = d.slot_base + item_row / a.group;
                dst = a.part_o + ((int64_t)slot * a.hq + qh) * HD;
                a.part_lse[(int64_t)slot * a.hq + qh] = m_used + __log2f(l);
            }
        }
        const float inv = 1.f / l;
        const uint64_t pol = l2_evict_last();
        // 32-byte stores (a full sector per lane) where the rows allow them:
        // the partial buffer always, the caller's O when its base is 32-byte
        // aligned (rows are multiples of 256 bytes, so the base decides)
        const bool wide = !final_out || (reinterpret_cast<uintptr_t>(a.out) & 31) == 0;
#pragma unroll 1
        for (int cc = 0; cc < HD / 32; cc += 2) {  // two 32-column loads in flight
            uint32_t ov[2][32];
            __syncwarp();  // the loads are warp-collective
            tmem_ld32_nowait(o_addr + cc * 32, ov[0]);
            tmem_ld32_nowait(o_addr + cc * 32 + 32, ov[1]);
            tmem_wait_ld();
#pragma unroll
            for (int h = 0; h < 2 && live; ++h) {
                const int c0 = (cc + h) * 32;
                if (final_out) {
                    uint32_t w[16];
#pragma unroll
                    for (int t = 0; t < 16; ++t)
                        w[t] = pack_bf16(__uint_as_float(ov[h][2 * t]) * inv, __uint_as_float(ov[h][2 * t + 1]) * inv);
                    if (wide) {
                        st_global_v8(dst16 + c0, w);
                        st_global_v8(dst16 + c0 + 16, w + 8);
                    } else {
#pragma unroll
                        for (int t = 0; t < 16; t += 4)
                            *reinterpret_cast<uint4*>(dst16 + c0 + 2 * t) = make_uint4(w[t], w[t + 1], w[t + 2], w[t + 3]);
                    }
                } else {
#pragma unroll
                    for (int t = 0; t < 32; t += 8) {
                        uint32_t w[8];
#pragma unroll
                        for (int e = 0; e < 8; ++e) w[e] = __float_as_uint(__uint_as_float(ov[h][t + e]) * inv);
                        st_global_v8_hint(dst + c0 + t, w, pol);
                    }
                }
            }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
            mbar_arrive(smem_u32(&c.o_free));
            mbar_arrive(smem_u32(&c.uempty[q]));
        }
    }
}

template <int HD, bool CAUSAL>
__global__ void __launch_bounds__(kTcThreads, 2) decode_tc_kernel(const DecodeArgs a) {
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    __shared__ __align__(16) CtlTc ctl;
    // 128-byte-swizzle operands need 1024-byte-aligned atoms
    uint8_t* base = smem_raw + ((1024 - (smem_u32(smem_raw) & 1023)) & 1023);
    uint8_t* ring = base;
    uint8_t* qbuf = base + TcSmem<HD>::kRingBytes;
    const int tid = threadIdx.x, warp = tid >> 5;
    {
        uint4* r4 = reinterpret_cast<uint4*>(ring);  // rows past a partial block must be finite
        for (int i = tid; i < TcSmem<HD>::kRingBytes / 16; i += kTcThreads) r4[i] = make_uint4(0, 0, 0, 0);
    }
    if (tid == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(smem_u32(&ctl.kfull[s]), 1);
            mbar_init(smem_u32(&ctl.vfull[s]), 1);
            mbar_init(smem_u32(&ctl.vempty[s]), 1);
        }
        for (int q = 0; q < 2; ++q) {
            mbar_init(smem_u32(&ctl.ufull[q]), 1);
            mbar_init(smem_u32(&ctl.uempty[q]), kTcConsumerWarps + 2);  // consumers + streamer + issuer
            mbar_init(smem_u32(&ctl.s_full[q]), 1);
            mbar_init(smem_u32(&ctl.p_full[q]), kTcConsumerWarps);
        }
        mbar_init(smem_u32(&ctl.qfull), 1);
        mbar_init(smem_u32(&ctl.qempty), 1);
        mbar_init(smem_u32(&ctl.o_full), 1);
        mbar_init(smem_u32(&ctl.o_free), kTcConsumerWarps);
        ctl.abort = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&ctl.tmem)),
                     "r"(kTmemCols));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
    fence_proxy_async();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp < kTcConsumerWarps)
        tc_consume<HD, CAUSAL>(a, ctl);
    else if (warp == kTcStreamerWarp) {
        if ((tid & 31) == 0) tc_stream<HD>(a, ctl, ring);
    } else if (warp == kTcFetcherWarp) {
        tc_fetch<HD>(a, ctl, qbuf);
    } else if (warp == kTcIssuerWarp) {
        if ((tid & 31) == 0) tc_issue<HD>(a, ctl, ring, qbuf);
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(ctl.tmem), "r"(kTmemCols));
}

// ------------------------------------------------------------------- merge --
// Fold up to four partial rows (j0 .. j0 + 3 of a chunk of at most 32 slots,
// rows past cnt masked) into acc; slot and w are the lanes' slot indices and
// weights (lane k: row k of the chunk). Each row's 128-byte L2 lines are
// dropped afterwards (a partial row is read by this warp only).
template <int HD>
__device__ __forceinline__ void merge_batch(const MergeArgs& a, int qh, int lane, int slot, float w, int j0, int cnt,
                                            uint64_t pol, float (&acc)[HD / 32]) {
    constexpr int DPL = HD / 32;
    constexpr int kLanesPerLine = 128 / (DPL * 4);
    float wj[4];
    float x[4][DPL];
    const float* srcs[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
        const bool on = j0 + u < cnt;
        const int64_t sl = __shfl_sync(0xffffffffu, slot, on ? j0 + u : j0);  // off: re-read row j0, weight 0
        wj[u] = __shfl_sync(0xffffffffu, w, on ? j0 + u : j0) * (on ? 1.f : 0.f);
        const float* src = a.part_o + (sl * a.hq + qh) * HD + lane * DPL;
        srcs[u] = on ? src : nullptr;
        if constexpr (DPL == 4) {
            const float4 v = ld_f4_hint(src, pol);
            x[u][0] = v.x, x[u][1] = v.y, x[u][2] = v.z, x[u][3] = v.w;
        } else {
            const float2 v = ld_f2_hint(src, pol);
            x[u][0] = v.x, x[u][1] = v.y;
        }
    }
#pragma unroll
    for (int u = 0; u < 4; ++u)
#pragma unroll
        for (int d = 0; d < DPL; ++d) acc[d] += wj[u] * x[u][d];
    __syncwarp();
    if ((lane & (kLanesPerLine - 1)) == 0)
#pragma unroll
        for (int u = 0; u < 4; ++u)
            if (srcs[u]) l2_discard(srcs[u]);
}

template <int HD>
__global__ void __launch_bounds__(128) merge_kernel(const MergeArgs a) {
    constexpr int DPL = HD / 32;  // dims per lane: 4 or 2
    const int warp_global = blockIdx.x * 4 + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (blockIdx.x == 0 && threadIdx.x < 3) a.counters[threadIdx.x] = 0;  // decode is done: re-arm its counters
    if (warp_global >= a.n * a.hq) return;
    const int i = warp_global / a.hq, qh = warp_global % a.hq;
    float acc[DPL];
#pragma unroll
    for (int d = 0; d < DPL; ++d) acc[d] = 0.f;
    float M = -INFINITY, L = 0.f;
    const uint64_t pol = l2_evict_first();  // each partial row is read once
    // The occurrence's merge record, in one round trip: lane k < 16 holds
    // word k ([count, slots...]).
    const int rw = a.merge_rec && lane < kMergeRecWords ? a.merge_rec[(int64_t)i * kMergeRecWords + lane] : -1;
    const int ns_rec = __shfl_sync(0xffffffffu, rw, 0);  // -1: the CSR (more than 15 slots, or no records)
    if (ns_rec >= 0) {
        // up to 15 slots: lane k takes slot k; its LSE and the first four
        // partial rows are loaded together, then folded
        const int ns = ns_rec;
        if (!check(ns < kMergeRecWords, a.err) || ns == 0) return;  // 0: written directly by its only unit
        int slot = __shfl_sync(0xffffffffu, rw, (lane + 1) & 31);  // every lane shuffles
        const int first = __shfl_sync(0xffffffffu, rw, 1);
        if (lane >= ns)
            slot = first;  // a valid row (weight 0)
        else if (!check(in_range(slot, a.n_slots), a.err))
            slot = 0;
        float x0[4][DPL];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int64_t sl = __shfl_sync(0xffffffffu, slot, u < ns ? u : 0);
            const float* src = a.part_o + (sl * a.hq + qh) * HD + lane * DPL;
            if constexpr (DPL == 4) {
                const float4 v = ld_f4_hint(src, pol);
                x0[u][0] = v.x, x0[u][1] = v.y, x0[u][2] = v.z, x0[u][3] = v.w;
            } else {
                const float2 v = ld_f2_hint(src, pol);
                x0[u][0] = v.x, x0[u][1] = v.y;
            }
        }
        const float lse = lane < ns ? a.part_lse[(int64_t)slot * a.hq + qh] : -INFINITY;
        M = lse;
#pragma unroll
        for (int off = 16; off; off >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, off));
        const float w = lane < ns ? fast_exp2(lse - M) : 0.f;
        L = w;
#pragma unroll
        for (int off = 16; off; off >>= 1) L += __shfl_xor_sync(0xffffffffu, L, off);
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const float wu = __shfl_sync(0xffffffffu, w, u) * (u < ns ? 1.f : 0.f);
#pragma unroll
            for (int d = 0; d < DPL; ++d) acc[d] += wu * x0[u][d];
        }
        {
            constexpr int kLanesPerLine = 128 / (DPL * 4);
            __syncwarp();
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int64_t sl = __shfl_sync(0xffffffffu, slot, u < ns ? u : 0);  // every lane shuffles
                if (u < ns && (lane & (kLanesPerLine - 1)) == 0) l2_discard(a.part_o + (sl * a.hq + qh) * HD + lane * DPL);
            }
        }
        for (int j = 4; j < ns; j += 4) merge_batch<HD>(a, qh, lane, slot, w, j, ns, pol, acc);
    } else {
        // more slots: the CSR, in chunks of 32 -- lane k fetches slot k's
        // index and LSE, then the warp folds the chunk's partial rows, four
        // loads in flight per lane
        const int beg = a.merge_off[i], ns = a.merge_off[i + 1] - beg;
        if (!check(merge_range_ok(beg, beg + ns, a.n_merge) && (ns == 0 || a.n_slots > 0), a.err)) return;
        if (ns == 0) return;
        for (int c0 = 0; c0 < ns; c0 += 32) {
            const int k = c0 + lane;
            int slot = 0;
            float lse = -INFINITY;
            if (k < ns) {
                slot = a.merge_slot[beg + k];
                if (check(in_range(slot, a.n_slots), a.err))
                    lse = a.part_lse[(int64_t)slot * a.hq + qh];
                else
                    slot = 0;  // weight 0, a valid row to read
            }
            float cm = lse;
#pragma unroll
            for (int off = 16; off; off >>= 1) cm = fmaxf(cm, __shfl_xor_sync(0xffffffffu, cm, off));
            const float m_new = fmaxf(M, cm);
            const float keep = (M == -INFINITY) ? 0.f : fast_exp2(M - m_new);
#pragma unroll
            for (int d = 0; d < DPL; ++d) acc[d] *= keep;
            L *= keep;
            M = m_new;
            const float w = (k < ns) ? fast_exp2(lse - M) : 0.f;
            float ws = w;
#pragma unroll
            for (int off = 16; off; off >>= 1) ws += __shfl_xor_sync(0xffffffffu, ws, off);
            L += ws;
            const int cnt = min(32, ns - c0);
            for (int j = 0; j < cnt; j += 4) merge_batch<HD>(a, qh, lane, slot, w, j, cnt, pol, acc);
        }
    }
    const float inv = 1.f / L;
    uint16_t* dst = a.out + ((int64_t)i * a.hq + qh) * HD + lane * DPL;
    if constexpr (DPL == 4) {
        const uint32_t lo = pack_bf16(acc[0] * inv, acc[1] * inv), hi = pack_bf16(acc[2] * inv, acc[3] * inv);
        *reinterpret_cast<uint2*>(dst) = make_uint2(lo, hi);
    } else {
        *reinterpret_cast<uint32_t*>(dst) = pack_bf16(acc[0] * inv, acc[1] * inv);
    }
    if (lane == 0) a.lse[(int64_t)i * a.hq + qh] = (M + __log2f(L)) * 0.69314718055994531f;
}

template <int HD, int KIND>
int decode_grid() {
    // persistent grid: every resident CTA slot of the device
    static int grid = [] {
        int dev = 0, sms = 0, per_sm = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        if (cudaFuncSetAttribute(decode_kernel<HD, KIND>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 decode_smem<HD, KIND>()) != cudaSuccess)
            return 0;
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, decode_kernel<HD, KIND>, kDecodeThreads,
                                                          decode_smem<HD, KIND>()) != cudaSuccess)
            return 0;
        return sms * std::max(per_sm, 1);
    }();
    return grid;
}

template <int HD, int KIND>
cudaError_t launch_range(DecodeArgs a, int begin, int end, int32_t* counter, cudaStream_t s) {
    if (end <= begin) return cudaSuccess;
    const int slots = decode_grid<HD, KIND>();
    if (slots == 0) return cudaErrorInvalidConfiguration;
    a.unit_begin = begin;
    a.unit_end = end;
    a.counter = counter;
    decode_kernel<HD, KIND><<<std::min(end - begin, slots), kDecodeThreads, decode_smem<HD, KIND>(), s>>>(a);
    return cudaGetLastError();
}

template <int HD, bool CAUSAL>
int decode_tc_grid() {
    static int grid = [] {
        int dev = 0, sms = 0, per_sm = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        if (cudaFuncSetAttribute(decode_tc_kernel<HD, CAUSAL>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 TcSmem<HD>::kBytes) != cudaSuccess)
            return 0;
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, decode_tc_kernel<HD, CAUSAL>, kTcThreads,
                                                          TcSmem<HD>::kBytes) != cudaSuccess)
            return 0;
        // The occupancy query answers 1 for this kernel on GB300 although its
        // registers (128 x 224 threads) and shared memory fit twice per SM, so
        // count from those resources too. Launching more CTAs than fit is
        // harmless for a persistent kernel: a CTA that starts late finds the
        // unit counter exhausted and exits.
        cudaFuncAttributes fa{};
        int smem_sm = 0, reserved = 0;
        if (cudaFuncGetAttributes(&fa, decode_tc_kernel<HD, CAUSAL>) != cudaSuccess) return 0;
        cudaDeviceGetAttribute(&smem_sm, cudaDevAttrMaxSharedMemoryPerMultiprocessor, dev);
        cudaDeviceGetAttribute(&reserved, cudaDevAttrReservedSharedMemoryPerBlock, dev);
        const int by_smem = smem_sm / (int)(TcSmem<HD>::kBytes + fa.sharedSizeBytes + reserved);
        const int by_regs = 65536 / (fa.numRegs * kTcThreads);
        per_sm = std::max(per_sm, std::min(by_smem, by_regs));
        // each resident CTA holds kTmemCols of the SM's 512 tensor-memory columns
        return sms * std::min(std::max(per_sm, 1), 512 / (int)kTmemCols);
    }();
    return grid;
}

template <int HD>
cudaError_t launch_tc_range(DecodeArgs a, int begin, int end, int32_t* counter, cudaStream_t s) {
    if (end <= begin) return cudaSuccess;
    const bool causal = a.vis != nullptr;
    const int slots = causal ? decode_tc_grid<HD, true>() : decode_tc_grid<HD, false>();
    if (slots == 0) return cudaErrorInvalidConfiguration;
    a.unit_begin = begin;
    a.unit_end = end;
    a.counter = counter;
    if (causal)
        decode_tc_kernel<HD, true><<<std::min(end - begin, slots), kTcThreads, TcSmem<HD>::kBytes, s>>>(a);
    else
        decode_tc_kernel<HD, false><<<std::min(end - begin, slots), kTcThreads, TcSmem<HD>::kBytes, s>>>(a);
    return cudaGetLastError();
}

template <int HD>
cudaError_t launch_decode_hd(const DecodeArgs& a, cudaStream_t s, cudaStream_t side, cudaEvent_t fork,
                             cudaEvent_t join) {
    const int tc_end = a.n_tc_units, mma_end = tc_end + a.n_tensor_units;
    cudaError_t e;
    const bool concurrent = side && fork && join && tc_end > 0 && a.n_units > tc_end;
    if (concurrent) {
        if ((e = cudaEventRecord(fork, s)) != cudaSuccess) return e;
        if ((e = cudaStreamWaitEvent(side, fork, 0)) != cudaSuccess) return e;
        if ((e = launch_tc_range<HD>(a, 0, tc_end, a.counters, side)) != cudaSuccess) return e;
        if ((e = cudaEventRecord(join, side)) != cudaSuccess) return e;
    } else {
        e = launch_tc_range<HD>(a, 0, tc_end, a.counters, s);
    }
    if (e != cudaSuccess) return e;
    e = a.vis ? launch_range<HD, KIND_PREFILL>(a, tc_end, mma_end, a.counters + 1, s)
              : launch_range<HD, KIND_TENSOR>(a, tc_end, mma_end, a.counters + 1, s);
    if (e != cudaSuccess) return e;
    e = launch_range<HD, KIND_CUDA_CORE>(a, mma_end, a.n_units, a.counters + 2, s);
    if (e != cudaSuccess) return e;
    return concurrent ? cudaStreamWaitEvent(s, join, 0) : cudaSuccess;
}

}  // namespace

int decode_smem_bytes(int head_dim) { return head_dim == 64 ? Smem<64>::kBytes : Smem<128>::kBytes; }

// ------------------------------------------------------- static scratch --
// Scratch of tp_decode_noalloc (schedule words, then fp32 partials): a
// file-scope device array, so that entry point never allocates. Device code
// could name it directly; host code only sees a host-side stand-in for it,
// so the launchers take the device address that cudaGetSymbolAddress gives,
// looked up once per device with that device current.
static __device__ __align__(256) uint8_t g_noalloc_scratch[TP_NOALLOC_SCRATCH_BYTES];

cudaError_t noalloc_scratch(void** device_ptr) {
    constexpr int kMaxDevices = 64;
    static void* addr[kMaxDevices] = {};
    static std::mutex lock;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> g(lock);
    if (!addr[dev]) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess) return e;
        addr[dev] = p;
    }
    *device_ptr = addr[dev];
    return cudaSuccess;
}

// Failure-reporting probe: the attention kernels' bounded wait, on a barrier
// nothing ever completes and with a short limit; when it runs out the kernel
// sets its bit of the device error flag and returns, as they do.
__global__ void wait_probe_kernel(int32_t* err, uint64_t limit_ns) {
    __shared__ uint64_t bar;
    if (threadIdx.x == 0) {
        mbar_init(smem_u32(&bar), 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();
    if (threadIdx.x == 0 && !mbar_wait(smem_u32(&bar), 0, limit_ns)) atomicOr(err, 32);
}

cudaError_t launch_wait_probe(int32_t* err, uint64_t limit_ns, cudaStream_t s) {
    wait_probe_kernel<<<1, 32, 0, s>>>(err, limit_ns);
    return cudaGetLastError();
}

cudaError_t launch_patch(int32_t* sched, const int32_t* pairs, int32_t n, cudaStream_t s, int64_t sched_words,
                         int32_t* err) {
    patch_kernel<<<(n + 255) / 256, 256, 0, s>>>(sched, pairs, n, sched_words, err);
    return cudaGetLastError();
}

cudaError_t launch_append_tokens(int hd, const AppendTokensArgs& a, cudaStream_t s) {
    const int64_t chunks = 2ll * a.n * a.hkv * (hd / 8);
    const int grid = (int)std::max<int64_t>(1, std::min<int64_t>((chunks + 255) / 256, 152 * 16));
    if (hd == 64)
        append_tokens_kernel<64><<<grid, 256, 0, s>>>(a);
    else
        append_tokens_kernel<128><<<grid, 256, 0, s>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_rollout_step(int hd, const StepArgs& a, cudaStream_t s) {
    const int64_t items = (int64_t)a.n * (2 * a.hkv * (hd / 8) + a.q_width / 4) + a.n_pairs;
    if (items == 0) return cudaSuccess;
    const int grid = (int)std::max<int64_t>(1, std::min<int64_t>((items + 255) / 256, 152 * 16));
    if (hd == 64)
        rollout_step_kernel<64><<<grid, 256, 0, s>>>(a);
    else
        rollout_step_kernel<128><<<grid, 256, 0, s>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_synth(const SynthArgs& a, cudaStream_t s) {
    const int64_t words =
        a.rows * ((a.k ? a.kv_width / 4 : 0) + (a.v ? a.kv_width / 4 : 0) + (a.q ? a.q_width / 4 : 0));
    if (words == 0) return cudaSuccess;
    const int grid = (int)std::max<int64_t>(1, std::min<int64_t>((words + 255) / 256, 152 * 16));
    synth_kernel<<<grid, 256, 0, s>>>(a);
    return cudaGetLastError();
}

int64_t advantage_ws_bytes(int64_t n_nodes, int64_t n_out) {
    return adv_tail_offset(n_nodes, n_out) + 2 * 8 + 2 * 4;
}

cudaError_t launch_advantage(const AdvantageArgs& a, cudaStream_t s) {
    const int init_grid = (int)std::min<int64_t>(std::max<int64_t>(1, (a.n_nodes + kAdvThreads - 1) / kAdvThreads),
                                                 152 * 8);
    advantage_init_kernel<<<init_grid, kAdvThreads, 0, s>>>(a);
    const int out_grid = (int)std::max<int64_t>(1, ((int64_t)a.n_out + kAdvWalkThreads - 1) / kAdvWalkThreads);
    if (a.n_out > 0) {
        advantage_walk_kernel<<<out_grid, kAdvWalkThreads, 0, s>>>(a);
        advantage_means_kernel<<<init_grid, kAdvThreads, 0, s>>>(a);
    }
    const int abar_grid = (int)std::max<int64_t>(1, ((int64_t)a.n_out + kAdvAbarThreads - 1) / kAdvAbarThreads);
    advantage_abar_kernel<<<abar_grid, kAdvAbarThreads, 0, s>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_append(int hd, const AppendArgs& a, cudaStream_t s) {
    const int64_t chunks = 2ll * a.n_tokens * a.hkv * (hd / 8);
    const int grid = (int)std::min<int64_t>((chunks + 255) / 256, 152 * 16);
    if (hd == 64)
        append_kernel<64><<<grid, 256, 0, s>>>(a);
    else
        append_kernel<128><<<grid, 256, 0, s>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_gather(int hd, const GatherArgs& a, int64_t n_tokens, cudaStream_t s) {
    const int64_t chunks = 2ll * n_tokens * a.hkv * (hd / 8);
    const int grid = (int)std::min<int64_t>((chunks + 255) / 256, 152 * 16);
    if (hd == 64)
        gather_kernel<64><<<grid, 256, 0, s>>>(a, n_tokens);
    else
        gather_kernel<128><<<grid, 256, 0, s>>>(a, n_tokens);
    return cudaGetLastError();
}

cudaError_t launch_decode(int hd, const DecodeArgs& a, cudaStream_t s, cudaStream_t side, cudaEvent_t fork,
                          cudaEvent_t join) {
    if (a.n_units == 0) return cudaSuccess;
    return hd == 64 ? launch_decode_hd<64>(a, s, side, fork, join) : launch_decode_hd<128>(a, s, side, fork, join);
}

cudaError_t launch_merge(int hd, const MergeArgs& a, cudaStream_t s) {
    const int64_t warps = (int64_t)a.n * a.hq;
    const int grid = (int)std::max<int64_t>(1, (warps + 3) / 4);  // one block at least: it re-arms the counters
    if (hd == 64)
        merge_kernel<64><<<grid, 128, 0, s>>>(a);
    else
        merge_kernel<128><<<grid, 128, 0, s>>>(a);
    return cudaGetLastError();
}

}  // namespace tp
