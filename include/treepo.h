/*
 * treepo.h -- C ABI of libtreepo: decode attention over a segment tree of
 * KV caches on one GB300 (sm_103a).
 *
 * TreePO samples each prompt as a tree (Sec. 2.2, Algorithm 1): the prompt is
 * the root at depth 0, each inference step appends a segment of at most l
 * tokens to every live path, branching forks a path into b copies, and early
 * stop drops a path. A trajectory is the concatenation s_1 (+) ... (+) s_j of
 * the segments on its root-to-leaf path (Sec. 2.3). Sibling branches share
 * their prefix, which this library stores once (Sec. 2.1: shared prefixes
 * represented only once; Sec. 1: paths with separate KV caches fail to share)
 * and reads from HBM once per decode call, not once per branch.
 *
 * Objects. One tp_tree owns a paged KV pool and a forest of trees (one root
 * per prompt). Nodes are dense int32 ids handed out in creation order and
 * never reused while the tp_tree lives. A node is a live leaf, a frozen
 * interior node (it has been forked), or dead (pruned).
 *
 * Pool. pool_blocks blocks of block_tokens token slots; a block holds K and V
 * of every kv head for its tokens. An append first fills the node's partly
 * used last block, then takes new blocks, lowest free index first. Forks move
 * no bytes: children start empty and read the parent's blocks through the
 * tree. Token t of a node sits in slot  block[t / block_tokens] * block_tokens
 * + t % block_tokens.
 *
 * Threading and streams. Calls on one tp_tree must not run concurrently. Host
 * work (validation, tree updates, scheduling) is synchronous; device work is
 * enqueued on the tree's stream and is asynchronous to the host.
 *
 * Errors. Every call returns a tp_status; on failure nothing in the tree
 * changes and tp_last_error() describes the failure. Kernels never trap: a
 * bounded wait that runs out sets a device flag that tp_sync() reports as
 * TP_ERR_DEVICE.
 *
 * Bounds-checked build. libtreepo_checked.so (build.py builds it beside
 * libtreepo.so, compiled with TP_BOUNDS_CHECK) exports the same calls; its
 * kernels check every index they take from a schedule or a slot list
 * before the access (see tp_debug_check_schedule) and, on a failed check,
 * skip the access and set a device flag that tp_sync() reports as
 * TP_ERR_DEVICE. It is a debugging aid: on valid input it computes the same
 * results as libtreepo.so, a little slower.
 *
 * Pointer conventions. "device" = CUDA device memory (any allocator); "host"
 * = ordinary host memory. The caller owns every buffer it passes; the library
 * keeps no pointer to a caller buffer after a call returns, except the pool
 * arena, which must outlive the tp_tree.
 */
#ifndef TREEPO_H_
#define TREEPO_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef int32_t tp_status;
#define TP_OK 0
#define TP_ERR_INVALID_ARG (-1) /* bad size, null or misaligned pointer, bad config */
#define TP_ERR_OOM (-2)         /* pool (or library scratch) exhausted            */
#define TP_ERR_BAD_NODE (-3)    /* unknown or pruned node id                       */
#define TP_ERR_FROZEN (-4)      /* append to a node that has been forked           */
#define TP_ERR_NOT_LEAF (-5)    /* decode/prune of an interior node                */
#define TP_ERR_EMPTY_PATH (-6)  /* decode of a leaf whose path holds no token      */
#define TP_ERR_CUDA (-7)        /* a CUDA runtime call failed                      */
#define TP_ERR_DEVICE (-8)      /* a kernel's bounded wait ran out, or (bounds-    */
                                /* checked build) an index failed its check        */

typedef int32_t tp_node;
typedef struct tp_tree tp_tree;

/*
 * Tree configuration.
 *   num_q_heads, num_kv_heads: num_q_heads % num_kv_heads == 0; q-head h reads
 *       kv head h / (num_q_heads / num_kv_heads) (contiguous GQA groups).
 *   head_dim: 64 or 128.
 *   block_tokens: tokens per pool block; 32.
 *   pool_blocks: 1 .. 2^24 blocks.
 *   pool: device arena of tp_pool_bytes(cfg) bytes, 256-byte aligned, owned
 *       by the caller and alive as long as the tree; its contents are the
 *       library's. NULL makes a metadata-only tree: every host operation
 *       works (append then takes K = V = NULL and copies nothing), device
 *       operations return TP_ERR_INVALID_ARG. Used to test the host logic
 *       without a GPU.
 *   cuda_stream: cudaStream_t for all device work; NULL = legacy default.
 */
typedef struct {
    int32_t num_q_heads;
    int32_t num_kv_heads;
    int32_t head_dim;
    int32_t block_tokens;
    int64_t pool_blocks;
    void* pool;
    void* cuda_stream;
} tp_config;

/* Bytes the pool arena must hold: pool_blocks * 2 * num_kv_heads *
 * block_tokens * head_dim * 2 (bf16 K and V). The pool is the KV cache of
 * every segment of the forest, each stored once (Sec. 2.1). Returns -1 on a
 * bad config. */
int64_t tp_pool_bytes(const tp_config* cfg);

/* Create an empty forest over cfg's pool: the batch of prompt trees one
 * rollout grows (Sec. 2.2, Algorithm 1 samples every query of a batch as a
 * tree; Sec. 2.1, their shared prefixes live once in one paged pool).
 * *out receives the handle. Errors: TP_ERR_INVALID_ARG (bad config),
 * TP_ERR_OOM / TP_ERR_CUDA (library scratch). */
tp_status tp_tree_create(const tp_config* cfg, tp_tree** out);

/* Destroy the forest at the end of a rollout (Sec. 2.2: the batch's trees
 * are done once every path has stopped); waits for its device work first
 * and frees the library's scratch, not the caller's pool arena. NULL is a
 * no-op. */
tp_status tp_tree_destroy(tp_tree* tree);

/* Use another stream for subsequent device work (cudaStream_t; NULL =
 * default). Plumbing with no counterpart in the paper. */
tp_status tp_set_stream(tp_tree* tree, void* cuda_stream);

/* New tree: an empty root node (a prompt at depth 0, Sec. 2.2). */
tp_status tp_add_root(tp_tree* tree, tp_node* out_root);

/*
 * Append n_tokens tokens to live leaf `node` (a prompt, or a generated
 * segment s_j: Algorithm 1 concatenates p (+) s). K and V are device bf16
 * [n_tokens][num_kv_heads][head_dim], 16-byte aligned, already position
 * encoded; they are copied into pool blocks on the tree's stream (the caller
 * may reuse them once that stream passes this point). n_tokens == 0 is a
 * no-op. Errors: TP_ERR_BAD_NODE, TP_ERR_FROZEN (node was forked),
 * TP_ERR_OOM (not enough free blocks; nothing is allocated),
 * TP_ERR_INVALID_ARG.
 */
tp_status tp_append_segment(tp_tree* tree, tp_node node, int32_t n_tokens, const void* K,
                            const void* V);

/*
 * Fork `node` into k >= 1 new empty children (branching, Sec. 2.2: a prompt
 * forked b times before the next segment). No KV bytes move: the children
 * read the node's blocks through the tree. The node is frozen (no further
 * appends); forking a frozen node adds children. out_children: host
 * array of k ids. Errors: TP_ERR_BAD_NODE, TP_ERR_INVALID_ARG.
 */
tp_status tp_fork(tp_tree* tree, tp_node node, int32_t k, tp_node* out_children);

/*
 * Early stop (Sec. 2.2, heuristic sampling): remove live leaf `leaf`, free
 * its blocks, and free every ancestor whose last live child it was (a tree
 * whose leaves are all pruned disappears, root included). Errors:
 * TP_ERR_BAD_NODE, TP_ERR_NOT_LEAF.
 */
tp_status tp_prune(tp_tree* tree, tp_node leaf);

/*
 * Decode attention for n leaf queries: the next-token step of every live
 * path in one segment-level inference step (Sec. 2.2, Algorithm 1). Row i
 * of Q (device bf16 [n][num_q_heads][head_dim]) attends over every token on
 * the root-to-leaf path of leaves[i] -- its trajectory so far, the
 * concatenation s_1 (+) ... (+) s_j of the path's segments (Sec. 2.3) -- and
 * every prefix segment shared by several listed leaves is read once for all
 * of them (Sec. 2.1 and Sec. 1: shared prefixes computed once). leaves is a
 * host array; a leaf may appear more than once, each occurrence is its own
 * row. Per q-head h (kv head c):
 *   s_j = q_h . k_{j,c} / sqrt(head_dim),  LSE = ln sum_j exp(s_j),
 *   O   = sum_j exp(s_j - LSE) v_{j,c}.
 * O: device bf16 [n][num_q_heads][head_dim]; LSE: device fp32
 * [n][num_q_heads], natural log. Q, O 16-byte aligned, LSE 4-byte aligned.
 * Each path segment shared by several listed leaves is read from HBM once
 * for all of them. n == 0 is a no-op. Asynchronous on the tree's stream.
 * Errors: TP_ERR_BAD_NODE, TP_ERR_NOT_LEAF, TP_ERR_EMPTY_PATH,
 * TP_ERR_INVALID_ARG, TP_ERR_OOM / TP_ERR_CUDA (library scratch).
 */
tp_status tp_decode(tp_tree* tree, const tp_node* leaves, int32_t n, const void* Q, void* O,
                    float* LSE);

/* tp_decode with options (bit flags below). */
#define TP_DECODE_NO_SHARE 1u         /* schedule every leaf's whole path on its own */
#define TP_DECODE_CUDA_CORE_SMALL 2u  /* units of < 16 query rows on the CUDA-core   */
                                      /* path (default: tensor cores, rows padded to */
                                      /* one 16-row MMA tile)                        */
#define TP_DECODE_NO_CACHE 4u         /* rebuild the schedule even if cached         */
#define TP_DECODE_TCGEN05 8u          /* tcgen05 only for chunks of >= 64 stacked    */
                                      /* rows and >= 32 blocks; the other stacked    */
                                      /* rows on mma.sync in 64-row units            */
#define TP_DECODE_ALL_TCGEN05 16u     /* the default: every unit of > 16 stacked     */
                                      /* rows on tcgen05 (128-row units, running     */
                                      /* concurrently with the mma.sync units of one */
                                      /* 16-row tile; measured fastest on GB300);    */
                                      /* by default a call reading < 1 MiB of K/V    */
                                      /* runs all on mma.sync (one kernel: latency-  */
                                      /* bound), this flag forces tcgen05 there too  */
#define TP_MMA_SYNC 32u               /* no tcgen05: stacked rows on mma.sync in     */
                                      /* 64-row units (decode and tp_prefill)        */
tp_status tp_decode_ex(tp_tree* tree, const tp_node* leaves, int32_t n, const void* Q, void* O,
                       float* LSE, uint32_t flags);

/*
 * tp_decode_ex without any device allocation. The paper has no counterpart:
 * this entry point exists for callers that cannot call cudaMalloc on the
 * decode path -- e.g. a serving process whose device memory is carved up at
 * start-up (the KV pool, weights, activations) and that forbids later
 * allocations, or a latency-critical loop that cannot afford cudaMalloc's
 * implicit device synchronisation. tp_decode_ex keeps its schedule and
 * partial results in buffers it grows with cudaMalloc; this variant keeps
 * them in one statically sized device array of TP_NOALLOC_SCRATCH_BYTES that
 * the library declares at file scope (every GPU that loads the library holds
 * it until the process exits) and calls no cudaMalloc, cudaFree or other
 * allocating routine. Arguments and results are those of tp_decode_ex.
 *   - A call whose schedule plus fp32 partials need more than
 *     TP_NOALLOC_SCRATCH_BYTES returns TP_ERR_OOM and launches nothing.
 *   - The first call on a device looks up the array's device address
 *     (cudaGetSymbolAddress, with that device current).
 *   - Every call in the process shares the one array and it keeps the last
 *     call's contents; the unit counters that must start at zero are
 *     cleared by each call. Calls whose device work overlaps -- on two
 *     streams, or from two trees -- race on the array and must not overlap.
 *   - The schedule is copied from a host buffer that lives only for the
 *     call (pageable memory, staged by the driver before the call returns),
 *     so the call is refused with TP_ERR_INVALID_ARG, launching nothing,
 *     while the tree's stream is being captured into a CUDA graph.
 */
#define TP_NOALLOC_SCRATCH_BYTES (32ll << 20)
tp_status tp_decode_noalloc(tp_tree* tree, const tp_node* leaves, int32_t n, const void* Q, void* O,
                            float* LSE, uint32_t flags);

/*
 * Decode-loop append: one token to each of n distinct live leaves (the step
 * of token-level decoding inside a segment, Sec. 2.2). Row i of K and V
 * (device bf16 [n][num_kv_heads][head_dim], 16-byte aligned) becomes the
 * next token of nodes[i] (host array). Equivalent to n calls of
 * tp_append_segment with one token each, in one kernel launch. A decode of
 * the same leaf list after appends that stayed inside the leaves' last
 * blocks reuses its cached schedule (only the leaves' last-block token
 * counts are rewritten on the device). n == 0 is a no-op. Errors:
 * TP_ERR_BAD_NODE, TP_ERR_FROZEN, TP_ERR_OOM (nothing is appended),
 * TP_ERR_INVALID_ARG (also for a node listed twice).
 */
tp_status tp_append_tokens(tp_tree* tree, const tp_node* nodes, int32_t n, const void* K, const void* V);

/*
 * Multi-query (prefill) attention over the tree: the last n_queries[i]
 * tokens of nodes[i] attend causally to that node's root-to-node path --
 * every ancestor token and the node's own tokens up to and including the
 * query's position (the segment-level prefill of Sec. 4.3: a segment's
 * tokens processed together, the shared prefix kept once). Query token j
 * (0-based) of node i sits at path position P_i - n_queries[i] + j, where P_i
 * is the node's path length, and sees positions 0 .. that position:
 *   s_t = q . k_t / sqrt(head_dim) for t <= pos,  LSE = ln sum_t exp(s_t),
 *   O = sum_t exp(s_t - LSE) v_t.
 * nodes: host [n] live nodes (leaves or interior, repeats allowed);
 * n_queries: host [n], 0 <= n_queries[i] <= tokens held by nodes[i]. Q and O:
 * device bf16 [sum n_queries][num_q_heads][head_dim], rows packed node by
 * node in token order; LSE: device fp32 [sum n_queries][num_q_heads]. Q, O
 * 16-byte aligned, LSE 4-byte aligned. Requires num_q_heads / num_kv_heads
 * <= 64. The work runs as tcgen05 units of up to 128 query rows (whole GQA
 * groups); flags = TP_MMA_SYNC runs it on the mma.sync path in 64-row
 * units instead. A row block whose path fits one unit writes O and
 * LSE directly; longer ones are split and merged by log-sum-exp.
 * Asynchronous on the tree's stream. Errors: TP_ERR_BAD_NODE,
 * TP_ERR_INVALID_ARG, TP_ERR_OOM / TP_ERR_CUDA (library scratch).
 */
tp_status tp_prefill(tp_tree* tree, const tp_node* nodes, const int32_t* n_queries, int32_t n, const void* Q,
                     void* O, float* LSE, uint32_t flags);

/* tp_decode_ex and tp_prefill with HOST buffers: the same operation (decode
 * attention over root-to-leaf paths, Sec. 2.3 and 4.3; causal prefill over
 * root-to-node paths), the same leaves / nodes / n_queries / flags and the
 * same row layouts, but Q_host, O_host and LSE_host are host memory. The
 * library uploads Q into device staging of its own, runs the attention there
 * and downloads O and LSE. Library engineering with no counterpart in the
 * paper.
 *
 * Asynchronous, like every attention call: the copies and the kernels are
 * enqueued and the call returns. Q_host must stay unchanged, and O_host /
 * LSE_host unread, until tp_sync returns (tp_sync also waits for these
 * copies). Consecutive host-buffer calls use two staging slots in turn, with
 * the uploads and downloads on copy streams of their own, so a call's copies
 * overlap the neighbouring calls' attention. Page-locked (pinned) host
 * memory makes the copies asynchronous; pageable memory is accepted, but
 * the CUDA runtime then stages it and the call may block. The staging grows
 * to the largest call seen (2 x (Q + O + LSE) bytes) and is freed with the
 * tree. Errors: those of tp_decode_ex / tp_prefill, TP_ERR_INVALID_ARG for a
 * NULL host pointer, TP_ERR_OOM / TP_ERR_CUDA (staging, copies). */
tp_status tp_decode_host(tp_tree* tree, const tp_node* leaves, int32_t n, const void* Q_host, void* O_host,
                         float* LSE_host, uint32_t flags);
tp_status tp_prefill_host(tp_tree* tree, const tp_node* nodes, const int32_t* n_queries, int32_t n,
                          const void* Q_host, void* O_host, float* LSE_host, uint32_t flags);

/* Failure-reporting probe (testing; no counterpart in the paper). Launches,
 * on the tree's stream, one small kernel that runs the attention kernels'
 * bounded wait on a barrier nothing ever completes, with a limit of limit_ns
 * (1e3 .. 1e9) instead of their 2 s; when it runs out the kernel sets the
 * device error flag and returns, so the next tp_sync returns TP_ERR_DEVICE
 * and the tree stays usable. No fault and no trap is involved. Errors:
 * TP_ERR_INVALID_ARG (limit out of range, metadata-only tree), TP_ERR_CUDA. */
tp_status tp_debug_wait_probe(tp_tree* tree, int64_t limit_ns);

/* Wait for the tree's stream (and the copy streams of the host-buffer
 * calls); TP_ERR_DEVICE if a kernel gave up a bounded wait since the last
 * tp_sync (the flag is then cleared), TP_ERR_CUDA on a CUDA error. */
tp_status tp_sync(tp_tree* tree);

/* Message for the last failed call on `tree` (or of tp_tree_create when
 * tree == NULL). Valid until the next call on that tree. Error reporting,
 * no counterpart in the paper. */
const char* tp_last_error(tp_tree* tree);

/* Node state. state: 0 live leaf, 1 frozen interior, 2 dead. */
typedef struct {
    tp_node parent; /* -1 for a root */
    int32_t state;
    int32_t n_tokens;
    int32_t n_live_children;
    int64_t path_tokens; /* tokens on the root-to-node path */
} tp_node_info;
tp_status tp_get_node_info(tp_tree* tree, tp_node node, tp_node_info* out);

/* Pool and forest counters. */
typedef struct {
    int64_t pool_blocks;
    int64_t free_blocks;
    int64_t live_nodes;
    int64_t total_nodes;
} tp_stats;
tp_status tp_get_stats(tp_tree* tree, tp_stats* out);

/* ---- kernel timing ------------------------------------------------------
 * While profiling is on, the library's launches on the tree's stream are
 * bracketed by pairs of CUDA events (the attention kernels of one call
 * together). tp_profile_stop waits for the stream and returns, per kernel
 * kind, the number of kernels launched and the sum of the event-measured
 * durations of their brackets. Index: 0 attention (decode and prefill; the
 * decode schedule's patch kernel is counted here, untimed), 1 LSE merge,
 * 2 appends (copies, stand-in activations, the rollout's token steps),
 * 3 inspection gather. tp_decode_noalloc and tp_tree_advantage are not
 * profiled. */
#define TP_KERNEL_KINDS 4
typedef struct {
    int64_t launches[TP_KERNEL_KINDS];
    double milliseconds[TP_KERNEL_KINDS];
} tp_kernel_times;
tp_status tp_profile_start(tp_tree* tree);
tp_status tp_profile_stop(tp_tree* tree, tp_kernel_times* out);

/* ---- tree sampling (Sec. 2.2, Algorithm 1) ------------------------------ */

/*
 * Branching budget split (Sec. 2.2 budget transfer; Sec. 4.6 probability-
 * based assignment): out[i] >= 1 branches for each of n active paths,
 * summing to budget (>= n). Policies:
 *   TP_BRANCH_EVEN       out[i] = budget / n, plus one for the first
 *                        budget % n paths (logp unused, may be NULL);
 *   TP_BRANCH_LOGP_HIGH  the budget - n branches beyond the first one per
 *   TP_BRANCH_LOGP_LOW   path are split by softmax(+-logp / temperature)
 *                        (HIGH favours paths whose last segment had the
 *                        higher log-probability, LOW the lower), rounded by
 *                        largest remainder, ties to the lower index.
 * logp: host double [n] (finite); out: host int32 [n]. Computed in double
 * precision in index order. Errors: TP_ERR_INVALID_ARG (budget < n,
 * temperature <= 0, non-finite logp, unknown policy).
 */
#define TP_BRANCH_EVEN 0
#define TP_BRANCH_LOGP_HIGH 1
#define TP_BRANCH_LOGP_LOW 2
tp_status tp_branch_assign(const double* logp, int32_t n, int32_t budget, int32_t policy, double temperature,
                           int32_t* out);

/*
 * Rollout parameters. The language model is replaced by a synthetic stand-
 * in whose every draw is SplitMix64 (Steele et al. 2014) element
 *   mix(seed + (ctr + 1) * 0x9E3779B97F4A7C15),
 *   ctr = tag << 60 | a << 32 | b << 12 | c   (a < 2^28, b < 2^20, c < 2^12),
 * read as u = (x >> 11) * 2^-53 in [0, 1) for decisions, or as four bf16
 * values (16 bits each, low bits first: sign bit 15, exponent 124 + bits
 * 7..8, mantissa bits 0..6; values in +-[0.125, 2)) for activations:
 *   K, V, Q of token b of node a: tags 1, 2, 3, c = word of the row
 *       ([heads][head_dim] row-major, 4 values per word);
 *   token b of segment node a is EOS if u(4, a, b, 0) < p_eos (the segment
 *       ends there; else it has seg_tokens tokens); its log-probability is
 *       kappa * ln(1 - u(5, a, b, 0)) with kappa = 2 u(6, a, 0, 0); the
 *       segment's logp is the mean over its tokens;
 *   the segment is "boxed" if u(6, a, 1, 0) < p_boxed, fails the
 *       repetition check if u(6, a, 2, 0) < p_fail; a boxed trajectory
 *       earns reward 1 if u(6, a, 3, 0) < p_correct, else 0;
 *   query q: b0 = 2 + floor(7 u(7, q, 0, 0)) when init_branches == 0; its
 *       k-th fallback picks candidate floor(m u(7, q, 1, k)) of its m live
 *       candidates and boundary floor(J u(7, q, 2, k)) of that candidate's
 *       J segments.
 * Algorithm 1 with these readings:
 *   - each query is a root holding prompt_tokens[q] tokens (depth 0), forked
 *     into min(b0, w) paths; each queued path generates one segment per
 *     loop pass as a new node (depth = parent's + 1);
 *   - a segment that fails is an output and is pruned at once; one that
 *     ends in EOS, is boxed or reaches max_depth finishes its trajectory
 *     (an output; a candidate for fallback if EOS or boxed); every other
 *     path continues;
 *   - branching: the continuing paths of query q at depth j are forked to
 *     min(b0 * arity^j, w - outputs_q) paths (never fewer than one each),
 *     split by `policy`; queries in ascending order, paths in queue order;
 *   - fallback (if enabled): after branching, a query with no path and
 *     fewer than w outputs forks one new path from the chosen boundary
 *     node of a live candidate; candidates stay alive (their KV kept) until
 *     their query is done, otherwise finished paths are pruned at once;
 *   - a query with no path after fallback is done: its candidates are pruned.
 * With decode != 0 (device pool needed), every generated token is appended
 * with tp_append_tokens and the paths still generating decode (tp_decode_ex
 * with decode_flags); with decode == 0 each segment is appended whole.
 */
typedef struct {
    int32_t n_queries;
    const int32_t* prompt_tokens; /* host [n_queries], each in [1, 2^20] */
    int32_t width;                /* w >= 1: trajectories per query      */
    int32_t max_depth;            /* d >= 1: segments per trajectory     */
    int32_t seg_tokens;           /* l >= 1: tokens per segment          */
    int32_t arity;                /* N >= 1                              */
    int32_t init_branches;        /* b0 >= 1, or 0: b0 drawn in [2, 8]   */
    int32_t policy;               /* TP_BRANCH_*                         */
    int32_t fallback;             /* nonzero: depth-first-search fallback */
    int32_t decode;               /* nonzero: decode after every token   */
    uint32_t decode_flags;        /* tp_decode_ex flags                  */
    int32_t reserved;
    double temperature;           /* > 0 for the log-prob policies       */
    double p_eos, p_boxed, p_fail, p_correct;
    uint64_t seed;
} tp_rollout_params;

/* Segment status bits (event TP_EV_SEGMENT). */
#define TP_SEG_EOS 1
#define TP_SEG_BOXED 2
#define TP_SEG_FAILED 4
#define TP_SEG_MAX_DEPTH 8

/* Events: int64 records of 8 words {kind, query, node, a, b, c, d, 0}.
 *   TP_EV_ROOT      node = root, a = prompt tokens, b = b0
 *   TP_EV_FORK      node = parent, a = first child (children are
 *                   consecutive ids), b = k
 *   TP_EV_SEGMENT   node, a = depth, b = tokens, c = TP_SEG_* bits,
 *                   d = bits of the double segment logp
 *   TP_EV_OUTPUT    node = leaf, a = depth, b = fallback candidate, c = reward
 *   TP_EV_PRUNE     node = leaf
 *   TP_EV_FALLBACK  node = candidate leaf, a = boundary node, b = its depth
 *   TP_EV_DONE      node = -1, a = outputs of the query */
#define TP_EV_ROOT 1
#define TP_EV_FORK 2
#define TP_EV_SEGMENT 3
#define TP_EV_OUTPUT 4
#define TP_EV_PRUNE 5
#define TP_EV_FALLBACK 6
#define TP_EV_DONE 7

typedef struct {
    int64_t iterations;    /* loop passes (Inference calls)          */
    int64_t segments;      /* generated segments                     */
    int64_t tokens;        /* generated tokens                       */
    int64_t prompt_tokens; /* prompt tokens appended                 */
    int64_t outputs;       /* trajectories in O                      */
    int64_t fallbacks;
    int64_t decode_calls;
    int64_t decode_rows;   /* leaf queries over all decode calls     */
    int64_t events;        /* events produced (may exceed the cap)   */
    int64_t peak_blocks;   /* most pool blocks in use at once        */
    int64_t nodes;         /* nodes created                          */
} tp_rollout_stats;

/* Optional copy-out of one decode call of a rollout (for checking it): the
 * call with index `call` (0-based over the rollout) copies its first
 * min(rows, cap) rows of O (device bf16 [cap][num_q_heads][head_dim]) and
 * LSE (device fp32 [cap][num_q_heads]); rows (host int32 [cap][2]) gets
 * each row's (leaf node, token index inside the leaf), *n_rows the count. */
typedef struct {
    int64_t call;
    int32_t cap;
    int32_t reserved;
    void* o;
    float* lse;
    int32_t* rows;
    int32_t* n_rows;
} tp_rollout_probe;

/*
 * Run Algorithm 1 for p->n_queries new prompts in `tree` (roots are added
 * to whatever the tree holds). events: host int64 [cap_events][8] or NULL;
 * stats->events tells how many were produced. probe, stats: optional.
 * Returns when the rollout is done; device work is enqueued on the tree's
 * stream. On error the rollout stops where it failed (the tree keeps what
 * was built). Errors: TP_ERR_INVALID_ARG, TP_ERR_OOM (pool exhausted),
 * and those of the calls above.
 */
tp_status tp_rollout(tp_tree* tree, const tp_rollout_params* params, int64_t* events, int64_t cap_events,
                     const tp_rollout_probe* probe, tp_rollout_stats* stats);

/*
 * Stand-in activations, as the rollout draws them: K, V ([n][num_kv_heads]
 * [head_dim]) and Q ([n][num_q_heads][head_dim]) bf16 rows of tokens
 * pos0 .. pos0 + n - 1 of node key `node` (device pointers, 8-byte aligned,
 * any may be NULL). The paper has no counterpart; it exposes the synthetic
 * inputs so they can be checked. node < 2^28, pos0 + n <= 2^20.
 */
tp_status tp_synth_tokens(tp_tree* tree, uint64_t seed, tp_node node, int32_t pos0, int32_t n_tokens, void* K,
                          void* V, void* Q);

/* ---- tree advantage (Sec. 2.3, Eq. tree_ae) ----------------------------- */

/*
 * Advantage of each trajectory from the sub-groups of the tree. Trajectory
 * i ends at node leaf[i] with reward[i]; its sub-groups are the strict
 * ancestors x of leaf[i] (depth 0 = the query's root, through the leaf's
 * parent), G_x = the trajectories below x. Then
 *   A_i   = (1 / |J_i|) sum_{x in J_i} (R_i - mean_{G_x} R)   (mean pooling)
 *   adv_i = A_i / std(A)                       (global normalisation)
 * where std is the population standard deviation over every accepted
 * trajectory of the call. A trajectory is rejected (adv 0, left out of the
 * std) when all rewards of its query (root) are equal (std(R) = 0) or its
 * leaf is a root; adv is 0 everywhere when std(A) = 0.
 * parent: device int32 [n_nodes] (-1 for roots; parent ids need not be
 * smaller than their children's), leaf: device int32 [n_out], reward:
 * device fp32 [n_out] (finite), adv: device fp32 [n_out]. stats: device
 * double [4] or NULL: accepted trajectories, mean(A), std(A), and 1 if the
 * parent table was malformed (an id out of range or a cycle; the affected
 * trajectories are rejected). workspace: device, 8-byte aligned, at least
 * tp_advantage_workspace_bytes(n_nodes, n_out) bytes. Fp64 accumulation,
 * four kernels (clear, ancestor sums, sub-group means, per-trajectory A_i
 * with the last CTA normalising), asynchronous on cuda_stream; calls
 * sharing a workspace must not overlap. Errors (tp_last_error(NULL)):
 * TP_ERR_INVALID_ARG, TP_ERR_CUDA.
 */
int64_t tp_advantage_workspace_bytes(int32_t n_nodes, int32_t n_out);
tp_status tp_tree_advantage(const int32_t* parent, int32_t n_nodes, const int32_t* leaf, const float* reward,
                            int32_t n_out, float* adv, double* stats, void* workspace, int64_t workspace_bytes,
                            void* cuda_stream);

/* ---- inspection (tests and tools) ------------------------------------ */

/* Pool slot of every token on leaf's root-to-leaf path (its trajectory
 * s_1 (+) ... (+) s_j, Sec. 2.3), root first.
 * slots: host int64 [cap]; *n receives the path length (slots untouched
 * beyond cap; TP_ERR_INVALID_ARG if cap < length). */
tp_status tp_debug_path(tp_tree* tree, tp_node leaf, int64_t* slots, int64_t cap, int64_t* n);

/* Copy leaf's path K and V out of the pool on the device, through the same
 * block tables the decode kernels read. K_out, V_out: device bf16
 * [cap_tokens][num_kv_heads][head_dim], 16-byte aligned; *n receives the
 * path length (TP_ERR_INVALID_ARG if cap_tokens < length). */
tp_status tp_debug_gather(tp_tree* tree, tp_node leaf, void* K_out, void* V_out,
                          int64_t cap_tokens, int64_t* n);

/*
 * The decode schedule tp_decode_ex(flags) would run, as int32 words in host
 * buf[cap]; *len receives the word count (TP_ERR_INVALID_ARG if cap is too
 * small; call with cap 0 to size). Layout:
 *   [0] magic 0x54505344, [1] n_units, [2] n_tiles, [3] n_occ_entries,
 *   [4] n (leaf occurrences), [5] n_slots, [6] n_merge_entries, [7] group g,
 *   [8] n_mma_units, [9] n_tcgen05_units, [10] 0 (1 for prefill schedules),
 *   [11] 16 (words per merge record; 0 in prefill schedules, which have
 *   none), [12..15] reserved (0),
 *   then units  [n_units][8]: tile_off, n_tiles, occ_off, row0, n_rows,
 *                             slot_base, kv_head, kind (0 CUDA-core,
 *                             1 mma.sync, 2 tcgen05); tcgen05 units first,
 *                             then mma.sync, then CUDA-core,
 *   then tiles  [n_tiles]: block << 7 | (valid_tokens - 1),
 *   then occ    [n_occ_entries]: leaf occurrence index (row i of Q),
 *   then merge_off [n + 1], then merge_slot [n_merge_entries],
 *   then merge_rec [n][16]: occurrence i's slot count and its slots in
 *                             merge_slot order, zero-padded ([-1, 0...] when
 *                             it has more than 15: the CSR holds them).
 * Unit row r (0 <= r < n_rows) is item row row0 + r = p * g + j: occurrence
 * occ[occ_off + p], q-head kv_head * g + j, written to partial slot
 * slot_base + p. Occurrence i merges slots merge_slot[merge_off[i] ..
 * merge_off[i+1]).
 */
tp_status tp_debug_schedule(tp_tree* tree, const tp_node* leaves, int32_t n, uint32_t flags,
                            int32_t* buf, int64_t cap, int64_t* len);

/*
 * Check a schedule (the word layout of tp_debug_schedule and
 * tp_debug_prefill_schedule) on the host with the index predicates that the
 * bounds-checked build of the kernels applies before every access: each
 * unit record's tiles inside the tile section (at most 128), its kind in
 * launch order, its rows' occurrence entries inside the occurrence list and
 * their partial slots below n_slots (slot_base -1 only in prefill
 * schedules), its kv head below num_kv_heads; each tile word's block below
 * the tree's pool_blocks with 1..32 valid tokens; each occurrence entry
 * below n; each occurrence's merge range inside the merge list, and its
 * merge record's count equal to the range's length (or -1 past 15); each
 * merge slot, and each slot of a merge record, below n_slots (a record's
 * slots equal to its CSR range). violations: host int64 [5] receives the number of bad
 * unit records, tile words, occurrence entries, merge ranges and merge
 * slots. Errors: TP_ERR_INVALID_ARG (not a schedule: bad magic, bad header,
 * shorter than its header says).
 */
tp_status tp_debug_check_schedule(tp_tree* tree, const int32_t* words, int64_t n_words, int64_t* violations);

/* The schedule tp_prefill would run, in the layout above with header word
 * [10] = 1, no merge records ([11] = 0) and two more sections in their
 * place: unit_pos [n_units] (path position of each unit's first token) and
 * vis [n] (tokens of its path that occurrence i -- query token i -- may
 * see). Occurrences are the query
 * tokens; units are tcgen05 units (mma.sync units with TP_MMA_SYNC); a unit
 * row whose occurrence sees nothing of the unit is computed but has no merge
 * entry. */
tp_status tp_debug_prefill_schedule(tp_tree* tree, const tp_node* nodes, const int32_t* n_queries, int32_t n,
                                    uint32_t flags, int32_t* buf, int64_t cap, int64_t* len);

#ifdef __cplusplus
}
#endif
#endif /* TREEPO_H_ */
