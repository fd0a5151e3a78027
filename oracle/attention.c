/*
 * oracle/attention.c -- TEST INFRASTRUCTURE ONLY.
 *
 * Plain, slow, fp64 decode attention over ONE materialised root-to-leaf path.
 * Only the tests, the smoke check and the benchmark's CPU-baseline leg may
 * load this file's library; the product library never does.
 *
 * What it computes. TreePO samples a trajectory as a concatenation of
 * segments s_1 (+) ... (+) s_j along a root-to-leaf path (Sec. 2.3, the
 * trajectory decomposition; Sec. 2.2, Algorithm 1 appends each generated
 * segment to its prompt). A decode query of that leaf attends to every token
 * cached on the path; sharing the prefix KV between sibling branches
 * (Sec. 1 and 2.1) changes where the bytes live, not the value. The paper
 * gives no attention formula, so the standard scaled-dot-product softmax
 * attention is written out, with these readings:
 *   scale 1/sqrt(head_dim); contiguous GQA groups (q-head h uses kv head
 *   h / (Hq/Hkv)); natural-log LSE; no positional transform inside.
 *
 * For q-head h (kv head c = h / g) over the N path tokens j:
 *   s_j  = (q_h . k_{j,c}) / sqrt(d)
 *   M    = max_j s_j
 *   LSE  = M + ln( sum_j exp(s_j - M) )
 *   O    = sum_j exp(s_j - LSE) v_{j,c}
 * Inputs are bf16 bit patterns, widened exactly to fp64.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

static double bf16_bits_to_f64(uint16_t b) {
    uint32_t u = ((uint32_t)b) << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/*
 * q: [Hq][d] bf16 bits; k, v: [N][Hkv][d] bf16 bits (the materialised path,
 * root first); out: [Hq][d] fp64; lse: [Hq] fp64.
 * Returns 0, or -1 on a bad argument (N < 1, Hq not a multiple of Hkv, ...).
 */
int oracle_path_attention(int64_t n_tokens, int32_t num_q_heads, int32_t num_kv_heads,
                          int32_t head_dim, const uint16_t* q, const uint16_t* k,
                          const uint16_t* v, double* out, double* lse) {
    if (n_tokens < 1 || num_q_heads < 1 || num_kv_heads < 1 || head_dim < 1) return -1;
    if (num_q_heads % num_kv_heads != 0) return -1;
    const int32_t g = num_q_heads / num_kv_heads;
    const double scale = 1.0 / sqrt((double)head_dim);
    double* s = (double*)malloc(sizeof(double) * (size_t)n_tokens);
    if (!s) return -1;
    for (int32_t h = 0; h < num_q_heads; ++h) {
        const int32_t c = h / g;
        const uint16_t* qh = q + (int64_t)h * head_dim;
        /* scores */
        for (int64_t j = 0; j < n_tokens; ++j) {
            const uint16_t* kj = k + (j * num_kv_heads + c) * head_dim;
            double dot = 0.0;
            for (int32_t d = 0; d < head_dim; ++d)
                dot += bf16_bits_to_f64(qh[d]) * bf16_bits_to_f64(kj[d]);
            s[j] = dot * scale;
        }
        /* log-sum-exp */
        double m = s[0];
        for (int64_t j = 1; j < n_tokens; ++j)
            if (s[j] > m) m = s[j];
        double sum = 0.0;
        for (int64_t j = 0; j < n_tokens; ++j) sum += exp(s[j] - m);
        const double l = m + log(sum);
        lse[h] = l;
        /* output */
        double* oh = out + (int64_t)h * head_dim;
        for (int32_t d = 0; d < head_dim; ++d) oh[d] = 0.0;
        for (int64_t j = 0; j < n_tokens; ++j) {
            const double p = exp(s[j] - l);
            const uint16_t* vj = v + (j * num_kv_heads + c) * head_dim;
            for (int32_t d = 0; d < head_dim; ++d) oh[d] += p * bf16_bits_to_f64(vj[d]);
        }
    }
    free(s);
    return 0;
}
