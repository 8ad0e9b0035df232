/*
 * attention_oracle.c -- reference oracle for decode attention over a paged
 * key/value cache.
 *
 * TEST INFRASTRUCTURE ONLY.  Plain, slow, single-threaded fp64 C: the
 * definition the CUDA attention path is checked against.  Only the test
 * suite, the smoke check and the benchmark's CPU-baseline leg may load it;
 * the product library never links or calls it and shares no code with it.
 *
 * The paper's compiled models use PagedAttention (a key/value cache held in
 * fixed-size pages addressed through a per-sequence page table) and
 * FlashAttention kernels (Section 2.3).  Both compute ordinary softmax
 * attention; what they change is where the cache lives and the order of the
 * arithmetic.  The oracle therefore writes out plain softmax attention of one
 * decode step, reading keys and values through the page table:
 *
 *   cache       K, V : fp16 [num_pages][n_kv_heads][page_size][head_dim];
 *   page table  P    : int32 [batch][pt_stride]; token t of sequence b lives
 *                      in page P[b][t / page_size], row t % page_size;
 *   query       q    : fp16, row b at q + b*q_stride, heads [n_q_heads][head_dim];
 *   grouping    query head j reads key/value head j / G, G = n_q_heads / n_kv_heads
 *                      (grouped-query attention);
 *   for T = seq_lens[b] > 0 and t < T:
 *     s_t   = scale * sum_d q[b][j][d] * K_t[d]               (fp64, increasing d)
 *     m     = max_t s_t
 *     e_t   = exp(s_t - m)
 *     Z     = sum_t e_t                                         (increasing t)
 *     o[d]  = sum_t e_t * V_t[d] / Z                            (increasing t)
 *     A[d]  = sum_t e_t * |V_t[d]| / Z    (magnitude used by the tolerance)
 *   T = 0 gives o = A = 0 (attention over nothing is defined as zero here).
 *   fp16 output: fp16_RNE(o).
 *
 * The subtraction of m changes nothing mathematically (softmax is invariant
 * to a common shift); it keeps exp() finite for large scores.
 *
 * The append step of a decode iteration writes the new token's key and value
 * into its page: cache[P[b][pos / page_size]][h][pos % page_size][:] = new[b][h][:].
 */
#include <math.h>
#include <stdint.h>
#include <string.h>

#define WQ4O_EXPORT __attribute__((visibility("default")))

/* fp16 codec of wq4_oracle.c (same library). */
double wq4o_half_to_double(uint16_t h);
uint16_t wq4o_double_to_half(double v);

static const uint16_t* cache_row(const uint16_t* cache, int n_kv_heads, int page_size, int head_dim, int page,
                                 int h, int row)
{
    return cache + (((int64_t)page * n_kv_heads + h) * page_size + row) * (int64_t)head_dim;
}

/*
 * Decode attention of every (sequence, query head).  o and A are fp64
 * [batch][n_q_heads][head_dim]; o16 the fp16 bits of o.  Returns 0, or -1 on
 * a page id outside [0, num_pages) or n_q_heads not a multiple of n_kv_heads.
 */
WQ4O_EXPORT int wq4o_paged_attention(const uint16_t* q, int q_stride, const uint16_t* k_cache,
                                     const uint16_t* v_cache, int num_pages, int page_size, const int32_t* page_table,
                                     int pt_stride, const int32_t* seq_lens, int batch, int n_q_heads, int n_kv_heads,
                                     int head_dim, double scale, double* o, double* A, uint16_t* o16)
{
    if (n_kv_heads < 1 || n_q_heads % n_kv_heads != 0) return -1;
    const int G = n_q_heads / n_kv_heads;
    for (int b = 0; b < batch; ++b) {
        const int T = seq_lens[b] > 0 ? seq_lens[b] : 0;
        for (int t = 0; t < T; ++t) {
            const int page = page_table[(int64_t)b * pt_stride + t / page_size];
            if (page < 0 || page >= num_pages) return -1;
        }
    }
    for (int b = 0; b < batch; ++b) {
        const int T = seq_lens[b] > 0 ? seq_lens[b] : 0;
        for (int j = 0; j < n_q_heads; ++j) {
            const int h = j / G;
            const uint16_t* qj = q + (int64_t)b * q_stride + (int64_t)j * head_dim;
            double* oj = o + ((int64_t)b * n_q_heads + j) * head_dim;
            double* Aj = A + ((int64_t)b * n_q_heads + j) * head_dim;
            uint16_t* o16j = o16 + ((int64_t)b * n_q_heads + j) * head_dim;
            for (int d = 0; d < head_dim; ++d) {
                oj[d] = 0.0;
                Aj[d] = 0.0;
            }
            if (T == 0) {
                for (int d = 0; d < head_dim; ++d) o16j[d] = wq4o_double_to_half(0.0);
                continue;
            }
            /* scores s_t (first pass), their maximum m */
            double m = -INFINITY;
            for (int t = 0; t < T; ++t) {
                const int page = page_table[(int64_t)b * pt_stride + t / page_size];
                const uint16_t* kt = cache_row(k_cache, n_kv_heads, page_size, head_dim, page, h, t % page_size);
                double dot = 0.0;
                for (int d = 0; d < head_dim; ++d) dot += wq4o_half_to_double(qj[d]) * wq4o_half_to_double(kt[d]);
                const double st = scale * dot;
                if (st > m) m = st;
            }
            /* e_t, Z and the weighted sums (second pass, recomputing s_t) */
            double Z = 0.0;
            for (int t = 0; t < T; ++t) {
                const int page = page_table[(int64_t)b * pt_stride + t / page_size];
                const uint16_t* kt = cache_row(k_cache, n_kv_heads, page_size, head_dim, page, h, t % page_size);
                const uint16_t* vt = cache_row(v_cache, n_kv_heads, page_size, head_dim, page, h, t % page_size);
                double dot = 0.0;
                for (int d = 0; d < head_dim; ++d) dot += wq4o_half_to_double(qj[d]) * wq4o_half_to_double(kt[d]);
                const double e = exp(scale * dot - m);
                Z += e;
                for (int d = 0; d < head_dim; ++d) {
                    const double v = wq4o_half_to_double(vt[d]);
                    oj[d] += e * v;
                    Aj[d] += e * fabs(v);
                }
            }
            for (int d = 0; d < head_dim; ++d) {
                oj[d] /= Z;
                Aj[d] /= Z;
                o16j[d] = wq4o_double_to_half(oj[d]);
            }
        }
    }
    return 0;
}

/*
 * Append step: writes new_k / new_v row b (heads [n_kv_heads][head_dim] at
 * new_k + b*new_stride) at position positions[b] of sequence b.  Returns 0,
 * or -1 when a position is negative or maps to a page id outside
 * [0, num_pages) (nothing is written for that sequence).
 */
WQ4O_EXPORT int wq4o_kv_append(const uint16_t* new_k, const uint16_t* new_v, int new_stride, uint16_t* k_cache,
                               uint16_t* v_cache, int num_pages, int page_size, const int32_t* page_table,
                               int pt_stride, const int32_t* positions, int batch, int n_kv_heads, int head_dim)
{
    int rc = 0;
    for (int b = 0; b < batch; ++b) {
        const int pos = positions[b];
        if (pos < 0) {
            rc = -1;
            continue;
        }
        const int page = page_table[(int64_t)b * pt_stride + pos / page_size];
        if (page < 0 || page >= num_pages) {
            rc = -1;
            continue;
        }
        for (int h = 0; h < n_kv_heads; ++h) {
            const int64_t dst = (((int64_t)page * n_kv_heads + h) * page_size + pos % page_size) * head_dim;
            const int64_t src = (int64_t)b * new_stride + (int64_t)h * head_dim;
            memcpy(k_cache + dst, new_k + src, sizeof(uint16_t) * (size_t)head_dim);
            memcpy(v_cache + dst, new_v + src, sizeof(uint16_t) * (size_t)head_dim);
        }
    }
    return rc;
}
