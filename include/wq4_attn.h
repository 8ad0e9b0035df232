/*
 * wq4_attn.h -- decode attention over a paged key/value cache (sm_103a),
 * part of the same library as wq4.h (libwq4.so).
 *
 * The paper's compiled models run PagedAttention (keys and values kept in
 * fixed-size pages reached through a per-sequence page table, Kwon et al.)
 * and FlashAttention (softmax computed in one pass with a running maximum,
 * Dao et al.) as their attention kernels (Section 2.3).  One decode step of
 * one layer computes, for sequence b and query head j (key/value head
 * h = j / G, G = n_q_heads / n_kv_heads: grouped-query attention),
 *
 *   s_t = scale * q[b][j] . K_t,   o[b][j] = sum_t softmax(s)_t * V_t,
 *
 * over the T = seq_lens[b] cached tokens t, token t being row t % page_size
 * of page page_table[b][t / page_size].
 *
 * Accuracy contract: |o - o_ref| <= 2e-3 * sum_t p_t |V_t| + ulp16(|o_ref|)
 * per element, o_ref and p the exact (fp64) result and weights.  The path
 * rounds each weight to fp16 for the value product and normalises by the sum
 * of the same rounded weights (<= 2 * 2^-11 relative per weight); scores and
 * all sums are fp32.  Valid while scale * sum_d |q_d K_t,d| <= 64.
 *
 * Conventions are those of wq4.h: device pointers owned by the caller,
 * asynchronous on `stream`, no allocation, argument errors returned before
 * anything is enqueued, device-side problems (a page id outside the pool, a
 * length beyond the page table, a wait that gave up) recorded in the status
 * word that wq4_device_status() reads and clears.
 */
#ifndef WQ4_ATTN_H
#define WQ4_ATTN_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* The paged cache of one layer. */
typedef struct {
    uint16_t* k;                 /* fp16 [num_pages][n_kv_heads][page_size][head_dim], 16-byte aligned */
    uint16_t* v;                 /* same shape and alignment; must not overlap k */
    int num_pages;               /* pages in the pool, >= 1 */
    int n_kv_heads;              /* >= 1 */
    int page_size;               /* tokens per page: a multiple of 16 */
    int head_dim;                /* 128 */
    const int32_t* page_table;   /* int32 [batch][page_table_stride]: page ids of each sequence */
    int page_table_stride;       /* >= 1: entries per sequence (max pages of a sequence) */
} wq4_kv_cache;

/* Largest batch wq4_paged_attention accepts. */
#define WQ4_ATTN_MAX_BATCH 1024

/*
 * Workspace wq4_paged_attention needs for this geometry on the current
 * device: arrival counters (batch * n_kv_heads words, which must be zero
 * before the first call and are left zero by every call that completes) and
 * fp32 partial results of sequences split across thread blocks.  0 on bad
 * arguments.
 */
size_t wq4_paged_attention_workspace_bytes(int batch, int n_q_heads, int n_kv_heads, int head_dim);

/*
 * Decode attention of every sequence and query head (definition above).
 *   cache      : the layer's paged cache (pointers are device pointers).
 *   q          : fp16 [batch] rows of q_stride elements, each holding
 *                [n_q_heads][head_dim] (a row of the fused QKV projection
 *                output works: its first n_q_heads*head_dim entries are q);
 *                16-byte aligned, q_stride % 8 == 0.
 *   seq_lens   : int32 [batch] device array, tokens in the cache per
 *                sequence (the current token included); 0 gives o = 0;
 *                larger than page_table_stride * page_size is clamped and
 *                flagged.
 *   out        : fp16 [batch] rows of out_stride elements, [n_q_heads][head_dim]
 *                each; 4-byte aligned, out_stride even; must not overlap the
 *                inputs or the workspace.
 *   n_q_heads  : a multiple of n_kv_heads with n_q_heads / n_kv_heads <= 8.
 *   scale      : the score scale (1/sqrt(head_dim) for standard attention).
 *   workspace  : device memory of wq4_paged_attention_workspace_bytes(),
 *                16-byte aligned, not shared by concurrent calls.
 * Sequences are split across the GPU's thread blocks by tokens in equal
 * shares and the shares are merged in a fixed order: the same inputs on the
 * same device give the same bits.  Returns WQ4_OK, WQ4_ERR_INVALID,
 * WQ4_ERR_ALIGN, WQ4_ERR_UNSUPPORTED (head_dim != 128, group > 8) or
 * WQ4_ERR_CUDA.
 */
int wq4_paged_attention(const wq4_kv_cache* cache, const uint16_t* q, int q_stride, const int32_t* seq_lens,
                        uint16_t* out, int out_stride, int batch, int n_q_heads, float scale, void* workspace,
                        size_t workspace_bytes, void* stream);

/*
 * Append step of a decode iteration: writes the new token's key and value of
 * every key/value head into the cache,
 *   cache.k[page_table[b][pos / page_size]][h][pos % page_size][:] = new_k[b][h][:]
 * (and likewise v) with pos = positions[b] (device int32 [batch]).
 *   new_k, new_v : fp16 [batch] rows of new_stride elements holding
 *                  [n_kv_heads][head_dim] (rows of the fused QKV output, offset
 *                  to their k and v parts, work); 16-byte aligned,
 *                  new_stride % 8 == 0.
 * A negative position, one beyond the page table, or a page id outside the
 * pool writes nothing for that sequence and is flagged.  Bit-exact copy.
 */
int wq4_kv_append(const wq4_kv_cache* cache, const uint16_t* new_k, const uint16_t* new_v, int new_stride,
                  const int32_t* positions, int batch, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* WQ4_ATTN_H */
