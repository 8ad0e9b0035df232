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

#include "wq4.h"

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

/* ------------------------------------------------------------------------ */
/* Decode step with attention                                               */
/* ------------------------------------------------------------------------ */

/*
 * The attention of one decode step (Section 2.3: the compiled models run
 * PagedAttention and FlashAttention between their projections).  The paper
 * names no positional encoding; its models (Llama-3.1, Phi-3.5) rotate q and
 * k, and this library's reading of that rotation is: within each head the
 * adjacent pair (x_2i, x_2i+1) turns by pos * rope_theta^(-2i / head_dim),
 * computed in fp64 on the fp16 values and rounded once to fp16.
 *   layers     : HOST array of num_layers caches (device pointers inside),
 *                all with the table's n_kv_heads, head_dim 128 and one common
 *                page_size (a multiple of 16); page tables [batch][stride].
 *                Sequences of a batch must not map their new positions to
 *                the same cache row.
 *   positions  : device int32 [batch]: the new token's place in its sequence
 *                (the number of tokens already cached).
 *   rope_theta : rotary base (> 1; Llama-3.x 500000, Phi-3.5 10000).
 *   scale      : attention score scale (> 0, normally 1/sqrt(head_dim)).
 */
typedef struct {
    const wq4_kv_cache* layers;
    const int32_t* positions;
    double rope_theta;
    float scale;
} wq4_decode_attn;

/* Workspace bytes (table->workspace_bytes) wq4_decode_step needs: the chain's
 * workspace plus the attention buffers (for batch 3-32 it includes
 * wq4_paged_attention's workspace, which depends on the current device).
 * 0 if the table is invalid or its heads are unsupported (head_dim != 128,
 * n_q_heads / n_kv_heads not a whole number <= 8). */
size_t wq4_decode_step_workspace_bytes(const wq4_layer_table* table);

/*
 * One decode step of every sequence of the batch: the chain of wq4_decode_chain
 * with the query-block stand-in replaced by attention.  For layer l and row b,
 * after the QKV projection:
 *   q = rope(qkv[:, :H]), k = rope(qkv[:, H:H + Hkv*128]), v = qkv[:, H + Hkv*128:]
 *   layers[l] gets k, v at position positions[b] (as wq4_kv_append)
 *   a = fp16( attention(q, layers[l], positions[b] + 1 tokens) )
 * and a is the O projection's input (o = r(a) W_o . a).  Batch 1-2 runs the
 * attention inside the persistent chain kernel (split over the GPU's blocks,
 * fp32 scores and softmax); batch 3-32 records wq4_paged_attention and a
 * rotation/append kernel into its CUDA graph.  Accuracy: rotated q and k
 * within one fp16 ulp of the exact rotation of the fp16 projection outputs;
 * a within the attention contract of wq4_paged_attention; the projections as
 * in wq4_decode_chain.  Device-side problems are flagged in the status word
 * (bit 5: a position or page id that makes the append impossible, nothing
 * written; bit 3: a length beyond the page table, clamped; bit 4: a page id
 * outside the pool, zeros read).  The plan is built at the first call (and
 * rebuilt when the table or this description changes) as for
 * wq4_decode_chain; table->workspace must hold
 * wq4_decode_step_workspace_bytes(table) bytes.
 * Returns WQ4_OK, WQ4_ERR_INVALID, WQ4_ERR_ALIGN, WQ4_ERR_UNSUPPORTED or
 * WQ4_ERR_CUDA.
 */
int wq4_decode_step(const wq4_layer_table* table, const wq4_decode_attn* attn, const uint16_t* x,
                    uint16_t* logits, void* stream);

/* The same step with HOST buffers (x_host fp16 [batch][hidden], logits_host
 * fp16 [batch][vocab]): copies x in, runs the step, copies the logits out and
 * synchronizes `stream`. */
int wq4_decode_step_host(const wq4_layer_table* table, const wq4_decode_attn* attn, const uint16_t* x_host,
                         uint16_t* logits_host, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* WQ4_ATTN_H */
