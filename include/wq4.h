/*
 * wq4.h -- C ABI of the GB300 (sm_103a) 4-bit weight-streaming GEMV library.
 *
 * The paper's decode workload is token generation with 4-bit quantized
 * models (Section 3, Table 1; Section 1 quotes about 90 tokens/s for a 4-bit
 * 3B model on a laptop GPU).  Each decoded token streams every weight matrix
 * once: the fused QKV, attention-output, gate_up and down projections of each
 * layer and the LM head.  The paper's compiler produces these kernels with
 * "kernel fusion" and "GEMM tiling" (Section 2.3) and ships the weights as an
 * offline-converted artifact (Section 2.3); this library is the GB300 form of
 * that hot path, written by hand.
 *
 * Weight format (the paper says only "4-bit quantized"; this library fixes it):
 *   W_packed  uint32 [N][K/8]  code k of row n is bits [4*(k%8), 4*(k%8)+4) of
 *                              word W[n][k/8] (lowest nibble first), 0..15;
 *   scales    fp16   [N][K/32] one scale per group of 32 consecutive codes;
 *   weight    w(n,k) = (q(n,k) - 7) * scales[n][k/32].
 * Activations x are fp16 [batch][K], outputs y are fp16 [batch][N]; products
 * are accumulated in fp32 and y is rounded to nearest even.
 * Accuracy contract: |y - y_ref| <= 1e-3 * sum_k |w*x| + ulp16(|y_ref|),
 * y_ref being the exact (fp64) sum.
 *
 * Conventions for every call below:
 *   - Pointers named W, scales, x, y, w_out, q_out, logits are DEVICE pointers
 *     (unless the name says host) owned by the caller; the library never frees
 *     them and never keeps them beyond the call, except the chain plan, which
 *     remembers the layer table's pointers until wq4_chain_plan_destroy.
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *     stream).  Device calls are asynchronous: they validate, enqueue and
 *     return; they never synchronize (except where stated) and never allocate
 *     device memory.
 *   - Argument errors return before anything is enqueued.  A CUDA launch
 *     failure returns WQ4_ERR_CUDA.
 *   - Device-side waits are bounded; a wait that gives up records a flag that
 *     wq4_device_status() reports, and the kernel still terminates.
 */
#ifndef WQ4_H
#define WQ4_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

enum wq4_status {
    WQ4_OK = 0,
    WQ4_ERR_INVALID = -1,     /* bad size, null pointer, aliasing, bad table */
    WQ4_ERR_ALIGN = -2,       /* a pointer is below the alignment the call needs */
    WQ4_ERR_UNSUPPORTED = -3, /* valid arguments outside what this build handles */
    WQ4_ERR_CUDA = -4,        /* a CUDA runtime call failed */
    WQ4_ERR_TIMEOUT = -5      /* a device-side wait gave up (see wq4_device_status) */
};

/* Largest batch (rows of x) any call accepts. */
#define WQ4_MAX_BATCH 32

/* Largest scale magnitude of the paths that round the dequantized weight
 * (q - 7) * s to fp16 (wq4_gemm, wq4_decode_chain at batch 3-32). */
#define WQ4_MAX_FP16_SCALE 8188.0f

/*
 * y[b][n] = fp16( sum_k (q(n,k) - 7) * scales[n][k/32] * x[b][k] )
 * for b < batch, n < N: the fused dequantize-and-multiply projection of one
 * decode step (Section 3, Table 1 workload; Section 2.3 "kernel fusion":
 * dequantization happens in registers, the fp32 weights never exist in
 * memory).
 *   W_packed : uint32 [N][K/8], 16-byte aligned.
 *   scales   : fp16 bits [N][K/32], 2-byte aligned (16-byte aligned and
 *              K % 256 == 0 select the TMA-staged fast paths: at batch 1-2
 *              from 12 Mi weights the legacy-tensor-path kernel, exact in
 *              fp16 products with fp32 sums, else the CUDA-core one).
 *   x        : fp16 bits [batch][K], 16-byte aligned.
 *   y        : fp16 bits [batch][N], 2-byte aligned; must not overlap x, W or
 *              scales.
 *   N >= 1, K >= 32 with K % 32 == 0, 1 <= batch <= WQ4_MAX_BATCH.
 * Returns WQ4_OK, WQ4_ERR_INVALID (sizes, null, overlap), WQ4_ERR_ALIGN, or
 * WQ4_ERR_CUDA.  Deterministic: the same inputs give the same bits.
 * Launched with programmatic dependent launch: x is read and y written only
 * after the previous kernel in `stream` has completed, but the weight
 * stream may start while it finishes if that kernel lets its dependents
 * launch early (griddepcontrol.launch_dependents), so such a kernel must not
 * write W_packed or scales.
 */
int wq4_gemv(const uint32_t* W_packed, const uint16_t* scales, const uint16_t* x,
             uint16_t* y, int N, int K, int batch, void* stream);

/*
 * The same product for many activation rows (prefill-shaped: the tokens of a
 * prompt through one projection), on the tensor cores:
 *   Y[m][n] = fp16( sum_k x[m][k] * fp16((q(n,k) - 7) * scales[n][k/32]) )
 * for m < M, n < N, sums in fp32.  Each dequantized weight is rounded to fp16
 * once (relative error <= 2^-11), so the accuracy contract above holds for
 * every scale with |s| <= 8188 (WQ4_MAX_FP16_SCALE; 8 * 8188 = 65504, the
 * fp16 maximum).  A larger scale makes some (q - 7) s overflow fp16: the call
 * still runs, sets bit 6 of the device status word (wq4_device_status) and
 * the outputs of those rows are not valid; wq4_gemv has no such limit.
 *   W_packed, scales : as wq4_gemv, both 16-byte aligned.
 *   x : fp16 bits [M][K], 16-byte aligned.   y : fp16 bits [M][N], 16-byte
 *       aligned, must not overlap x, W or scales.
 *   M >= 1 (any size), N >= 1 with N % 8 == 0, K % 256 == 0 (other valid
 *   sizes return WQ4_ERR_UNSUPPORTED: use wq4_gemv for them).
 * Deterministic (no split K).  Returns WQ4_OK, WQ4_ERR_INVALID,
 * WQ4_ERR_UNSUPPORTED, WQ4_ERR_ALIGN or WQ4_ERR_CUDA.
 */
int wq4_gemm(const uint32_t* W_packed, const uint16_t* scales, const uint16_t* x,
             uint16_t* y, int N, int K, int M, void* stream);

/*
 * Test hook for the unpack step: runs the same in-register unpack the GEMV
 * uses and writes its results, so that they can be compared bit for bit.
 *   q_out : uint8 [N][K] codes 0..15 (may be NULL)
 *   w_out : fp32  [N][K] = (q - 7) * scale, exact in fp32 (may be NULL)
 * Same size and alignment rules as wq4_gemv (batch not used).
 */
int wq4_unpack_debug(const uint32_t* W_packed, const uint16_t* scales,
                     float* w_out, uint8_t* q_out, int N, int K, void* stream);

/*
 * Host-side packer of the weight format (the offline weight conversion of
 * Section 2.3): q_host uint8 [N][K] with values 0..15 -> W_host uint32
 * [N][K/8].  HOST pointers.  Returns WQ4_ERR_INVALID for a code above 15,
 * null pointers or bad sizes (K % 8 != 0).
 */
int wq4_pack_host(const uint8_t* q_host, uint32_t* W_host, int N, int K);

/*
 * Test hook: which kernel wq4_gemv takes at batch 1-2 with K % 256 == 0 and
 * 16-byte aligned scales, for every later call in this process.  0 (the
 * default) picks by size (the legacy-tensor-path kernel from 12 Mi weights
 * up, the CUDA-core kernel below), 1 always the legacy-tensor-path kernel,
 * 2 always the CUDA-core kernel.  Results agree within the tolerance; no
 * counterpart in the paper.  WQ4_ERR_INVALID for another value.
 */
int wq4_test_gemv_path(int path);

/* Static, human-readable text of a status code. */
const char* wq4_status_string(int status);

/*
 * Reads and clears the library's device status word on `stream` (this call
 * synchronizes the stream).  *flags_out receives the bits that were set:
 * bit 0 = an mbarrier wait of a weight pipeline gave up, bit 1 = a wait on
 * another CTA's activations gave up; wq4_attn.h calls add bit 3 = a sequence
 * length beyond its page table (clamped), bit 4 = a page id outside the pool
 * (zeros read in its place), bit 5 = an append with a bad position or page
 * id (nothing written); bit 6 = wq4_gemm met a scale beyond
 * WQ4_MAX_FP16_SCALE (its outputs are not valid).  Returns WQ4_ERR_TIMEOUT if
 * any bit was set, WQ4_OK otherwise, WQ4_ERR_CUDA on a CUDA failure.
 */
int wq4_device_status(void* stream, int* flags_out);

/* ------------------------------------------------------------------------ */
/* Per-token decode chain                                                     */
/* ------------------------------------------------------------------------ */

/* One packed projection: W uint32 [N][K/8], s fp16 [N][K/32] (device). */
typedef struct {
    const uint32_t* W;
    const uint16_t* s;
} wq4_mat;

/* One layer's four projections (shapes follow from the table below):
 *   qkv     : N = (n_q_heads + 2*n_kv_heads) * head_dim, K = hidden
 *   o       : N = hidden,  K = hidden
 *   gate_up : N = 2*ffn,   K = hidden (rows [0,ffn) gate, [ffn,2ffn) up)
 *   down    : N = hidden,  K = ffn                                          */
typedef struct {
    wq4_mat qkv, o, gate_up, down;
} wq4_layer;

/*
 * A decoder's weights and the caller-owned workspace of the chain.
 *   layers     : HOST array of num_layers entries holding device pointers.
 *   lm_head    : N = vocab, K = hidden.
 *   n_q_heads * head_dim must equal hidden (the query block of the QKV output
 *   is the stand-in attention output, see wq4_decode_chain).
 *   workspace  : device buffer of at least wq4_chain_workspace_bytes(table)
 *                bytes, 256-byte aligned, used only by this table's chain.
 *   hidden and ffn must be multiples of 256, vocab any >= 1, batch 1..32;
 *   batch 1-2 takes at most 128 layers (WQ4_ERR_UNSUPPORTED beyond).
 */
typedef struct {
    int num_layers, hidden, ffn, n_q_heads, n_kv_heads, head_dim, vocab, batch;
    float rms_eps;
    const wq4_layer* layers;
    wq4_mat lm_head;
    void* workspace;
    size_t workspace_bytes;
} wq4_layer_table;

/* Bytes of workspace the chain needs for this table (0 if the table is
 * invalid).  Host-only, no CUDA call. */
size_t wq4_chain_workspace_bytes(const wq4_layer_table* table);

/*
 * One decoded token through every projection of every layer and the LM head
 * (the per-token GPU work measured by Table 1, Section 3), as ONE persistent
 * kernel whose CTAs stream the weights through shared memory and pass the
 * activations between stages through flagged words in the workspace.
 * Layer l takes u (fp16 [batch][hidden]: x for l = 0, else the previous
 * layer's output), re-feeds it after RMS normalisation, and rounds every
 * stage output to fp16:
 *   v   = r(u) * u                     r(t) = 1/sqrt(mean(t^2) + rms_eps)
 *   qkv = r(u)  * W_qkv . u
 *   o   = r(a)  * W_o   . a            a = qkv[:, :hidden] (stands in for
 *   x1  = v + o                            attention, which is not in the chain)
 *   gu  = r(x1) * W_gu  . x1
 *   m   = silu(gu[:, :ffn]) * gu[:, ffn:]
 *   x2  = x1 + W_down . m              (the layer output, next layer's u)
 * then logits = r(xL) * W_lm . xL.  RMS normalisation has no learned gain and
 * enters every projection as a per-row factor (r(t) W.t = W.(r(t) t); Section
 * 2.3 "kernel fusion"); the normalised v is materialised only in the
 * residual stream.
 *   x      : fp16 [batch][hidden] device, 16-byte aligned
 *   logits : fp16 [batch][vocab]  device, 2-byte aligned
 * Batch 1-2 runs as the persistent kernel above (exact dequantization, any
 * fp16 scale).  Batch 3-32 runs as a CUDA graph, captured once per table, of
 * one tensor-core kernel per projection (dequantized fp16 weights
 * w = fp16((q - 7) s) times the batch's inputs, tcgen05 MMAs with fp32
 * accumulation, the chain's row factors, residual adds and SiLU fused into
 * each stage's epilogue); each call copies x into the workspace, replays the
 * graph and copies the logits out (all on `stream`).
 * The first call for a table (or after its contents changed) builds its plan:
 * at batch 1-2 it validates the table and uploads its pointer table into the
 * workspace (cudaMemcpyAsync on `stream`); at batch 3-32 it also scans every
 * scale (a table with a scale beyond WQ4_MAX_FP16_SCALE is rejected with
 * WQ4_ERR_UNSUPPORTED), synchronizes `stream`, and captures and instantiates
 * the CUDA graph (driver-side resources, no device memory of this library);
 * rebuilding a batch 3-32 plan also synchronizes `stream` before freeing the
 * old graph.  Later calls only launch.  Calls on one table must not overlap
 * on the GPU.
 * Returns WQ4_OK, WQ4_ERR_INVALID, WQ4_ERR_ALIGN, WQ4_ERR_UNSUPPORTED or
 * WQ4_ERR_CUDA (including a GPU that cannot co-schedule the persistent grid).
 */
int wq4_decode_chain(const wq4_layer_table* table, const uint16_t* x,
                     uint16_t* logits, void* stream);

/*
 * The same token with HOST buffers: copies x_host (pinned or pageable fp16
 * [batch][hidden]) into the workspace, runs wq4_decode_chain, copies the
 * logits back into logits_host (fp16 [batch][vocab]) and synchronizes
 * `stream` before returning.
 */
int wq4_decode_chain_host(const wq4_layer_table* table, const uint16_t* x_host,
                          uint16_t* logits_host, void* stream);

/*
 * Size of the device array wq4_decode_chain_noalloc uses as its workspace
 * (16 MiB: the 3B-shaped chain at batch 1-2, the 8B-shaped one at batch 1).
 */
#define WQ4_NOALLOC_SCRATCH_BYTES (16u << 20)

/*
 * wq4_decode_chain without a caller-allocated workspace.  The paper has no
 * counterpart: this is for callers that cannot call cudaMalloc -- a plug-in
 * inside a host framework that owns all device memory through its own pool
 * and permits no other allocation, or a latency-critical loop where
 * cudaMalloc's implicit device synchronization is not acceptable.
 *
 * The workspace is a fixed device array of WQ4_NOALLOC_SCRATCH_BYTES inside
 * this library: every GPU that loads the library holds it until the process
 * exits.  table->workspace and table->workspace_bytes are ignored; everything
 * else, x and logits are as for wq4_decode_chain.  The call allocates no
 * device memory (no cudaMalloc, cudaFree or allocating library routine).
 *   - The first call on a device looks up the array's device address
 *     (cudaGetSymbolAddress, with that device current); make that first call
 *     before any stream capture.
 *   - All calls on a device share the one array, which keeps the last call's
 *     contents; the first call for a table, or a call with a different table
 *     than the previous one, rebuilds the plan and clears the array's
 *     counters and flags again.  A rebuild enqueues copies on `stream`; at
 *     batch 3-32 (the tables that fit: the tiny and small shapes) it also
 *     scans the scales, synchronizes `stream` and captures and instantiates
 *     a CUDA graph (driver-side resources, but no device memory).  Make every
 *     call that switches tables outside stream capture: a rebuild requested
 *     while `stream` is capturing returns WQ4_ERR_UNSUPPORTED.
 *     Calls that overlap on the GPU race on the array: serialize them.
 *   - A table whose wq4_chain_workspace_bytes exceeds
 *     WQ4_NOALLOC_SCRATCH_BYTES is rejected with WQ4_ERR_UNSUPPORTED before
 *     anything is enqueued.
 */
int wq4_decode_chain_noalloc(const wq4_layer_table* table, const uint16_t* x,
                             uint16_t* logits, void* stream);

/*
 * Which kernel the cached plan of `table` runs (an inspection call, no
 * counterpart in the paper): 1 for the persistent chain kernel (batch 1-2),
 * 2 for the CUDA graph of tensor-core stage kernels (batch 3-32);
 * decode_step != 0 asks about the plan of wq4_decode_step, else of
 * wq4_decode_chain.  Returns WQ4_ERR_INVALID when no plan exists yet (the
 * first call builds it).
 */
int wq4_chain_path(const wq4_layer_table* table, int decode_step);

/* Releases the cached plan of `table` (host-side state only; the workspace
 * stays the caller's).  A batch 3-32 plan owns a CUDA graph: synchronize every
 * stream that ran the table before calling this.  Plans are cached by the
 * table's address and contents: release a table's plan before freeing any
 * buffer it names, or a later table at the same address with the same
 * pointers reuses the plan without re-initialising its workspace.  (The batch
 * 1-2 kernel takes the weight pointers in its launch parameters, so such a
 * reuse reads no pointer from the workspace.)  Returns WQ4_ERR_INVALID if no
 * plan exists. */
int wq4_chain_plan_destroy(const wq4_layer_table* table);

/*
 * Byte offsets into the workspace of the plain fp16 copies of one layer's
 * stage outputs, each [batch][len] row-major, for inspection after a call
 * (layer in [0, num_layers)); layer == num_layers gives the LM head's input
 * in x_in and 0 in the other fields.  q_rot, k_rot and attn are written only
 * by wq4_decode_step and lie beyond wq4_chain_workspace_bytes (inside
 * wq4_decode_step_workspace_bytes); they are 0 when the table's heads do not
 * allow the decode step.
 */
typedef struct {
    size_t x_in;     /* [batch][hidden]  v: layer input after RMS norm */
    size_t qkv;      /* [batch][n_qkv]   QKV projection              */
    size_t o;        /* [batch][hidden]  O projection                */
    size_t x_mid;    /* [batch][hidden]  x + o                        */
    size_t gate_up;  /* [batch][2*ffn]   gate_up projection           */
    size_t act;      /* [batch][ffn]     silu(gate) * up              */
    size_t down;     /* [batch][hidden]  down projection              */
    size_t x_out;    /* [batch][hidden]  x2: layer output (not normalised) */
    size_t q_rot;    /* [batch][hidden]  rotated queries (decode step)   */
    size_t k_rot;    /* [batch][n_kv_heads*head_dim] rotated keys (idem) */
    size_t attn;     /* [batch][hidden]  attention output = O input (idem) */
} wq4_chain_trace;

int wq4_chain_trace_offsets(const wq4_layer_table* table, int layer, wq4_chain_trace* out);

/*
 * Test hook of the bounded device waits (no counterpart in the paper: the
 * paper's kernels run as separate launches and never wait on one another).
 * Sets, for every later launch of the batch 1-2 chain kernel in this process
 * (wq4_decode_chain, _host, _noalloc; a CUDA graph that captured a launch
 * keeps the values of its capture):
 *   wait_limit_ns : how long one wait on another CTA's activations polls
 *                   before it gives up (1 .. 500,000,000; the default is
 *                   500,000,000 = 0.5 s).  The weight pipeline's mbarrier
 *                   waits keep the default.
 *   stall_stage   : -1 (default) for none, else the stage 4*layer + t
 *                   (t = 0 QKV, 1 O, 2 gate_up, 3 down; 4*n_layers = LM head)
 *                   whose input waits poll for an epoch that no CTA writes,
 *                   so that they run out.  Stage 0 reads x directly and has
 *                   no such wait.
 * After a stalled stage the kernel still finishes (its outputs are not
 * valid), every access stays within the workspace, and wq4_device_status
 * reports bit 1.  Returns WQ4_ERR_INVALID for a limit of 0 or above the
 * default, or a stage below -1.
 */
int wq4_test_chain_waits(uint64_t wait_limit_ns, int stall_stage);

#ifdef __cplusplus
}
#endif

#endif /* WQ4_H */
