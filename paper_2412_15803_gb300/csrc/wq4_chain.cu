// wq4_chain.cu -- one decoded token through every projection of every layer
// and the LM head, as one persistent kernel (the per-token GPU work whose
// throughput Table 1 of Section 3 reports).
//
// Structure (GB300-first; the paper's WebGPU engine launches one compiled
// kernel per operator, Section 2.3):
//  * One CTA per SM, co-resident (cooperative launch).  Each CTA owns a fixed
//    slice of the output words (two fp16 outputs each) of every stage (QKV, O,
//    gate_up, down per layer, then the LM head).
//  * A producer warp walks the CTA's slices of ALL stages in order and streams
//    their packed weights through a ring of shared-memory slots with 1-D bulk
//    copies (TMA) and mbarriers.  Weights do not depend on activations, so the
//    stream runs ahead across stage boundaries and HBM keeps working while the
//    consumers wait for the next activation vector.
//  * Each layer re-feeds its input after RMS normalisation.  Every CTA
//    computes the same factor in the same order (identical bits everywhere),
//    applies it as a row factor of its projection, and publishes its slice of
//    the normalised vector for the O stage's residual add.
//  * Work items are (superpair, K part): a superpair is two row pairs (two
//    output words, or gate_up's gate and up rows of one word; one row pair
//    for very long rows), and K is cut into q equal parts chosen per stage
//    so that the 15 consumer warps, taking items round-robin in ring order,
//    get nearly equal work.  An item is a run of units of 256 codes; per row
//    pair a unit is two mma.sync m16n8k16 on the legacy tensor path: A holds
//    exact fp16 (q - 7) of 16 (row, group) combinations (two rows x eight
//    groups of 32 codes), B holds the eight groups' activations as its eight
//    columns (loaded once for both pairs), and the group scales multiply the
//    diagonal of the fp32 result on the CUDA cores (no fp16 rounding of a
//    weight or a product).  After the stage, the parts of every word are
//    added in part order and the fused epilogue (RMS factor, residual add,
//    SiLU(gate) * up) publishes the words.
//  * Stage outputs travel between CTAs as 8-byte words {2 x fp16 data, 32-bit
//    token epoch} written with single 64-bit stores; a consumer polls the
//    words of its input until every epoch matches.  No grid-wide barrier and
//    no separate flag round trip: one L2 round trip per stage boundary.
//    Every poll is bounded in time.
//  * Plain fp16 copies of every stage output are written to the workspace for
//    inspection.
#include "wq4_device.cuh"
#include "wq4_items.cuh"
#include "wq4_host.h"
#include "wq4_tc_host.h"
#include "wq4.h"
#include "wq4_attn.h"

#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstring>
#include <atomic>
#include <map>
#include <type_traits>
#include <mutex>
#include <vector>

namespace wq4 {
namespace {

constexpr int kChainMaxSlots = 16;
// Chunk c of the ring lives in slot c % nslots and lands on full barrier
// c % nbars, nbars = (kFullBars / nslots) * nslots.  A parity wait only tells
// the wanted phase from the one before it, so a warp may wait on chunk c only
// once chunk c - nbars has landed; consumer warps skip the chunks without
// their items, and the plan keeps nslots + ceil(NW / items per slot) <= nbars
// for every stage, which bounds how far ahead of the oldest unconsumed chunk
// a warp can be (nslots - 1 + ceil(NW / items per slot) chunks).
constexpr int kFullBars = 48;
constexpr int kMaxChainBatch = 2;   // larger batches take the tensor-core graph path
// A ring slot is released after kSlotRelease arrivals: one per item consumed
// from it, plus (kSlotRelease - items) from the warp that consumed its first
// item.  Only warps that own items of a chunk touch its barriers.
constexpr uint32_t kSlotRelease = 1024;
// Shared-memory header: mbarriers (kFullBars full, kChainMaxSlots empty) |
// RMS partial sums | epoch | stage table | warp table | residual words of the
// CTA's words (O and down stages) | per-item partial row sums; then the
// staged input vector, then the weight ring.
constexpr int kHdrRed = 512;                 // float red[kMaxChainBatch][32]: per-warp sums of squares
static_assert(8 * (kFullBars + kChainMaxSlots) <= kHdrRed, "mbarriers overlap the header");
static_assert(kHdrRed + 4 * 2 * 32 <= 768, "RMS partial sums overlap the header");
constexpr int kHdrEpoch = 768;               // uint32 epoch, then int vw0, vw1 (the CTA's slice of v)
constexpr int kHdrInfo = 784;                // StageInfo info[5], one per stage type
constexpr int kHdrRes = 1152;                // uint32 res[kMaxResWords]: prefetched residual words
constexpr int kMaxResWords = 256;
constexpr int kHdrPart = kHdrRes + 4 * kMaxResWords;   // float4 part[superpair][K part][B]: row sums
constexpr int kMaxPart = 384;
constexpr int kChainHeader = kHdrPart + 16 * kMaxPart;
static_assert(kHdrPart % 16 == 0 && kChainHeader % 128 == 0, "header alignment");

// Consumer warps per CTA: with the producer warp, 16 warps (128 registers a
// thread).
constexpr int kChainWarps = 15;

enum StageType { kQKV = 0, kO = 1, kGU = 2, kDOWN = 3, kLM = 4 };

struct DevMat {
    const uint32_t* W;
    const uint16_t* s;
};

// Largest layer count of the persistent chain: its weight pointers travel in
// the launch parameters (a __grid_constant__ struct), not in the workspace, so
// no plan depends on device memory the caller could have freed or zeroed.
constexpr int kChainMaxLayers = 128;

struct ChainParams {
    int L, H, F, Nqkv, V;
    float eps;
    int q[5];            // K parts per superpair, per stage type (divides K / 256)
    int spw[5];          // words per superpair, per stage type (gate_up: 1)
    const uint16_t* x;   // [B][H] token input
    uint16_t* logits;    // [B][V]
    uint32_t* seq;       // token counter (workspace header)
    uint32_t* done;      // CTAs finished with this token
    uint32_t* abort;     // epoch of a token whose waits gave up (stops the others early)
    uint64_t* llA;       // [L][B][H/2]   query block of qkv (attention stand-in)
    uint64_t* llX1;      // [L][B][H/2]   x + o
    uint64_t* llM;       // [L][B][F/2]   silu(gate) * up
    uint64_t* llX;       // [L+1][B][H/2] layer outputs (index 0 unused)
    uint64_t* llV;       // [L][B][H/2]   RMS-normalised layer inputs (residual of O)
    // Every flagged vector is written twice (replica 1 at llX + rep.X etc., in
    // uint64 words); CTA c reads replica c & 1, which halves the number of
    // CTAs polling each line of a stage boundary.
    struct { uint32_t A, X1, M, X, V; } rep;
    uint16_t* pV;        // [L+1][B][H]   RMS-normalised layer inputs; [L] feeds the LM head
    uint16_t* pX2;       // [L][B][H]     layer outputs
    uint16_t* pQKV;      // [L][B][Nqkv]
    uint16_t* pO;        // [L][B][H]
    uint16_t* pX1;       // [L][B][H]
    uint16_t* pGU;       // [L][B][2F]
    uint16_t* pM;        // [L][B][F]
    uint16_t* pD;        // [L][B][H]
    int nslots;
    int nbars;           // full barriers: a multiple of nslots
    uint32_t slot_bytes;
    uint32_t x_bytes;
    uint32_t* err;
    uint64_t wait_ns;    // limit of a wait on flagged words (kWaitTimeoutNs unless a test sets it)
    int stall_stage;     // test hook: this stage waits for an epoch nobody writes (-1: none)
    DevMat mats[4 * kChainMaxLayers + 1];   // [4L + 1]: per layer qkv, o, gate_up, down; then lm_head
};
static_assert(sizeof(ChainParams) <= 32764, "kernel parameter space");

// ------------------------------------------------- decode step (attention) --
//
// With attention (wq4_decode_step) the QKV epilogue rotates q and k (rotary
// embedding, adjacent pairs, fp64 rotation of the fp16 outputs), appends the
// new k and v to the layer's paged cache and publishes them as flagged words;
// at the start of the O stage every CTA computes its splits of the decode
// attention (a (row, kv head, token range) each, fp32 online softmax over the
// cached tokens plus the new one), the last split of each (row, kv head) to
// arrive merges the partials and publishes the attention output, which the O
// stage stages in place of the query block.
constexpr int kAttnD = 128;          // head dimension
constexpr int kAttnMaxGroup = 8;     // query heads per kv head
constexpr int kAttnMaxSplits = 32;   // token ranges per (row, kv head)
constexpr int kAttnPart = kAttnD + 4;   // floats of one split partial: o[128], m, l, pad

struct KvLayer {
    uint16_t* k;          // [num_pages][Hkv][P][128]
    uint16_t* v;
    const int32_t* pt;    // [B][pt_stride]
    int pt_stride, num_pages;
};

struct ChainParamsA : ChainParams {
    int Hkv, G, P, S;              // kv heads, query heads per kv head, page size, splits per (row, kv head)
    float scale;                   // score scale
    const int32_t* positions;      // [B] place of the new token
    uint64_t* llK;                 // [L][B][Hkv 128 / 2] the new token's rotated keys (flagged)
    uint64_t* llVn;                // [L][B][Hkv 128 / 2] its values (flagged)
    uint64_t* llAt;                // [L][B][H / 2] attention output (flagged), two replicas
    uint32_t repAt;
    uint32_t rope_off;             // shared-memory byte offset of the rotation table and positions
    uint16_t* pQr;                 // [L][B][H] rotated queries
    uint16_t* pKr;                 // [L][B][Hkv 128] rotated keys
    uint16_t* pAt;                 // [L][B][H] attention output
    float* apart;                  // [L][B][Hkv][S][G][kAttnPart] split partials
    uint32_t* acnt;                // [L][B][Hkv] splits arrived
    double inv_freq[kAttnD / 2];   // theta^(-2i / 128)
    KvLayer kv[kChainMaxLayers];
};
static_assert(sizeof(ChainParamsA) <= 32764, "kernel parameter space");

// One stage: N output rows of K codes, `words` output words of rpw rows each
// (gate_up: gate rows 2w, 2w+1 and up rows F+2w, F+2w+1; the LM head's last
// word may hold one row).
struct Stage {
    int type, layer, N, K, words, rpw;
    const uint32_t* W;
    const uint16_t* s;
};

__device__ __forceinline__ Stage stage_at(const ChainParams& p, int st)
{
    Stage g;
    if (st == 4 * p.L) {
        g.type = kLM; g.layer = p.L; g.N = p.V; g.K = p.H; g.rpw = 2; g.words = (p.V + 1) / 2;
    } else {
        g.layer = st >> 2;
        g.type = st & 3;
        switch (g.type) {
            case kQKV: g.N = p.Nqkv; g.K = p.H; g.rpw = 2; g.words = p.Nqkv / 2; break;
            case kO: g.N = p.H; g.K = p.H; g.rpw = 2; g.words = p.H / 2; break;
            case kGU: g.N = 2 * p.F; g.K = p.H; g.rpw = 4; g.words = p.F / 2; break;
            default: g.N = p.H; g.K = p.F; g.rpw = 2; g.words = p.H / 2; break;
        }
    }
    g.W = p.mats[st].W;
    g.s = p.mats[st].s;
    return g;
}

// Byte layout of one chunk (words [wa, wb) of a stage) inside a slot: the
// chunk's rows (gate_up: its gate rows, then its up rows), then their scales.
struct ChunkLayout {
    int nrows;          // rows in the chunk (both halves for gate_up)
    int nh;             // rows per half (gate_up) / nrows otherwise
    uint32_t codes_bytes, scale_bytes;
};

__device__ __forceinline__ ChunkLayout chunk_layout(const Stage& g, int wa, int wb)
{
    ChunkLayout c;
    if (g.type == kGU) {
        c.nh = 2 * (wb - wa);
        c.nrows = 2 * c.nh;
    } else {
        const int r1 = min(2 * wb, g.N);
        c.nrows = r1 - 2 * wa;
        c.nh = c.nrows;
    }
    c.codes_bytes = static_cast<uint32_t>(c.nrows) * (g.K / 2);
    c.scale_bytes = static_cast<uint32_t>(c.nrows) * (g.K / 16);
    return c;
}

// What one CTA does in every stage of one type, computed once per launch:
// its words [w0, w0 + nwords) = superpairs [0, nsp), words per chunk (a
// multiple of the words per superpair, spw), the number of chunks and that
// number modulo the slot and barrier counts (flip: parity changes of the
// barrier ring beyond the wrap), units (256 codes) per superpair J, K parts q
// and units per part upp.  Items are (superpair i / q, part i % q).
struct StageInfo {
    int w0, nwords, wps, nchunks, nmod_slots, nmod_bars, flip, J, spw, q, upp, nsp;
};
static_assert(kHdrInfo + 5 * sizeof(StageInfo) <= kHdrRes, "stage table overlaps the header");

__device__ __forceinline__ void cta_words(int words, int* w0, int* w1)
{
    *w0 = static_cast<int>(static_cast<int64_t>(blockIdx.x) * words / gridDim.x);
    *w1 = static_cast<int>(static_cast<int64_t>(blockIdx.x + 1) * words / gridDim.x);
}

// Words per superpair (the plan's choice: 2, or 1 for large words; gate_up's
// word already holds two row pairs).
__device__ __forceinline__ int words_per_superpair(const ChainParams& p, const Stage& g)
{
    return p.spw[g.type];
}

// Words per ring slot: a whole number of superpairs (the plan's slot holds at
// least one).
__device__ __forceinline__ int words_per_slot(const ChainParams& p, const Stage& g)
{
    const uint32_t word_bytes = static_cast<uint32_t>(g.rpw) * (g.K / 2 + g.K / 16);
    const int spw = words_per_superpair(p, g);
    const int wps = static_cast<int>(p.slot_bytes / word_bytes) / spw * spw;
    return wps < spw ? spw : wps;
}

// A representative stage of each type (layer 0, or the LM head).
__device__ __forceinline__ int stage_of_type(const ChainParams& p, int t)
{
    return t == kLM ? 4 * p.L : t;
}




// ------------------------------------------------------- flagged words --

__device__ __forceinline__ void ll_store(uint64_t* addr, uint32_t data, uint32_t epoch)
{
    const uint64_t v = (static_cast<uint64_t>(epoch) << 32) | data;
    asm volatile("st.relaxed.gpu.global.b64 [%0], %1;" ::"l"(addr), "l"(v) : "memory");
}

// A flagged word into both replicas of its vector (replica 1 `rep` words on).
__device__ __forceinline__ void ll_store2(uint64_t* addr, uint32_t rep, uint32_t data, uint32_t epoch)
{
    ll_store(addr, data, epoch);
    ll_store(addr + rep, data, epoch);
}

__device__ __forceinline__ void ll_load2_raw(const uint64_t* addr, uint64_t& a, uint64_t& b)
{
    asm volatile("ld.relaxed.gpu.global.v2.b64 {%0, %1}, [%2];" : "=l"(a), "=l"(b) : "l"(addr) : "memory");
}

__device__ __forceinline__ uint64_t ll_load1_raw(const uint64_t* addr)
{
    uint64_t a;
    asm volatile("ld.relaxed.gpu.global.b64 %0, [%1];" : "=l"(a) : "l"(addr) : "memory");
    return a;
}

// A wait gives up after limit_ns, or at once when another CTA already gave
// up on this token (epoch); the first to give up records the token in *abort.
__device__ __forceinline__ bool gave_up(uint64_t t0, uint32_t epoch, uint32_t* abort, uint64_t limit_ns)
{
    if (*reinterpret_cast<const volatile uint32_t*>(abort) == epoch) return true;
    if (globaltimer_ns() - t0 > limit_ns) {
        atomicExch(abort, epoch);
        return true;
    }
    return false;
}

// Four consecutive flagged words (8 fp16 values) at a 32-byte aligned address;
// polls until all four carry `tag` (the token's epoch, or under the stall test
// hook an epoch that no CTA writes during the token).
__device__ __forceinline__ uint4 ll_load4(const uint64_t* addr, uint32_t tag, uint32_t epoch, uint32_t* err,
                                         uint32_t* abort, uint64_t limit_ns)
{
    uint64_t a, b, c, d;
    ll_load2_raw(addr, a, b);
    ll_load2_raw(addr + 2, c, d);
    if (static_cast<uint32_t>(a >> 32) != tag || static_cast<uint32_t>(b >> 32) != tag ||
        static_cast<uint32_t>(c >> 32) != tag || static_cast<uint32_t>(d >> 32) != tag) {
        const uint64_t t0 = globaltimer_ns();
        for (uint32_t it = 0;; ++it) {
            ll_load2_raw(addr, a, b);
            ll_load2_raw(addr + 2, c, d);
            if (static_cast<uint32_t>(a >> 32) == tag && static_cast<uint32_t>(b >> 32) == tag &&
                static_cast<uint32_t>(c >> 32) == tag && static_cast<uint32_t>(d >> 32) == tag)
                break;
            if ((it & 63) == 63 && gave_up(t0, epoch, abort, limit_ns)) {
                atomicOr(err, kErrFlagTimeout);
                break;
            }
        }
    }
    return make_uint4(static_cast<uint32_t>(a), static_cast<uint32_t>(b), static_cast<uint32_t>(c),
                      static_cast<uint32_t>(d));
}

__device__ __forceinline__ uint32_t ll_load(const uint64_t* addr, uint32_t tag, uint32_t epoch, uint32_t* err,
                                           uint32_t* abort, uint64_t limit_ns)
{
    uint64_t a = ll_load1_raw(addr);
    if (static_cast<uint32_t>(a >> 32) != tag) {
        const uint64_t t0 = globaltimer_ns();
        for (uint32_t it = 0;; ++it) {
            a = ll_load1_raw(addr);
            if (static_cast<uint32_t>(a >> 32) == tag) break;
            if ((it & 63) == 63 && gave_up(t0, epoch, abort, limit_ns)) {
                atomicOr(err, kErrFlagTimeout);
                break;
            }
        }
    }
    return static_cast<uint32_t>(a);
}

// fp16(a + b): the fp32 sum of two fp16 values rounded to fp16 equals the
// correctly rounded fp16 sum (fp32 carries more than 2 * 11 + 2 bits).
__device__ __forceinline__ uint16_t add_h(float a, float b) { return float_to_half_bits(a + b); }

__device__ __forceinline__ float sum8_sq(uint4 v)
{
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
    float s = 0.f;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const float a = lo_f(w[i]), b = hi_f(w[i]);
        s = fmaf(a, a, s);
        s = fmaf(b, b, s);
    }
    return s;
}


// Word w (activations 2w, 2w+1) of a pair-permuted row staged at xw (uint32).
__device__ __forceinline__ uint32_t permuted_word(const uint32_t* xw, int w)
{
    const int c = w >> 2, i = w & 3;
    const uint32_t* u = xw + 4 * c + ((i & 1) ? 2 : 0);
    return (i & 2) ? __byte_perm(u[0], u[1], 0x7632) : __byte_perm(u[0], u[1], 0x5410);
}

// ---------------------------------------------------------- the kernel --


// Fused epilogue of one word w for batch row b: v0..v3 are its row sums (rows
// 2w, 2w+1; gate_up: gate 2w, 2w+1 then up 2w, 2w+1; LM head: rows 2w, 2w+1);
// resw is the word's residual (O: the normalised layer input, down: x + o).
template <int B>
__device__ __forceinline__ void word_epilogue(const ChainParams& p, const Stage& g, int w, int b, float v0, float v1,
                                              float v2, float v3, float rf, uint32_t resw, uint32_t epoch)
{
    const int H = p.H, F = p.F, l = g.layer;
    const int n = 2 * w;
    if (g.type == kQKV) {
        const uint32_t wd = pack2(float_to_half_bits(rf * v0), float_to_half_bits(rf * v1));
        *reinterpret_cast<uint32_t*>(p.pQKV + (static_cast<size_t>(l) * B + b) * p.Nqkv + n) = wd;
        if (n < H) ll_store2(p.llA + (static_cast<size_t>(l) * B + b) * (H / 2) + w, p.rep.A, wd, epoch);
    } else if (g.type == kO) {
        const uint16_t o0 = float_to_half_bits(rf * v0);
        const uint16_t o1 = float_to_half_bits(rf * v1);
        const uint32_t x1 = pack2(add_h(lo_f(resw), half_bits_to_float(o0)), add_h(hi_f(resw), half_bits_to_float(o1)));
        const size_t off = (static_cast<size_t>(l) * B + b) * H + n;
        *reinterpret_cast<uint32_t*>(p.pO + off) = pack2(o0, o1);
        *reinterpret_cast<uint32_t*>(p.pX1 + off) = x1;
        ll_store2(p.llX1 + (static_cast<size_t>(l) * B + b) * (H / 2) + w, p.rep.X1, x1, epoch);
    } else if (g.type == kGU) {
        const uint16_t g0 = float_to_half_bits(rf * v0);
        const uint16_t g1 = float_to_half_bits(rf * v1);
        const uint16_t u0 = float_to_half_bits(rf * v2);
        const uint16_t u1 = float_to_half_bits(rf * v3);
        const float gf0 = half_bits_to_float(g0), gf1 = half_bits_to_float(g1);
        const uint16_t m0 = float_to_half_bits(gf0 / (1.f + expf(-gf0)) * half_bits_to_float(u0));
        const uint16_t m1 = float_to_half_bits(gf1 / (1.f + expf(-gf1)) * half_bits_to_float(u1));
        const size_t gu = (static_cast<size_t>(l) * B + b) * (2 * F);
        *reinterpret_cast<uint32_t*>(p.pGU + gu + n) = pack2(g0, g1);
        *reinterpret_cast<uint32_t*>(p.pGU + gu + F + n) = pack2(u0, u1);
        const uint32_t mw = pack2(m0, m1);
        *reinterpret_cast<uint32_t*>(p.pM + (static_cast<size_t>(l) * B + b) * F + n) = mw;
        ll_store2(p.llM + (static_cast<size_t>(l) * B + b) * (F / 2) + w, p.rep.M, mw, epoch);
    } else if (g.type == kDOWN) {
        const uint16_t d0 = float_to_half_bits(v0);
        const uint16_t d1 = float_to_half_bits(v1);
        const uint32_t x2 = pack2(add_h(lo_f(resw), half_bits_to_float(d0)), add_h(hi_f(resw), half_bits_to_float(d1)));
        *reinterpret_cast<uint32_t*>(p.pD + (static_cast<size_t>(l) * B + b) * H + n) = pack2(d0, d1);
        *reinterpret_cast<uint32_t*>(p.pX2 + (static_cast<size_t>(l) * B + b) * H + n) = x2;
        ll_store2(p.llX + (static_cast<size_t>(l + 1) * B + b) * (H / 2) + w, p.rep.X, x2, epoch);
    } else {
        uint16_t* out = p.logits + static_cast<size_t>(b) * p.V + n;
        out[0] = float_to_half_bits(rf * v0);
        if (n + 1 < p.V) out[1] = float_to_half_bits(rf * v1);
    }
}

// fp16 bits of v rounded once (round to nearest even) from fp64.
__device__ __forceinline__ uint16_t double_to_half_bits(double v)
{
    uint16_t h;
    asm("cvt.rn.f16.f64 %0, %1;" : "=h"(h) : "d"(v));
    return h;
}

// The new token's cache row of kv head `kh` (of Hkv, pages of P tokens) in
// `pool` for batch row b, or null when its position or page id is outside
// the page table.
__device__ __forceinline__ uint16_t* append_row(const KvLayer& kv, int P, int Hkv, uint16_t* pool, int b, int pos, int kh)
{
    if (pos < 0) return nullptr;
    const int pi = pos / P;
    if (pi >= kv.pt_stride) return nullptr;
    const int page = kv.pt[static_cast<size_t>(b) * kv.pt_stride + pi];
    if (page < 0 || page >= kv.num_pages) return nullptr;
    return pool + ((static_cast<size_t>(page) * Hkv + kh) * P + (pos - pi * P)) * kAttnD;
}

// QKV epilogue of the decode step for word w (rows n = 2w, 2w + 1) of batch
// row b: the plain fp16 output for the trace; q and k pairs rotated by the
// token's angle (rope: cos, sin of pos * theta^(-2i/128) for i = (n % 128) / 2),
// q published for the attention, k and v appended to the cache and published
// as the new token's key and value.
template <int B>
__device__ __forceinline__ void qkv_epilogue_attn(const ChainParamsA& p, int l, int w, int b, float v0, float v1,
                                                  float rf, uint32_t epoch, const double2* rope, const int* pos_sh)
{
    const int H = p.H, n = 2 * w, KD = p.Hkv * kAttnD;
    const uint16_t h0 = float_to_half_bits(rf * v0), h1 = float_to_half_bits(rf * v1);
    *reinterpret_cast<uint32_t*>(p.pQKV + (static_cast<size_t>(l) * B + b) * p.Nqkv + n) = pack2(h0, h1);
    const int pos = pos_sh[b];
    if (n < H + KD) {
        const double2 cs = rope[b * (kAttnD / 2) + ((n & (kAttnD - 1)) >> 1)];
        const double a = half_bits_to_float(h0), c = half_bits_to_float(h1);
        const uint32_t rw = pack2(double_to_half_bits(a * cs.x - c * cs.y), double_to_half_bits(a * cs.y + c * cs.x));
        if (n < H) {
            *reinterpret_cast<uint32_t*>(p.pQr + (static_cast<size_t>(l) * B + b) * H + n) = rw;
            ll_store2(p.llA + (static_cast<size_t>(l) * B + b) * (H / 2) + w, p.rep.A, rw, epoch);
        } else {
            const int kn = n - H;
            *reinterpret_cast<uint32_t*>(p.pKr + (static_cast<size_t>(l) * B + b) * KD + kn) = rw;
            ll_store(p.llK + (static_cast<size_t>(l) * B + b) * (KD / 2) + kn / 2, rw, epoch);
            uint16_t* row = append_row(p.kv[l], p.P, p.Hkv, p.kv[l].k, b, pos, kn / kAttnD);
            if (row) *reinterpret_cast<uint32_t*>(row + (kn & (kAttnD - 1))) = rw;
            else if ((kn & (kAttnD - 1)) == 0) atomicOr(p.err, kErrAppend);
        }
    } else {
        const int vn = n - H - KD;
        const uint32_t vw = pack2(h0, h1);
        ll_store(p.llVn + (static_cast<size_t>(l) * B + b) * (KD / 2) + vn / 2, vw, epoch);
        uint16_t* row = append_row(p.kv[l], p.P, p.Hkv, p.kv[l].v, b, pos, vn / kAttnD);
        if (row) *reinterpret_cast<uint32_t*>(row + (vn & (kAttnD - 1))) = vw;
    }
}

// The rotation table of the token: cos, sin of pos_b * theta^(-2i/128) in
// fp64 (a separate function: fp64 sincos needs registers the kernel's main
// loop should not pay for).
template <int B>
__device__ __noinline__ void rope_table(const ChainParamsA& p, double2* rope)
{
    for (int e = threadIdx.x; e < B * (kAttnD / 2); e += blockDim.x) {
        const int b = e / (kAttnD / 2), i = e - b * (kAttnD / 2);
        const int pos = __ldg(p.positions + b);
        double sn, cn;
        sincos(static_cast<double>(pos < 0 ? 0 : pos) * p.inv_freq[i], &sn, &cn);
        rope[e] = make_double2(cn, sn);
    }
}

// 2^x (ex2.approx: relative error ~2^-22; 2^-inf = 0).  The attention keeps
// its scores in the base-2 domain (scale * log2 e folded into the score
// scale), so one instruction replaces the range reduction of expf.
__device__ __forceinline__ float fast_exp2(float x)
{
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// acc + a.lo * b.lo + a.hi * b.hi for two fp16 pairs: products exact in fp32,
// fp32 adds (the mixed-precision fma of sm_100+).
__device__ __forceinline__ float fma_h2(float acc, uint32_t a, uint32_t b)
{
    asm("{\n\t.reg .f16 a0, a1, b0, b1;\n\t"
        "mov.b32 {a0, a1}, %1;\n\t"
        "mov.b32 {b0, b1}, %2;\n\t"
        "fma.rn.f32.f16 %0, a0, b0, %0;\n\t"
        "fma.rn.f32.f16 %0, a1, b1, %0;\n\t}"
        : "+f"(acc)
        : "r"(a), "r"(b));
    return acc;
}

// Sum over the 32 lanes, every lane gets it.
__device__ __forceinline__ float warp_allsum(float v)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// The decode attention of layer l, run by the consumer warps of every CTA at
// the start of the O stage.  Row b's T = positions[b] + 1 tokens are cut into
// S_b = min(S, ceil(T / kAttnSplitTokens)) equal ranges; unit u = blockIdx.x
// + k * gridDim.x is (row b, kv head h, range c), ranges c >= S_b are empty.
// The unit's warps take U consecutive tokens at a time (lane: dimensions
// 4 lane .. 4 lane + 3; the range's page ids are staged in shared memory
// first), keeping a running maximum, sum and weighted value sum per query
// head of the group; the warps are combined in shared memory in warp order
// (one head at a time).  With one range the unit publishes a = o / l
// itself; otherwise it stores its (o, m, l) and the last range of (b, h) to
// arrive merges all S_b of them in range order and publishes a.
// Shared memory: xs area = qs[G][128] | wp[NW][kAttnPart]; header area from
// kHdrRes (res and part are free until the O stage's staging) = acc[G][kAttnPart] |
// pages[kAttnPageWindow].
constexpr int kAttnSplitTokens = 128;
constexpr int kAttnPageWindow = 256;
static_assert(kHdrRes + 4 * (kAttnMaxGroup * kAttnPart + kAttnPageWindow + kAttnD) <= kChainHeader,
              "attention scratch overlaps the staged input");

template <int B, int NW, int G>
__device__ __forceinline__ void attention_phase(const ChainParamsA& p, int l, uint32_t epoch, float* scratch, const int* pos_sh,
                                             int* flag_sh, uint8_t* smem)
{
    constexpr int kConsumers = NW * 32;
    constexpr int kBlk = 16;                   // tokens of a warp's block: one per lane pair
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int H = p.H, Hkv = p.Hkv, S = p.S, KD = Hkv * kAttnD, P = p.P;
    const float scale = p.scale * 1.4426950408889634f;   // base-2 scores
    // the layer's cache and the outputs in registers (the parameter block is
    // reached through a generic pointer here)
    const KvLayer kv = p.kv[l];
    uint16_t* const pAt = p.pAt;
    uint64_t* const llAt = p.llAt;
    const uint32_t repAt = p.repAt;
    float* const apart = p.apart;
    uint32_t* const acnt = p.acnt;
    uint32_t* const err = p.err;
    uint32_t* qh = reinterpret_cast<uint32_t*>(scratch);                        // [G][64] fp16 pairs of q
    float* wp = scratch + G * kAttnD;
    float* acc = reinterpret_cast<float*>(smem + kHdrRes);                       // [G][kAttnPart]
    int* pages = reinterpret_cast<int*>(smem + kHdrRes) + G * kAttnPart;          // [kAttnPageWindow]
    uint32_t* newkv = reinterpret_cast<uint32_t*>(pages + kAttnPageWindow);      // [2][64] the new key, value words
    const int nunits = B * Hkv * S;
    const uint64_t* qsrc = p.llA + ((blockIdx.x & 1) ? p.rep.A : 0u) + static_cast<size_t>(l) * B * (H / 2);
    for (int u = blockIdx.x; u < nunits; u += gridDim.x) {
        const int b = u / (Hkv * S);
        const int rr = u - b * (Hkv * S);
        const int h = rr / S, c = rr - h * S;
        const int pos = pos_sh[b];
        int T = pos + 1;                                        // 0 for an invalid position
        const int cap = kv.pt_stride * P;
        if (T > cap) {
            T = cap;
            if (threadIdx.x == 0 && c == 0) atomicOr(err, kErrSeqLen);
        }
        int Sb = (T + kAttnSplitTokens - 1) / kAttnSplitTokens;
        Sb = Sb < 1 ? 1 : (Sb > S ? S : Sb);
        if (c >= Sb) continue;                                  // uniform over the CTA
        const int t0 = static_cast<int>(static_cast<int64_t>(c) * T / Sb);
        const int t1 = static_cast<int>(static_cast<int64_t>(c + 1) * T / Sb);
        named_barrier_sync(1, kConsumers);                      // scratch free
        // the group's queries and, in the range holding the new token, its key
        // and value words: all polled at once
        const bool has_new = pos >= t0 && pos < t1;
        for (int e = threadIdx.x; e < G * (kAttnD / 2) + (has_new ? kAttnD : 0); e += kConsumers) {
            if (e < G * (kAttnD / 2)) {
                const int j = e / (kAttnD / 2), w = e - j * (kAttnD / 2);
                qh[j * (kAttnD / 2) + w] = ll_load(qsrc + static_cast<size_t>(b) * (H / 2) + (h * G + j) * (kAttnD / 2) + w,
                                                   epoch, epoch, p.err, p.abort, p.wait_ns);
            } else {
                const int i = e - G * (kAttnD / 2);             // 0..63 key words, 64..127 value words
                const uint64_t* src = (i < kAttnD / 2 ? p.llK : p.llVn) +
                                      (static_cast<size_t>(l) * B + b) * (KD / 2) + h * (kAttnD / 2) + (i & 63);
                newkv[i] = ll_load(src, epoch, epoch, p.err, p.abort, p.wait_ns);
            }
        }
        float m[G], ls[G], o[G][4];
#pragma unroll
        for (int j = 0; j < G; ++j) {
            m[j] = -INFINITY;
            ls[j] = 0.f;
            o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;
        }
        const int32_t* ptb = kv.pt + static_cast<size_t>(b) * kv.pt_stride;
        const int half = lane & 1, ti = lane >> 1;
        // the range in windows of kAttnPageWindow pages
        for (int wbeg = t0; wbeg < t1; wbeg += kAttnPageWindow * P - (wbeg % P)) {
            const int wp0 = wbeg / P;
            const int wend = min(t1, (wp0 + kAttnPageWindow) * P);
            const int npg = (wend - 1) / P - wp0 + 1;
            named_barrier_sync(1, kConsumers);                  // previous window's pages consumed; q written
            for (int i = threadIdx.x; i < npg; i += kConsumers) {
                const int pid = __ldg(ptb + wp0 + i);
                pages[i] = (pid >= 0 && pid < kv.num_pages) ? pid : -1;
                if (pid < 0 || pid >= kv.num_pages) atomicOr(err, kErrPageId);
            }
            named_barrier_sync(1, kConsumers);
            // blocks of 16 tokens per warp: lane pair (2 i, 2 i + 1) scores token
            // base + i over dimensions 64 half .. 64 half + 63 (fp16 products
            // exact in fp32, fp32 sums), then every lane accumulates the value
            // rows' dimensions 4 lane .. 4 lane + 3 with the broadcast weights
            for (int base = wbeg + warp * kBlk; base < wend; base += NW * kBlk) {
                const int t = base + ti;
                const bool valid = t < wend;
                float sp[G][2];
#pragma unroll
                for (int j = 0; j < G; ++j) sp[j][0] = sp[j][1] = 0.f;
                // the key half-row in two passes of four 16-byte chunks
                const uint4* krow = nullptr;
                const uint4* knew4 = nullptr;
                if (valid && t == pos) {
                    knew4 = reinterpret_cast<const uint4*>(newkv + 32 * half);
                } else if (valid) {
                    const int pi = t / P;
                    const int page = pages[pi - wp0];
                    if (page >= 0)
                        krow = reinterpret_cast<const uint4*>(
                            kv.k + ((static_cast<size_t>(page) * Hkv + h) * P + (t - pi * P)) * kAttnD + 64 * half);
                }
#pragma unroll
                for (int ps = 0; ps < 2; ++ps) {
                    uint4 kc[4];
#pragma unroll
                    for (int cc = 0; cc < 4; ++cc)
                        kc[cc] = knew4 ? knew4[4 * ps + cc] : (krow ? __ldg(krow + 4 * ps + cc) : make_uint4(0u, 0u, 0u, 0u));
#pragma unroll
                    for (int cc = 0; cc < 4; ++cc) {
#pragma unroll
                        for (int j = 0; j < G; ++j) {
                            // a shared-memory load per use: held in registers across the
                            // blocks, the group's queries would spill
                            const uint4 qc = lds_v4(smem_addr(qh + j * (kAttnD / 2) + 32 * half + 4 * (4 * ps + cc)));
                            float& a = sp[j][cc & 1];
                            a = fma_h2(a, qc.x, kc[cc].x);
                            a = fma_h2(a, qc.y, kc[cc].y);
                            a = fma_h2(a, qc.z, kc[cc].z);
                            a = fma_h2(a, qc.w, kc[cc].w);
                        }
                    }
                }
                float pw[G];
#pragma unroll
                for (int j = 0; j < G; ++j) {
                    float sc = sp[j][0] + sp[j][1];
                    sc = (sc + __shfl_xor_sync(0xffffffffu, sc, 1)) * scale;
                    if (!valid) sc = -INFINITY;
                    float bm = sc;                             // the block's maximum (token base is valid)
#pragma unroll
                    for (int off = 16; off > 1; off >>= 1) bm = fmaxf(bm, __shfl_xor_sync(0xffffffffu, bm, off));
                    const float mn = fmaxf(m[j], bm);
                    const float corr = fast_exp2(m[j] - mn);
                    pw[j] = valid ? fast_exp2(sc - mn) : 0.f;
                    float bs = half ? 0.f : pw[j];             // each token once
#pragma unroll
                    for (int off = 16; off > 0; off >>= 1) bs += __shfl_xor_sync(0xffffffffu, bs, off);
                    ls[j] = fmaf(ls[j], corr, bs);
                    o[j][0] *= corr;
                    o[j][1] *= corr;
                    o[j][2] *= corr;
                    o[j][3] *= corr;
                    m[j] = mn;
                }
                const int nb = min(kBlk, wend - base);
                // every value row of the block in flight at once, then the sums
                uint2 vv[kBlk];
#pragma unroll
                for (int i = 0; i < kBlk; ++i) {
                    const int tt = base + i;
                    vv[i] = make_uint2(0u, 0u);
                    if (i < nb) {
                        if (tt == pos) {
                            vv[i] = make_uint2(newkv[64 + 2 * lane], newkv[64 + 2 * lane + 1]);
                        } else {
                            const int pi = tt / P;
                            const int page = pages[pi - wp0];
                            if (page >= 0)
                                vv[i] = __ldg(reinterpret_cast<const uint2*>(
                                                  kv.v + ((static_cast<size_t>(page) * Hkv + h) * P + (tt - pi * P)) * kAttnD) +
                                              lane);
                        }
                    }
                }
#pragma unroll
                for (int i = 0; i < kBlk; ++i) {
                    const float w0 = lo_f(vv[i].x), w1 = hi_f(vv[i].x), w2 = lo_f(vv[i].y), w3 = hi_f(vv[i].y);
#pragma unroll
                    for (int j = 0; j < G; ++j) {
                        const float pi_ = __shfl_sync(0xffffffffu, pw[j], 2 * i);   // 0 past the window's end
                        o[j][0] = fmaf(pi_, w0, o[j][0]);
                        o[j][1] = fmaf(pi_, w1, o[j][1]);
                        o[j][2] = fmaf(pi_, w2, o[j][2]);
                        o[j][3] = fmaf(pi_, w3, o[j][3]);
                    }
                }
            }
        }
        // combine the warps in warp order, one query head at a time, into acc
#pragma unroll
        for (int j = 0; j < G; ++j) {
            float* mine = wp + warp * kAttnPart;
            reinterpret_cast<float4*>(mine)[lane] = make_float4(o[j][0], o[j][1], o[j][2], o[j][3]);
            if (lane == 0) {
                mine[kAttnD] = m[j];
                mine[kAttnD + 1] = ls[j];
            }
            named_barrier_sync(1, kConsumers);
            if (threadIdx.x < kAttnD) {
                const int d = threadIdx.x;
                float M = -INFINITY;
#pragma unroll
                for (int w = 0; w < NW; ++w) M = fmaxf(M, wp[w * kAttnPart + kAttnD]);
                float Ls = 0.f, Od = 0.f;
                if (M != -INFINITY) {
#pragma unroll
                    for (int w = 0; w < NW; ++w) {
                        const float f = fast_exp2(wp[w * kAttnPart + kAttnD] - M);   // 0 for a warp without tokens
                        Ls = fmaf(f, wp[w * kAttnPart + kAttnD + 1], Ls);
                        Od = fmaf(f, wp[w * kAttnPart + d], Od);
                    }
                }
                acc[j * kAttnPart + d] = Od;
                if (d == 0) {
                    acc[j * kAttnPart + kAttnD] = M;
                    acc[j * kAttnPart + kAttnD + 1] = Ls;
                }
            }
            named_barrier_sync(1, kConsumers);
        }
        if (Sb == 1) {
            // one range: this unit's result is the attention output
            for (int e = threadIdx.x; e < G * (kAttnD / 2); e += kConsumers) {
                const int j = e / (kAttnD / 2), w = e - j * (kAttnD / 2);
                const float Ls = acc[j * kAttnPart + kAttnD + 1];
                const float a0 = Ls > 0.f ? acc[j * kAttnPart + 2 * w] / Ls : 0.f;
                const float a1 = Ls > 0.f ? acc[j * kAttnPart + 2 * w + 1] / Ls : 0.f;
                const uint32_t aw = pack2(float_to_half_bits(a0), float_to_half_bits(a1));
                const int n = (h * G + j) * kAttnD + 2 * w;
                *reinterpret_cast<uint32_t*>(pAt + (static_cast<size_t>(l) * B + b) * H + n) = aw;
                ll_store2(llAt + (static_cast<size_t>(l) * B + b) * (H / 2) + n / 2, repAt, aw, epoch);
            }
            continue;                                           // the next unit starts with a barrier
        }
        // store the range's partial, then arrive
        float* dst = apart + ((((static_cast<size_t>(l) * B + b) * Hkv + h) * S + c) * G) * kAttnPart;
        for (int e = threadIdx.x; e < G * (kAttnD + 2); e += kConsumers) {
            const int j = e / (kAttnD + 2), d = e - j * (kAttnD + 2);
            dst[j * kAttnPart + d] = acc[j * kAttnPart + d];
        }
        __threadfence();
        named_barrier_sync(1, kConsumers);
        if (threadIdx.x == 0) {
            const uint32_t prev = atomicAdd(acnt + (static_cast<size_t>(l) * B + b) * Hkv + h, 1u);
            *flag_sh = (prev == static_cast<uint32_t>(Sb - 1)) ? 1 : 0;
            __threadfence();
        }
        named_barrier_sync(1, kConsumers);
        if (*flag_sh) {
            // every range of (b, h) is in: merge them in range order; the ranges'
            // (m, l) first (all loads in flight), then per thread a pair of
            // dimensions of a head with its Sb loads in flight
            const float* src = apart + (((static_cast<size_t>(l) * B + b) * Hkv + h) * S) * G * kAttnPart;
            float2* ml = reinterpret_cast<float2*>(wp);              // [Sb][G]
            for (int e = threadIdx.x; e < Sb * G; e += kConsumers)
                ml[e] = __ldcg(reinterpret_cast<const float2*>(src + e * kAttnPart + kAttnD));
            named_barrier_sync(1, kConsumers);
            for (int e = threadIdx.x; e < G * (kAttnD / 2); e += kConsumers) {
                const int j = e / (kAttnD / 2), w = e - j * (kAttnD / 2);
                float M = -INFINITY;
                for (int cc = 0; cc < Sb; ++cc) M = fmaxf(M, ml[cc * G + j].x);
                float Ls = 0.f, O0 = 0.f, O1 = 0.f;
                if (M != -INFINITY) {
                    constexpr int kBatch = 16;                  // loads in flight per thread
                    for (int c0 = 0; c0 < Sb; c0 += kBatch) {
                        float2 ov[kBatch];
#pragma unroll
                        for (int i = 0; i < kBatch; ++i)
                            ov[i] = (c0 + i < Sb)
                                        ? __ldcg(reinterpret_cast<const float2*>(src + ((c0 + i) * G + j) * kAttnPart) + w)
                                        : make_float2(0.f, 0.f);
#pragma unroll
                        for (int i = 0; i < kBatch; ++i) {
                            if (c0 + i >= Sb) break;
                            const float2 mlc = ml[(c0 + i) * G + j];
                            const float f = fast_exp2(mlc.x - M);
                            Ls = fmaf(f, mlc.y, Ls);
                            O0 = fmaf(f, ov[i].x, O0);
                            O1 = fmaf(f, ov[i].y, O1);
                        }
                    }
                }
                const float a0 = Ls > 0.f ? O0 / Ls : 0.f, a1 = Ls > 0.f ? O1 / Ls : 0.f;
                const uint32_t aw = pack2(float_to_half_bits(a0), float_to_half_bits(a1));
                const int n = (h * G + j) * kAttnD + 2 * w;
                *reinterpret_cast<uint32_t*>(pAt + (static_cast<size_t>(l) * B + b) * H + n) = aw;
                ll_store2(llAt + (static_cast<size_t>(l) * B + b) * (H / 2) + n / 2, repAt, aw, epoch);
            }
            if (threadIdx.x == 0) acnt[(static_cast<size_t>(l) * B + b) * Hkv + h] = 0u;   // for the next token
        }
    }
    named_barrier_sync(1, kConsumers);                          // scratch free for the staging
}

template <int B, int NW>
__device__ __forceinline__ void attention_dispatch(const ChainParamsA& p, int l, uint32_t epoch, float* scratch,
                                                   const int* pos_sh, int* flag_sh, uint8_t* smem)
{
    switch (p.G) {
        case 1: attention_phase<B, NW, 1>(p, l, epoch, scratch, pos_sh, flag_sh, smem); break;
        case 2: attention_phase<B, NW, 2>(p, l, epoch, scratch, pos_sh, flag_sh, smem); break;
        case 3: attention_phase<B, NW, 3>(p, l, epoch, scratch, pos_sh, flag_sh, smem); break;
        case 4: attention_phase<B, NW, 4>(p, l, epoch, scratch, pos_sh, flag_sh, smem); break;
        case 5: attention_phase<B, NW, 5>(p, l, epoch, scratch, pos_sh, flag_sh, smem); break;
        case 6: attention_phase<B, NW, 6>(p, l, epoch, scratch, pos_sh, flag_sh, smem); break;
        case 7: attention_phase<B, NW, 7>(p, l, epoch, scratch, pos_sh, flag_sh, smem); break;
        default: attention_phase<B, NW, 8>(p, l, epoch, scratch, pos_sh, flag_sh, smem); break;
    }
}

template <int B, int NW, bool ATT>
__global__ void __launch_bounds__((NW + 1) * 32, 1)
    chain_kernel(const __grid_constant__ typename std::conditional<ATT, ChainParamsA, ChainParams>::type p)
{
    extern __shared__ __align__(1024) uint8_t smem[];
    uint64_t* full = reinterpret_cast<uint64_t*>(smem);
    uint64_t* empty = full + kFullBars;
    float* red = reinterpret_cast<float*>(smem + kHdrRed);          // [kMaxChainBatch][32]
    uint32_t* epoch_sh = reinterpret_cast<uint32_t*>(smem + kHdrEpoch);
    StageInfo* info = reinterpret_cast<StageInfo*>(smem + kHdrInfo);
    uint32_t* res = reinterpret_cast<uint32_t*>(smem + kHdrRes);    // [B][words of the CTA]
    float4* part = reinterpret_cast<float4*>(smem + kHdrPart);      // [word][part][B]
    uint4* xs = reinterpret_cast<uint4*>(smem + kChainHeader);       // [B][K / 8], pair-permuted
    uint8_t* slots = smem + kChainHeader + p.x_bytes;
    constexpr int kConsumers = NW * 32;
    constexpr int kPoll = 3;     // input chunks a thread has in flight at once

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nstages = 4 * p.L + 1;

    if (threadIdx.x == 0) {
        for (int i = 0; i < p.nbars; ++i) mbar_init(&full[i], 1);
        for (int i = 0; i < p.nslots; ++i) mbar_init(&empty[i], kSlotRelease);
        mbar_fence_init();
        uint32_t s;
        asm volatile("ld.relaxed.gpu.global.b32 %0, [%1];" : "=r"(s) : "l"(p.seq) : "memory");
        *epoch_sh = s + 1u;
        // the CTA's slice of the normalised input v that it publishes
        const int nw = p.H / 2;
        epoch_sh[1] = static_cast<int>(static_cast<int64_t>(blockIdx.x) * nw / gridDim.x);
        epoch_sh[2] = static_cast<int>(static_cast<int64_t>(blockIdx.x + 1) * nw / gridDim.x);
    }
    if (threadIdx.x < kMaxChainBatch * 32) red[threadIdx.x] = 0.f;   // warps >= NW stay zero
    // decode step: the rotation table (cos, sin of pos * theta^(-2i/128) per
    // row, fp64) and the rows' positions (-1 for an invalid one), after the
    // ring; their addresses are recomputed where used (no registers held)
    constexpr uint32_t kPosOff = B * (kAttnD / 2) * sizeof(double2);
    if constexpr (ATT) {
        rope_table<B>(p, reinterpret_cast<double2*>(smem + p.rope_off));
        int* pos_sh = reinterpret_cast<int*>(smem + p.rope_off + kPosOff);
        if (threadIdx.x < B) {
            const int pos = __ldg(p.positions + threadIdx.x);
            pos_sh[threadIdx.x] = pos < 0 ? -1 : pos;
        }
    }
    if (threadIdx.x >= 32 && threadIdx.x < 32 + 5) {
        const int t = threadIdx.x - 32;
        const Stage g = stage_at(p, stage_of_type(p, t));
        StageInfo in;
        int w0, w1;
        cta_words(g.words, &w0, &w1);
        in.w0 = w0;
        in.nwords = w1 - w0;
        in.wps = words_per_slot(p, g);
        in.nchunks = (in.nwords + in.wps - 1) / in.wps;
        in.nmod_slots = in.nchunks % p.nslots;
        in.nmod_bars = in.nchunks % p.nbars;
        in.flip = (in.nchunks / p.nbars) & 1;
        in.J = g.K >> 8;
        in.spw = words_per_superpair(p, g);
        in.q = p.q[t];
        in.upp = in.J / in.q;
        in.nsp = (in.nwords + in.spw - 1) / in.spw;
        info[t] = in;
    }
    __syncthreads();
    const uint32_t epoch = *epoch_sh;

    if (warp == NW) {
        // ------------------------------------------------ producer warp
        if (lane == 0) {
            const uint64_t pol = l2_policy_evict_first();
            int ord = 0;                // ring ordinal of the next chunk
            int slot = 0, round = 0;    // its slot and the slot's use count
            int fbi = 0;                // its full barrier
            for (int st = 0; st < nstages; ++st) {
                const Stage g = stage_at(p, st);
                const StageInfo in = info[g.type];
                const int w0 = in.w0, w1 = in.w0 + in.nwords, wps = in.wps;
                const int wpr = g.K >> 3, gpr = g.K >> 5;
                for (int wa = w0; wa < w1; wa += wps, ++ord) {
                    const int wb = min(w1, wa + wps);
                    if (round > 0) mbar_wait(&empty[slot], (round - 1) & 1, p.err);
                    const ChunkLayout c = chunk_layout(g, wa, wb);
                    uint8_t* dst = slots + static_cast<size_t>(slot) * p.slot_bytes;
                    uint64_t* fb = &full[fbi];
                    if (++slot == p.nslots) {
                        slot = 0;
                        ++round;
                    }
                    if (++fbi == p.nbars) fbi = 0;
                    mbar_arrive_expect_tx(fb, c.codes_bytes + c.scale_bytes);
                    if (g.type == kGU) {
                        const uint32_t hc = c.codes_bytes / 2, hs = c.scale_bytes / 2;
                        const size_t up = static_cast<size_t>(p.F);
                        bulk_g2s(dst, g.W + static_cast<size_t>(2 * wa) * wpr, hc, fb, pol);
                        bulk_g2s(dst + hc, g.W + (up + 2 * wa) * wpr, hc, fb, pol);
                        bulk_g2s(dst + c.codes_bytes, g.s + static_cast<size_t>(2 * wa) * gpr, hs, fb, pol);
                        bulk_g2s(dst + c.codes_bytes + hs, g.s + (up + 2 * wa) * gpr, hs, fb, pol);
                    } else {
                        bulk_g2s(dst, g.W + static_cast<size_t>(2 * wa) * wpr, c.codes_bytes, fb, pol);
                        bulk_g2s(dst + c.codes_bytes, g.s + static_cast<size_t>(2 * wa) * gpr, c.scale_bytes, fb, pol);
                    }
                }
            }
            // every chunk before the last nslots was consumed, so has landed:
            // wait for the rest before the CTA's shared memory goes away
            const int first = ord > p.nslots ? ord - p.nslots : 0;
            for (int o = first; o < ord; ++o) mbar_wait(&full[o % p.nbars], (o / p.nbars) & 1, p.err);
        }
    } else {
        // ------------------------------------------------ consumer warps
        const int H = p.H, F = p.F;
        int cord0 = 0;   // ring ordinal of the stage's first chunk
        for (int st = 0; st < nstages; ++st) {
            const Stage g = stage_at(p, st);
            const StageInfo& in = info[g.type];
            if constexpr (ATT) {
                // every CTA takes its splits of the layer's attention, words or not
                if (g.type == kO) {
                    int* pos_sh = reinterpret_cast<int*>(smem + p.rope_off + kPosOff);
                    attention_dispatch<B, NW>(p, g.layer, epoch, reinterpret_cast<float*>(xs), pos_sh,
                                              pos_sh + kMaxChainBatch, smem);
                }
            }
            if (in.nwords <= 0) continue;
            const int l = g.layer;
            const int K = g.K, cpr = K >> 3;
            const int nwd = in.nwords, w0 = in.w0;

            // -- stage the input vector (all consumer warps, pair-permuted),
            //    its RMS factor and the residual words of the CTA's words
            //    (the stall test hook makes one stage wait for an epoch that no
            //    producer writes: its waits run out, bounded)
            const uint32_t want = (st == p.stall_stage) ? (epoch + 0x80000000u) : epoch;
            named_barrier_sync(1, kConsumers);   // every warp is done with the previous xs, res and part
            {
                const uint64_t* ll = nullptr;
                const bool plain = (g.type == kQKV && l == 0);
                const bool r1 = (blockIdx.x & 1) != 0;   // this CTA's replica
                if (g.type == kQKV) ll = p.llX + (r1 ? p.rep.X : 0u) + static_cast<size_t>(l) * B * (H / 2);
                else if (g.type == kO) {
                    if constexpr (ATT) ll = p.llAt + (r1 ? p.repAt : 0u) + static_cast<size_t>(l) * B * (H / 2);
                    else ll = p.llA + (r1 ? p.rep.A : 0u) + static_cast<size_t>(l) * B * (H / 2);
                }
                else if (g.type == kGU) ll = p.llX1 + (r1 ? p.rep.X1 : 0u) + static_cast<size_t>(l) * B * (H / 2);
                else if (g.type == kDOWN) ll = p.llM + (r1 ? p.rep.M : 0u) + static_cast<size_t>(l) * B * (F / 2);
                else ll = p.llX + (r1 ? p.rep.X : 0u) + static_cast<size_t>(p.L) * B * (H / 2);
                const uint64_t* rl = nullptr;
                if (g.type == kO) rl = p.llV + (r1 ? p.rep.V : 0u) + static_cast<size_t>(l) * B * (H / 2);
                else if (g.type == kDOWN) rl = p.llX1 + (r1 ? p.rep.X1 : 0u) + static_cast<size_t>(l) * B * (H / 2);
                if (rl) {
#pragma unroll
                    for (int b = 0; b < B; ++b)
                        for (int k = threadIdx.x; k < nwd; k += kConsumers)
                            res[b * nwd + k] = ll_load(rl + static_cast<size_t>(b) * (H / 2) + w0 + k, want, epoch, p.err, p.abort, p.wait_ns);
                }
                float ss[B];
#pragma unroll
                for (int b = 0; b < B; ++b) ss[b] = 0.f;
                const int total = B * cpr;
                for (int ib = threadIdx.x; ib < total; ib += kPoll * kConsumers) {
                    uint4 v[kPoll];
                    if (plain) {
#pragma unroll
                        for (int k = 0; k < kPoll; ++k) {
                            const int i = ib + k * kConsumers;
                            if (i < total) v[k] = reinterpret_cast<const uint4*>(p.x)[i];
                        }
                    } else {
                        // issue every load first, then wait for the ones not yet published
                        uint64_t w[kPoll][4];
#pragma unroll
                        for (int k = 0; k < kPoll; ++k) {
                            const int i = ib + k * kConsumers;
                            if (i < total) {
                                const int b = i / cpr, c = i - b * cpr;
                                const uint64_t* a = ll + static_cast<size_t>(b) * (K / 2) + 4 * c;
                                ll_load2_raw(a, w[k][0], w[k][1]);
                                ll_load2_raw(a + 2, w[k][2], w[k][3]);
                            }
                        }
#pragma unroll
                        for (int k = 0; k < kPoll; ++k) {
                            const int i = ib + k * kConsumers;
                            if (i < total) {
                                bool ok = true;
#pragma unroll
                                for (int j = 0; j < 4; ++j) ok = ok && static_cast<uint32_t>(w[k][j] >> 32) == want;
                                if (ok) {
                                    v[k] = make_uint4(static_cast<uint32_t>(w[k][0]), static_cast<uint32_t>(w[k][1]),
                                                      static_cast<uint32_t>(w[k][2]), static_cast<uint32_t>(w[k][3]));
                                } else {
                                    const int b = i / cpr, c = i - b * cpr;
                                    v[k] = ll_load4(ll + static_cast<size_t>(b) * (K / 2) + 4 * c, want, epoch, p.err, p.abort, p.wait_ns);
                                }
                            }
                        }
                    }
#pragma unroll
                    for (int k = 0; k < kPoll; ++k) {
                        const int i = ib + k * kConsumers;
                        if (i < total) {
                            const int b = i / cpr;
                            xs[i] = pair_permute(v[k]);
#pragma unroll
                            for (int bb = 0; bb < B; ++bb)
                                if (bb == b) ss[bb] += sum8_sq(v[k]);
                        }
                    }
                }
#pragma unroll
                for (int b = 0; b < B; ++b) {
                    const float v = warp_sum(ss[b]);
                    if (lane == 0) red[b * 32 + warp] = v;
                }
            }
            named_barrier_sync(1, kConsumers);
            float rf[B];
#pragma unroll
            for (int b = 0; b < B; ++b) {
                // the same sum, in the same order, in every warp and every CTA
                const float4* r4 = reinterpret_cast<const float4*>(red + b * 32);
                float q4[8];
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    const float4 a = r4[i];
                    q4[i] = (a.x + a.y) + (a.z + a.w);
                }
                const float t = ((q4[0] + q4[1]) + (q4[2] + q4[3])) + ((q4[4] + q4[5]) + (q4[6] + q4[7]));
                rf[b] = (g.type == kDOWN) ? 1.f : rsqrtf(t * (1.f / static_cast<float>(K)) + p.eps);
            }
            // -- items (superpair, K part) round-robin over the warps, in ring
            //    order: item k goes to warp k % NW; a warp visits only the
            //    chunks that hold its items
            const int spw = in.spw, wps = in.wps, nch = in.nchunks, q = in.q, upp = in.upp;
            const int nsp = in.nsp, nitems = nsp * q;
            const int sps = spw - 1;                                        // log2 of words per superpair
            const int spc = wps >> sps;                                     // superpairs per chunk
            const int ips = spc * q;                                        // items per chunk
            const uint32_t xsa = smem_addr(xs);
            const FDiv fq = fdiv_make(q), fips = fdiv_make(ips), fns = fdiv_make(p.nslots), fnb = fdiv_make(p.nbars);
            int it = warp;
            if (it < nitems) {
                int k = fdiv(it, fips);                                     // chunk of the warp's first item
                int ia = k * ips, ib = min(nitems, ia + ips);
                int ord = cord0 + k;
                int slot = ord - fdiv(ord, fns) * p.nslots;
                const int qb = fdiv(ord, fnb);
                int bar = ord - qb * p.nbars;
                uint32_t par = static_cast<uint32_t>(qb) & 1u;
                while (it < nitems) {
                    while (it >= ib) {                      // next chunk
                        ++k;
                        ia += ips;
                        ib = min(nitems, ia + ips);
                        if (++slot == p.nslots) slot = 0;
                        if (++bar == p.nbars) {
                            bar = 0;
                            par ^= 1u;
                        }
                    }
                    mbar_wait(&full[bar], par, p.err);
                    const int kw0 = k * wps, kw1 = min(nwd, kw0 + wps);   // the chunk's words
                    const ChunkLayout c = chunk_layout(g, w0 + kw0, w0 + kw1);
                    const uint32_t cbase = smem_addr(slots + static_cast<size_t>(slot) * p.slot_bytes);
                    const uint32_t sbase = cbase + c.codes_bytes;
                    uint32_t arrivals = (it == ia) ? kSlotRelease - static_cast<uint32_t>(ib - ia) : 0u;
                    for (; it < ib; it += NW) {
                        ++arrivals;
                        const int sl = fdiv(it, fq);         // the item's superpair and K part
                        const int pt = it - sl * q;
                        const int jb = pt * upp, je = jb + upp;
                        const int sw0 = sl << sps;           // the superpair's first word (stage-relative)
                        const int wl = sw0 - kw0;            // ... within the chunk
                        uint32_t ra[2], rb[2];
                        if (g.type == kGU) {
                            // pairs (gate 2w + pr, up 2w + pr) of word w
#pragma unroll
                            for (int pr = 0; pr < 2; ++pr) {
                                ra[pr] = 2 * wl + pr;
                                rb[pr] = c.nh + 2 * wl + pr;
                            }
                        } else {
                            // pairs (2w, 2w + 1) of words w, w + 1 (one-word superpairs, or
                            // the second word missing at the end of the CTA's words: pair 0
                            // again, not computed or ignored; rows past N -- the LM head's
                            // last -- read row 2w again, ignored)
#pragma unroll
                            for (int pr = 0; pr < 2; ++pr) {
                                const int wr = (sw0 + pr < nwd) ? wl + pr : wl;
                                ra[pr] = 2 * wr;
                                rb[pr] = (2 * (w0 + kw0 + wr) + 1 < g.N) ? 2 * wr + 1 : 2 * wr;
                            }
                        }
                        uint32_t ca[2], cb2[2], sa[2], sb2[2];
#pragma unroll
                        for (int pr = 0; pr < 2; ++pr) {
                            ca[pr] = cbase + ra[pr] * (K / 2);
                            cb2[pr] = cbase + rb[pr] * (K / 2);
                            sa[pr] = sbase + ra[pr] * (K / 16);
                            sb2[pr] = sbase + rb[pr] * (K / 16);
                        }
                        float acc[2][B];
#pragma unroll
                        for (int pr = 0; pr < 2; ++pr)
#pragma unroll
                            for (int b = 0; b < B; ++b) acc[pr][b] = 0.f;
                        const bool two = g.type == kGU || spw == 2;
                        if (two) {
                            item_units<B, 2>(ca, cb2, sa, sb2, xsa, cpr, jb, je, acc);
                        } else {
                            const uint32_t ca1[1] = {ca[0]}, cb1[1] = {cb2[0]}, sa1[1] = {sa[0]}, sb1[1] = {sb2[0]};
                            float (&acc1)[1][B] = *reinterpret_cast<float (*)[1][B]>(&acc[0]);
                            item_units<B, 1>(ca1, cb1, sa1, sb1, xsa, cpr, jb, je, acc1);
                        }
#pragma unroll
                        for (int pr = 0; pr < 2; ++pr)
#pragma unroll
                            for (int b = 0; b < B; ++b) acc[pr][b] = pair_reduce(acc[pr][b]);
                        // this item's part of the superpair's row sums: (pair 0 row a,
                        // pair 0 row b, pair 1 row a, pair 1 row b); lane 0 holds the
                        // a rows, lane 16 the b rows
                        if (g.type == kLM) {
                            // whole superpairs (one part): lane 0 writes rows 2w and
                            // 2w + 2, lane 16 rows 2w + 1 and 2w + 3 of words w, w + 1
                            const int n0 = 2 * (w0 + sw0) + (lane == 16 ? 1 : 0);
#pragma unroll
                            for (int b = 0; b < B; ++b) {
                                uint16_t* out = p.logits + static_cast<size_t>(b) * p.V;
                                if (lane == 0 || lane == 16) {
                                    if (n0 < p.V) out[n0] = float_to_half_bits(rf[b] * acc[0][b]);
                                    if (spw == 2 && sw0 + 1 < nwd && n0 + 2 < p.V)
                                        out[n0 + 2] = float_to_half_bits(rf[b] * acc[1][b]);
                                }
                            }
                        } else {
                            float* pf = reinterpret_cast<float*>(part + (sl * q + pt) * B);
#pragma unroll
                            for (int b = 0; b < B; ++b) {
                                if (lane == 0) { pf[4 * b + 0] = acc[0][b]; pf[4 * b + 2] = acc[1][b]; }
                                if (lane == 16) { pf[4 * b + 1] = acc[0][b]; pf[4 * b + 3] = acc[1][b]; }
                            }
                        }
                    }
                    __syncwarp();
                    if (lane == 0) mbar_arrive_count(&empty[slot], arrivals);
                }
            }
            if (g.type == kQKV || g.type == kLM) {
                // the normalised layer input v = fp16(r * u) is kept for the
                // residual stream (and the trace): every CTA publishes its
                // slice of it; the projections below use r as a row factor
                const int vw0 = static_cast<int>(epoch_sh[1]), vw1 = static_cast<int>(epoch_sh[2]);
                const uint32_t* xw = reinterpret_cast<const uint32_t*>(xs);
#pragma unroll
                for (int b = 0; b < B; ++b) {
                    for (int w = vw0 + threadIdx.x; w < vw1; w += kConsumers) {
                        const uint32_t u = permuted_word(xw + 4 * b * cpr, w);
                        const uint32_t v = pack2(float_to_half_bits(rf[b] * lo_f(u)), float_to_half_bits(rf[b] * hi_f(u)));
                        reinterpret_cast<uint32_t*>(p.pV + (static_cast<size_t>(l) * B + b) * H)[w] = v;
                        if (g.type == kQKV) ll_store2(p.llV + (static_cast<size_t>(l) * B + b) * (H / 2) + w, p.rep.V, v, epoch);
                    }
                }
            }

            // -- every part of every word is in: add the parts in part order and
            //    publish the words, one thread per (superpair, batch row) on the
            //    first warps (spreading the entries over all warps, one lane
            //    each, measured 0.2 ms a token slower)
            if (g.type != kLM) named_barrier_sync(1, kConsumers);
            for (int e = threadIdx.x; g.type != kLM && e < nsp * B; e += kConsumers) {
                const int sl = e / B, b = e - sl * B;
                const float4* pp = part + sl * q * B + b;
                float4 sum = pp[0];
                for (int r = 1; r < q; ++r) {
                    const float4 t4 = pp[r * B];
                    sum.x += t4.x; sum.y += t4.y; sum.z += t4.z; sum.w += t4.w;
                }
                const int wc = sl << sps;                     // first word (stage-relative)
#pragma unroll
                for (int bb = 0; bb < B; ++bb) {
                    if (bb != b) continue;
                    if constexpr (ATT) {
                        if (g.type == kQKV) {
                            const double2* rope = reinterpret_cast<const double2*>(smem + p.rope_off);
                            const int* pos_sh = reinterpret_cast<const int*>(smem + p.rope_off + kPosOff);
                            qkv_epilogue_attn<B>(p, l, w0 + wc, bb, sum.x, sum.y, rf[bb], epoch, rope, pos_sh);
                            if (spw == 2 && wc + 1 < nwd)
                                qkv_epilogue_attn<B>(p, l, w0 + wc + 1, bb, sum.z, sum.w, rf[bb], epoch, rope, pos_sh);
                            continue;
                        }
                    }
                    if (g.type == kGU) {
                        word_epilogue<B>(p, g, w0 + wc, bb, sum.x, sum.z, sum.y, sum.w, rf[bb], 0u, epoch);
                    } else {
                        const bool resid = (g.type == kO || g.type == kDOWN);
                        word_epilogue<B>(p, g, w0 + wc, bb, sum.x, sum.y, 0.f, 0.f, rf[bb],
                                         resid ? res[bb * nwd + wc] : 0u, epoch);
                        if (spw == 2 && wc + 1 < nwd)
                            word_epilogue<B>(p, g, w0 + wc + 1, bb, sum.z, sum.w, 0.f, 0.f, rf[bb],
                                             resid ? res[bb * nwd + wc + 1] : 0u, epoch);
                    }
                }
            }
            cord0 += nch;
        }
    }

    // ---------------------------------------------------- token epilogue
    __syncthreads();
    if (threadIdx.x == 0) {
        __threadfence();
        const uint32_t prev = atomicAdd(p.done, 1u);
        if (prev == gridDim.x - 1) {
            atomicExch(p.done, 0u);
            __threadfence();
            atomicExch(p.seq, epoch);
        }
    }
}

// ------------------------------------------------- graph path (batch 3-32) --
//
// For batches beyond what the persistent kernel stages in shared memory, the
// token runs as a CUDA graph (captured once per plan) of tensor-core stage
// kernels and per-stage epilogues (wq4_tc.cu); they write the same workspace
// traces as the persistent kernel.

// Decode step of the graph path: one block per batch row rotates q and k of
// layer l's QKV output (the same fp64 rotation as the persistent kernel),
// writes the traces, appends k and v to the cache and sets the row's
// sequence length (positions + 1; 0 for an invalid position).  Launched
// after the QKV stage with programmatic dependent launch: it reads the QKV
// output only after that grid has completed.
struct RopeAppendArgs {
    const uint16_t* qkv;        // [B][Nqkv]
    uint16_t* qr;               // [B][H] rotated queries
    uint16_t* kr;               // [B][Hkv 128] rotated keys
    int32_t* seq_lens;          // [B]
    const int32_t* positions;   // [B]
    KvLayer kv;
    int P, Hkv, H, Nqkv;
    uint32_t* err;
    double inv_freq[kAttnD / 2];
};

__global__ void __launch_bounds__(256) rope_append_kernel(const __grid_constant__ RopeAppendArgs a)
{
    __shared__ double2 rope[kAttnD / 2];
    asm volatile("griddepcontrol.wait;" ::: "memory");
    const int b = blockIdx.x;
    const int pos = __ldg(a.positions + b);
    if (threadIdx.x < kAttnD / 2) {
        double sn, cn;
        sincos(static_cast<double>(pos < 0 ? 0 : pos) * a.inv_freq[threadIdx.x], &sn, &cn);
        rope[threadIdx.x] = make_double2(cn, sn);
    }
    if (threadIdx.x == 0) a.seq_lens[b] = pos < 0 ? 0 : pos + 1;
    __syncthreads();
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    const int H = a.H, KD = a.Hkv * kAttnD;
    const uint32_t* row = reinterpret_cast<const uint32_t*>(a.qkv + static_cast<size_t>(b) * a.Nqkv);
    for (int w = threadIdx.x; w < (H + 2 * KD) / 2; w += blockDim.x) {
        const int n = 2 * w;
        const uint32_t x = row[w];
        if (n < H + KD) {
            const double2 cs = rope[(n & (kAttnD - 1)) >> 1];
            const double u0 = half_bits_to_float(static_cast<uint16_t>(x & 0xFFFFu));
            const double u1 = half_bits_to_float(static_cast<uint16_t>(x >> 16));
            const uint32_t rw = pack2(double_to_half_bits(u0 * cs.x - u1 * cs.y), double_to_half_bits(u0 * cs.y + u1 * cs.x));
            if (n < H) {
                *reinterpret_cast<uint32_t*>(a.qr + static_cast<size_t>(b) * H + n) = rw;
            } else {
                const int kn = n - H;
                *reinterpret_cast<uint32_t*>(a.kr + static_cast<size_t>(b) * KD + kn) = rw;
                uint16_t* r = append_row(a.kv, a.P, a.Hkv, a.kv.k, b, pos, kn / kAttnD);
                if (r) *reinterpret_cast<uint32_t*>(r + (kn & (kAttnD - 1))) = rw;
                else if ((kn & (kAttnD - 1)) == 0) atomicOr(a.err, kErrAppend);
            }
        } else {
            const int vn = n - H - KD;
            uint16_t* r = append_row(a.kv, a.P, a.Hkv, a.kv.v, b, pos, vn / kAttnD);
            if (r) *reinterpret_cast<uint32_t*>(r + (vn & (kAttnD - 1))) = x;
        }
    }
}

// ---------------------------------------------------------------- host --

struct Layout {
    size_t header, llA, llX1, llM, llX, llV, pV, pX2, pQKV, pO, pX1, pGU, pM, pD, x_stage, logits_stage, rfac,
        xpH0, xpH1, xpF, cnt, part, total;
    size_t ll_begin, ll_end;
    // decode step (after everything above, so that the chain's offsets stay):
    // flagged words of the new keys, values and attention output (zeroed),
    // traces, split partials and counters (batch 1-2), or the sequence
    // lengths and wq4_paged_attention's workspace (batch 3-32)
    size_t att_ll_begin, att_ll_end, llK, llVn, llAt, pQr, pKr, pAt, apart, acnt, seq_lens, attn_ws, attn_ws_bytes;
};

struct Dims {
    int L, H, F, Nqkv, V, B;
    int nq, Hkv, Dh;     // query heads, kv heads, head dimension
};

// Heads the decode step's attention handles: head dimension 128, a whole
// number of query heads (at most kAttnMaxGroup) per kv head.
bool attn_heads_ok(const Dims& d)
{
    return d.Dh == kAttnD && d.Hkv >= 1 && d.nq % d.Hkv == 0 && d.nq / d.Hkv <= kAttnMaxGroup;
}

bool table_dims(const wq4_layer_table* t, Dims* d)
{
    if (!t) return false;
    if (t->num_layers < 1 || t->num_layers > 4096) return false;
    if (t->hidden < 256 || t->hidden % 256) return false;
    if (t->ffn < 256 || t->ffn % 256) return false;
    if (t->n_q_heads < 1 || t->n_kv_heads < 0 || t->head_dim < 1) return false;
    if (static_cast<int64_t>(t->n_q_heads) * t->head_dim != t->hidden) return false;
    const int64_t nqkv = static_cast<int64_t>(t->n_q_heads + 2 * t->n_kv_heads) * t->head_dim;
    if (nqkv % 2 || nqkv > (1 << 24)) return false;
    if (t->vocab < 1 || t->vocab > (1 << 24)) return false;
    if (t->batch < 1 || t->batch > WQ4_MAX_BATCH) return false;
    if (!(t->rms_eps > 0.f) || !std::isfinite(t->rms_eps)) return false;
    if (!t->layers) return false;
    d->L = t->num_layers;
    d->H = t->hidden;
    d->F = t->ffn;
    d->Nqkv = static_cast<int>(nqkv);
    d->V = t->vocab;
    d->B = t->batch;
    d->nq = t->n_q_heads;
    d->Hkv = t->n_kv_heads;
    d->Dh = t->head_dim;
    return true;
}

Layout make_layout(const Dims& d, bool att = false, size_t attn_ws_bytes = 0)
{
    Layout y;
    size_t o = 0;
    auto take = [&](size_t bytes) {
        const size_t at = o;
        o = align_up(o + bytes, 256);
        return at;
    };
    const size_t B = d.B, L = d.L, H = d.H, F = d.F;
    y.header = take(256);
    y.ll_begin = o;
    y.llA = take(8 * 2 * L * B * (H / 2));        // two replicas each
    y.llX1 = take(8 * 2 * L * B * (H / 2));
    y.llM = take(8 * 2 * L * B * (F / 2));
    y.llX = take(8 * 2 * (L + 1) * B * (H / 2));
    y.llV = take(8 * 2 * L * B * (H / 2));
    y.ll_end = o;
    y.pV = take(2 * (L + 1) * B * H);
    y.pX2 = take(2 * L * B * H);
    y.pQKV = take(2 * L * B * d.Nqkv);
    y.pO = take(2 * L * B * H);
    y.pX1 = take(2 * L * B * H);
    y.pGU = take(2 * L * B * 2 * F);
    y.pM = take(2 * L * B * F);
    y.pD = take(2 * L * B * H);
    y.x_stage = take(2 * B * H);
    y.logits_stage = take(2 * B * static_cast<size_t>(d.V));
    if (d.B > kMaxChainBatch) {
        // batched path: sums of squares of 128-element tiles (u, a, x1),
        // arrival counters, permuted stage inputs, K-part partial sums
        y.rfac = take(4 * 3 * (H / 128) * B);
        y.cnt = take(4 * static_cast<size_t>(kTcCounterWords));
        y.xpH0 = take(2 * 32 * H);
        y.xpH1 = take(2 * 32 * H);
        y.xpF = take(2 * 32 * F);
        y.part = take(4 * tc_part_floats(d.L, d.H, d.F, d.Nqkv, d.V, d.B, 256));
    } else {
        y.rfac = y.cnt = y.xpH0 = y.xpH1 = y.xpF = y.part = 0;
    }
    y.att_ll_begin = y.att_ll_end = y.llK = y.llVn = y.llAt = y.pQr = y.pKr = y.pAt = 0;
    y.apart = y.acnt = y.seq_lens = y.attn_ws = y.attn_ws_bytes = 0;
    if (att) {
        const size_t KD = static_cast<size_t>(d.Hkv) * kAttnD, G = d.Hkv > 0 ? d.nq / d.Hkv : 0;
        y.att_ll_begin = o;
        y.llK = take(8 * L * B * (KD / 2));
        y.llVn = take(8 * L * B * (KD / 2));
        y.llAt = take(8 * 2 * L * B * (H / 2));          // two replicas
        y.att_ll_end = o;
        y.pQr = take(2 * L * B * H);
        y.pKr = take(2 * L * B * KD);
        y.pAt = take(2 * L * B * H);
        if (d.B <= kMaxChainBatch) {
            y.apart = take(4 * L * B * d.Hkv * kAttnMaxSplits * G * kAttnPart);
            y.acnt = take(4 * L * B * d.Hkv);
        } else {
            y.seq_lens = take(4 * B);
            y.attn_ws = take(attn_ws_bytes);
            y.attn_ws_bytes = attn_ws_bytes;
        }
    }
    y.total = o;
    return y;
}

struct Plan {
    wq4_layer_table table;
    std::vector<wq4_layer> layers;
    Dims dims;
    Layout lay;
    int device;
    int grid;
    int nslots, nbars;
    uint32_t slot_bytes, x_bytes;
    size_t smem;
    int nw;
    int q[5];                // K parts per superpair, per stage type
    int spw[5];              // words per superpair, per stage type
    cudaGraphExec_t graph;   // graph path (batch > kMaxChainBatch), else null
    // decode step only
    bool att = false;
    std::vector<wq4_kv_cache> kv;
    const int32_t* positions = nullptr;
    double theta = 0.0;
    float scale = 0.f;
    int S = 0;               // splits per (row, kv head)
    uint32_t rope_off = 0;
};

std::mutex g_plan_mu;
// plans by (table, decode step or chain)
std::map<std::pair<const wq4_layer_table*, bool>, Plan> g_plans;

// Test hook state (wq4_test_chain_waits): the limit of the chain kernel's
// waits on flagged words and the stage whose input waits can never be
// satisfied.  The mbarrier waits of the weight ring keep kWaitTimeoutNs: a
// producer that gave up early would refill a slot that is still being read.
std::atomic<uint64_t> g_wait_ns{kWaitTimeoutNs};
std::atomic<int> g_stall_stage{-1};

bool same_contents(const Plan& pl, const wq4_layer_table* t, const wq4_decode_attn* a)
{
    if (std::memcmp(&pl.table, t, sizeof(*t)) != 0) return false;
    if (std::memcmp(pl.layers.data(), t->layers, sizeof(wq4_layer) * t->num_layers) != 0) return false;
    if (pl.att != (a != nullptr)) return false;
    if (!a) return true;
    return pl.positions == a->positions && pl.theta == a->rope_theta && pl.scale == a->scale &&
           std::memcmp(pl.kv.data(), a->layers, sizeof(wq4_kv_cache) * t->num_layers) == 0;
}

// The attention description of a decode step, checked against the table.
int check_attn(const wq4_layer_table* t, const Dims& d, const wq4_decode_attn* a)
{
    if (!a || !a->layers || !a->positions) return WQ4_ERR_INVALID;
    if (!attn_heads_ok(d)) return WQ4_ERR_UNSUPPORTED;
    if (!(a->rope_theta > 1.0) || !std::isfinite(a->rope_theta)) return WQ4_ERR_INVALID;
    if (!(a->scale > 0.f) || !std::isfinite(a->scale)) return WQ4_ERR_INVALID;
    if (!aligned(a->positions, 4)) return WQ4_ERR_ALIGN;
    const int P = a->layers[0].page_size;
    for (int l = 0; l < d.L; ++l) {
        const wq4_kv_cache& c = a->layers[l];
        if (!c.k || !c.v || !c.page_table || c.num_pages < 1 || c.page_table_stride < 1) return WQ4_ERR_INVALID;
        if (c.n_kv_heads != d.Hkv || c.head_dim != kAttnD) return WQ4_ERR_INVALID;
        if (c.page_size != P || P < 16 || P % 16) return WQ4_ERR_INVALID;
        if (!aligned(c.k, 16) || !aligned(c.v, 16) || !aligned(c.page_table, 4)) return WQ4_ERR_ALIGN;
        const int64_t rows = static_cast<int64_t>(c.num_pages) * d.Hkv * P;
        if (rows >= (int64_t(1) << 31)) return WQ4_ERR_UNSUPPORTED;
        if (static_cast<int64_t>(c.page_table_stride) * P >= (int64_t(1) << 30)) return WQ4_ERR_UNSUPPORTED;
        const size_t cb = static_cast<size_t>(rows) * kAttnD * 2;
        if (overlaps(c.k, cb, c.v, cb) || overlaps(c.k, cb, t->workspace, t->workspace_bytes) ||
            overlaps(c.v, cb, t->workspace, t->workspace_bytes))
            return WQ4_ERR_INVALID;
    }
    return WQ4_OK;
}

bool mat_ok(const wq4_mat& m)
{
    return m.W && m.s && aligned(m.W, 16) && aligned(m.s, 16);
}

template <int B, bool ATT>
cudaError_t set_chain_attr(int smem)
{
    return cudaFuncSetAttribute(chain_kernel<B, kChainWarps, ATT>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
}

// Bytes of one output word of each stage type (two rows; gate_up four).
void word_bytes(const Dims& d, size_t out[5])
{
    const size_t rowH = static_cast<size_t>(d.H) / 2 + d.H / 16, rowF = static_cast<size_t>(d.F) / 2 + d.F / 16;
    out[0] = 2 * rowH;   // QKV
    out[1] = 2 * rowH;   // O
    out[2] = 4 * rowH;   // gate_up
    out[3] = 2 * rowF;   // down
    out[4] = 2 * rowH;   // LM head
}

// Words of each stage type.
void stage_words(const Dims& d, int out[5])
{
    out[0] = d.Nqkv / 2;
    out[1] = d.H / 2;
    out[2] = d.F / 2;
    out[3] = d.H / 2;
    out[4] = (d.V + 1) / 2;
}

// Words per superpair of each stage type: two words (four rows sharing the
// activations) unless that is more than kMaxSuperpairBytes of weights;
// gate_up's word already holds two row pairs.
constexpr size_t kMaxSuperpairBytes = 20 * 1024;
void choose_spw(const Dims& d, int spw[5])
{
    size_t wb[5];
    word_bytes(d, wb);
    for (int t = 0; t < 5; ++t) spw[t] = (t == 2 || 2 * wb[t] > kMaxSuperpairBytes) ? 1 : 2;
}

// Slot size: a multiple of 128 bytes holding at least one superpair of every
// stage, chosen to waste the least ring space over the chain's byte mix.
uint32_t choose_slot_bytes(const Dims& d, const int spw[5])
{
    size_t wb[5];
    word_bytes(d, wb);
    int words[5];
    stage_words(d, words);
    size_t max_item = 0;
    for (int t = 0; t < 5; ++t) max_item = wb[t] * spw[t] > max_item ? wb[t] * spw[t] : max_item;
    size_t lo = align_up(max_item, 128);
    if (lo < 16384) lo = 16384;
    size_t best = lo;
    double best_waste = 1e300;
    for (size_t sb = lo; sb <= lo + 8192; sb += 128) {
        double waste = 0;
        for (int t = 0; t < 5; ++t) {
            const size_t wps = sb / wb[t] / spw[t] * spw[t];
            waste += static_cast<double>(words[t]) * wb[t] * (1.0 - static_cast<double>(wps * wb[t]) / sb);
        }
        if (waste < best_waste) {
            best_waste = waste;
            best = sb;
        }
    }
    return static_cast<uint32_t>(best);
}

int full_bars(int nslots)
{
    return (kFullBars / nslots) * nslots;
}

// K parts per superpair for each stage type: a divisor q of the stage's
// 256-code group sets that gives the least per-warp time when the CTA's
// superpairs x q items are taken round-robin by the consumer warps: rounds x
// (units x unit cost + item cost), with the costs measured on this kernel
// (a unit of two row pairs ~300 cycles, one row pair ~200, an item ~1200:
// the first unit's latency, the reduction and the chunk hand-over).  The
// items the warps run at once must sit in at most nslots - 2 chunks, or the
// last warps wait for slots; the partial sums of all the CTA's superpairs
// must fit in shared memory.  The LM head keeps whole superpairs (q = 1, no
// partial sums).  Returns false if some stage has no admissible q.
bool choose_parts(const Dims& d, int grid, int nw, const int spw[5], int nslots, uint32_t slot_bytes, int q[5])
{
    int words[5];
    stage_words(d, words);
    size_t wb[5];
    word_bytes(d, wb);
    const int J[5] = {d.H / 256, d.H / 256, d.H / 256, d.F / 256, d.H / 256};
    q[4] = 1;
    for (int t = 0; t < 4; ++t) {
        q[t] = 0;
        const long wmax = (words[t] + grid - 1) / grid;
        const long spmax = (wmax + spw[t] - 1) / spw[t];
        size_t spc = slot_bytes / wb[t] / spw[t];
        if (spc < 1) spc = 1;
        const bool two = t == 2 || spw[t] == 2;
        const double unit = two ? 300.0 * (1.0 + 0.5 * (d.B - 1)) : 200.0 * (1.0 + 0.5 * (d.B - 1));
        double best = 1e300;
        for (int c = 1; c <= J[t]; ++c) {
            if (J[t] % c || spmax * c * d.B > kMaxPart) continue;
            const size_t ips = spc * static_cast<size_t>(c);
            if ((static_cast<size_t>(nw) + ips - 1) / ips > static_cast<size_t>(nslots > 3 ? nslots - 2 : 1)) continue;
            const long rounds = (spmax * c + nw - 1) / nw;
            const double cost = static_cast<double>(rounds) * ((J[t] / c) * unit + 1200.0);
            if (cost <= best) {   // ties: more, shorter items (measured faster)
                best = cost;
                q[t] = c;
            }
        }
        if (q[t] == 0) return false;
    }
    return true;
}

// True when no consumer wait on the ring can alias: for every stage,
// nslots + ceil(NW / items per slot) <= the number of full barriers (items
// per slot = superpairs per slot x K parts).
bool ring_ok(const Dims& d, int nslots, uint32_t slot_bytes, int nw, const int spw[5], const int q[5])
{
    size_t wb[5];
    word_bytes(d, wb);
    for (int t = 0; t < 5; ++t) {
        size_t sps = slot_bytes / wb[t] / spw[t];
        if (sps < 1) sps = 1;
        const size_t ips = sps * static_cast<size_t>(q[t]);
        if (static_cast<size_t>(nslots) + (nw + ips - 1) / ips > static_cast<size_t>(full_bars(nslots))) return false;
    }
    return true;
}

// Largest |scale| (as fp16 bits without the sign) of n scales into *out.
__global__ void scale_max_kernel(const uint16_t* s, size_t n, uint32_t* out)
{
    uint32_t m = 0;
    for (size_t i = static_cast<size_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n;
         i += static_cast<size_t>(gridDim.x) * blockDim.x) {
        const uint32_t b = s[i] & 0x7FFFu;
        m = b > m ? b : m;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const uint32_t t = __shfl_xor_sync(0xffffffffu, m, o);
        m = t > m ? t : m;
    }
    if ((threadIdx.x & 31) == 0) atomicMax(out, m);
}

// The batched path rounds each dequantized weight (q - 7) s to fp16: every
// scale of the table must be within +-8188.  Scans all scales once (at plan
// build) and synchronizes `stream` to read the result.
int check_scales_fp16(const wq4_layer_table* t, const Dims& d, uint32_t* scratch_word, cudaStream_t stream)
{
    if (cudaMemsetAsync(scratch_word, 0, 4, stream) != cudaSuccess) return WQ4_ERR_CUDA;
    auto scan = [&](const wq4_mat& m, size_t n) {
        scale_max_kernel<<<64, 256, 0, stream>>>(m.s, n, scratch_word);
        return cudaGetLastError() == cudaSuccess;
    };
    const size_t H = d.H, F = d.F;
    for (int l = 0; l < d.L; ++l) {
        const wq4_layer& ly = t->layers[l];
        if (!scan(ly.qkv, static_cast<size_t>(d.Nqkv) * (H / 32)) || !scan(ly.o, H * (H / 32)) ||
            !scan(ly.gate_up, 2 * F * (H / 32)) || !scan(ly.down, H * (F / 32)))
            return WQ4_ERR_CUDA;
    }
    if (!scan(t->lm_head, static_cast<size_t>(d.V) * (H / 32))) return WQ4_ERR_CUDA;
    uint32_t m = 0;
    if (cudaMemcpyAsync(&m, scratch_word, 4, cudaMemcpyDeviceToHost, stream) != cudaSuccess) return WQ4_ERR_CUDA;
    if (cudaStreamSynchronize(stream) != cudaSuccess) return WQ4_ERR_CUDA;
    return m > kMaxFp16ScaleBits ? WQ4_ERR_UNSUPPORTED : WQ4_OK;
}

KvLayer kv_layer(const wq4_kv_cache& c)
{
    KvLayer k;
    k.k = c.k;
    k.v = c.v;
    k.pt = c.page_table;
    k.pt_stride = c.page_table_stride;
    k.num_pages = c.num_pages;
    return k;
}

void fill_inv_freq(double theta, double* out)
{
    for (int i = 0; i < kAttnD / 2; ++i) out[i] = std::pow(theta, -2.0 * i / kAttnD);
}

// The decode step's attention nodes of the graph path (see TcAttnHook): the
// rotation/append kernel, wq4_paged_attention on the rotated queries, and the
// token-start kernel on the attention output (O's permuted input).
struct GraphAttn {
    const Plan* pl;
    const Dims* d;
    const Layout* lay;
    uint8_t* ws;
};

int record_graph_attention(void* ctx, int l, cudaStream_t cs, uint16_t* xp, float* sq)
{
    const GraphAttn& g = *static_cast<const GraphAttn*>(ctx);
    const Dims& d = *g.d;
    const Layout& y = *g.lay;
    const size_t B = d.B, H = d.H, KD = static_cast<size_t>(d.Hkv) * kAttnD;
    const wq4_kv_cache& c = g.pl->kv[l];
    RopeAppendArgs a;
    std::memset(&a, 0, sizeof(a));
    a.qkv = reinterpret_cast<const uint16_t*>(g.ws + y.pQKV) + static_cast<size_t>(l) * B * d.Nqkv;
    a.qr = reinterpret_cast<uint16_t*>(g.ws + y.pQr) + static_cast<size_t>(l) * B * H;
    a.kr = reinterpret_cast<uint16_t*>(g.ws + y.pKr) + static_cast<size_t>(l) * B * KD;
    a.seq_lens = reinterpret_cast<int32_t*>(g.ws + y.seq_lens);
    a.positions = g.pl->positions;
    a.kv = kv_layer(c);
    a.P = c.page_size;
    a.Hkv = d.Hkv;
    a.H = d.H;
    a.Nqkv = d.Nqkv;
    a.err = status_word();
    if (!a.err) return WQ4_ERR_CUDA;
    fill_inv_freq(g.pl->theta, a.inv_freq);
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(d.B);
    cfg.blockDim = dim3(256);
    cfg.stream = cs;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (cudaLaunchKernelEx(&cfg, rope_append_kernel, a) != cudaSuccess) return WQ4_ERR_CUDA;
    uint16_t* at = reinterpret_cast<uint16_t*>(g.ws + y.pAt) + static_cast<size_t>(l) * B * H;
    int rc = wq4_paged_attention(&c, a.qr, d.H, a.seq_lens, at, d.H, d.B, d.nq, g.pl->scale, g.ws + y.attn_ws,
                                 y.attn_ws_bytes, cs);
    if (rc != WQ4_OK) return rc;
    return tc_launch_prologue(at, d.H, d.B, sq, xp, cs);
}

// Records one token of the graph path on `cs`: every stage kernel of every
// layer (and with pl->att the attention of each), reading the token input
// from the workspace staging area and writing the logits to the workspace
// logits area.
int build_graph_plan(const wq4_layer_table* t, const Dims& d, const Layout& lay, int dev, const DeviceInfo* di,
                     Plan* pl, cudaStream_t stream)
{
    uint8_t* ws = static_cast<uint8_t*>(t->workspace);
    // scales beyond +-8188 would overflow the fp16 dequantized weights
    const int rs = check_scales_fp16(t, d, reinterpret_cast<uint32_t*>(ws + lay.header) + 3, stream);
    if (rs != WQ4_OK) return rs;
    auto U16 = [&](size_t off) { return reinterpret_cast<uint16_t*>(ws + off); };
    TcBuffers buf;
    buf.x_stage = U16(lay.x_stage);
    buf.pV = U16(lay.pV);
    buf.pQKV = U16(lay.pQKV);
    buf.pO = U16(lay.pO);
    buf.pX1 = U16(lay.pX1);
    buf.pGU = U16(lay.pGU);
    buf.pM = U16(lay.pM);
    buf.pD = U16(lay.pD);
    buf.pX2 = U16(lay.pX2);
    buf.logits = U16(lay.logits_stage);
    buf.sq = reinterpret_cast<float*>(ws + lay.rfac);
    buf.cnt = reinterpret_cast<uint32_t*>(ws + lay.cnt);
    buf.xpH[0] = U16(lay.xpH0);
    buf.xpH[1] = U16(lay.xpH1);
    buf.xpF = U16(lay.xpF);
    buf.part = reinterpret_cast<float*>(ws + lay.part);
    TcPlan* tc = nullptr;
    int rc = tc_plan_create(t, d.H, d.F, d.Nqkv, d.V, d.B, buf, di->sm_count, status_word(), &tc);
    if (rc != WQ4_OK) return rc;
    cudaStream_t cs = nullptr;
    if (cudaStreamCreateWithFlags(&cs, cudaStreamNonBlocking) != cudaSuccess) {
        tc_plan_destroy(tc);
        return WQ4_ERR_CUDA;
    }
    cudaGraph_t graph = nullptr;
    cudaGraphExec_t exec = nullptr;
    rc = WQ4_ERR_CUDA;
    if (cudaStreamBeginCapture(cs, cudaStreamCaptureModeThreadLocal) == cudaSuccess) {
        // every token starts with zero arrival counters (a stage whose waits gave
        // up may leave some non-zero; the next token must not inherit them)
        int rrec = cudaMemsetAsync(ws + lay.cnt, 0, 4 * static_cast<size_t>(kTcCounterWords), cs) == cudaSuccess
                       ? WQ4_OK
                       : WQ4_ERR_CUDA;
        GraphAttn ga{pl, &d, &lay, ws};
        const TcAttnHook hook{record_graph_attention, &ga};
        if (rrec == WQ4_OK) rrec = tc_record_token(tc, cs, pl->att ? &hook : nullptr);
        if (cudaStreamEndCapture(cs, &graph) == cudaSuccess && graph && rrec == WQ4_OK &&
            cudaGraphInstantiate(&exec, graph, 0) == cudaSuccess)
            rc = WQ4_OK;
    }
    if (graph) cudaGraphDestroy(graph);
    cudaStreamDestroy(cs);
    tc_plan_destroy(tc);   // the graph holds copies of every launch argument
    if (rc != WQ4_OK) return rc;
    pl->table = *t;
    pl->layers.assign(t->layers, t->layers + d.L);
    pl->dims = d;
    pl->lay = lay;
    pl->device = dev;
    pl->grid = di->sm_count;
    pl->nslots = 0;
    pl->nbars = 0;
    pl->slot_bytes = 0;
    pl->x_bytes = 0;
    pl->smem = 0;
    pl->nw = 0;
    pl->graph = exec;
    return WQ4_OK;
}

int build_plan(const wq4_layer_table* t, const wq4_decode_attn* a, Plan* pl, cudaStream_t stream)
{
    Dims d;
    if (!table_dims(t, &d)) return WQ4_ERR_INVALID;
    pl->graph = nullptr;
    for (int l = 0; l < d.L; ++l) {
        const wq4_layer& ly = t->layers[l];
        if (!mat_ok(ly.qkv) || !mat_ok(ly.o) || !mat_ok(ly.gate_up) || !mat_ok(ly.down)) return WQ4_ERR_INVALID;
    }
    if (!mat_ok(t->lm_head)) return WQ4_ERR_INVALID;
    if (!t->workspace || !aligned(t->workspace, 256)) return WQ4_ERR_ALIGN;
    size_t attn_ws = 0;
    if (a) {
        const int ra = check_attn(t, d, a);
        if (ra != WQ4_OK) return ra;
        if (d.B > kMaxChainBatch) {
            attn_ws = wq4_paged_attention_workspace_bytes(d.B, d.nq, d.Hkv, kAttnD);
            if (attn_ws == 0) return WQ4_ERR_CUDA;
        }
    }
    const Layout lay = make_layout(d, a != nullptr, attn_ws);
    if (t->workspace_bytes < lay.total) return WQ4_ERR_INVALID;
    int dev = 0;
    const DeviceInfo* di = current_device_info(&dev);
    if (!di) return WQ4_ERR_CUDA;
    if (a) {
        pl->att = true;
        pl->kv.assign(a->layers, a->layers + d.L);
        pl->positions = a->positions;
        pl->theta = a->rope_theta;
        pl->scale = a->scale;
        uint8_t* ws = static_cast<uint8_t*>(t->workspace);
        // flagged words start at zero (epoch 0 never matches); counters at zero
        if (cudaMemsetAsync(ws + lay.att_ll_begin, 0, lay.att_ll_end - lay.att_ll_begin, stream) != cudaSuccess)
            return WQ4_ERR_CUDA;
        if (lay.acnt && cudaMemsetAsync(ws + lay.acnt, 0, 4 * static_cast<size_t>(d.L) * d.B * d.Hkv, stream) !=
                            cudaSuccess)
            return WQ4_ERR_CUDA;
        if (lay.attn_ws && cudaMemsetAsync(ws + lay.attn_ws, 0, lay.attn_ws_bytes, stream) != cudaSuccess)
            return WQ4_ERR_CUDA;
    }
    if (d.B > kMaxChainBatch) {
        if (d.Nqkv % 8) return WQ4_ERR_UNSUPPORTED;   // the O stage reads qkv rows with 16-byte loads
        return build_graph_plan(t, d, lay, dev, di, pl, stream);
    }
    if (!di->coop_launch) return WQ4_ERR_UNSUPPORTED;
    if (d.L > kChainMaxLayers) return WQ4_ERR_UNSUPPORTED;
    size_t xb = align_up(static_cast<size_t>(d.B) * 2 * (d.H > d.F ? d.H : d.F), 128);
    // the attention's scratch (queries of a group, per-warp partials) lives in the staging area
    if (a) xb = std::max(xb, align_up(4 * static_cast<size_t>(kAttnMaxGroup * kAttnD + kChainWarps * kAttnPart), 128));
    const uint32_t x_bytes = static_cast<uint32_t>(xb);
    // the rotation table (double2 [B][64]), the positions and a flag sit after the ring
    const size_t rope_bytes = a ? align_up(static_cast<size_t>(d.B) * (kAttnD / 2) * 16 + 16, 128) : 0;
    // the residual words of a CTA's words must fit in shared memory
    if (static_cast<long>((d.H / 2 + di->sm_count - 1) / di->sm_count) * d.B > kMaxResWords) return WQ4_ERR_UNSUPPORTED;
    int spw[5];
    choose_spw(d, spw);
    const uint32_t slot_bytes = choose_slot_bytes(d, spw);
    const int header = kChainHeader;
    const long avail = static_cast<long>(di->smem_optin) - header - static_cast<long>(x_bytes) -
                       static_cast<long>(rope_bytes);
    int nslots = avail > 0 ? static_cast<int>(avail / slot_bytes) : 0;
    if (nslots > kChainMaxSlots) nslots = kChainMaxSlots;
    int q[5];
    if (!choose_parts(d, di->sm_count, kChainWarps, spw, nslots, slot_bytes, q)) return WQ4_ERR_UNSUPPORTED;
    // fewer slots give more full barriers per slot: take the deepest ring
    // whose barriers cannot alias
    while (nslots >= 2 && !ring_ok(d, nslots, slot_bytes, kChainWarps, spw, q)) --nslots;
    if (nslots < 2) return WQ4_ERR_UNSUPPORTED;
    const size_t smem = header + x_bytes + static_cast<size_t>(nslots) * slot_bytes + rope_bytes;
    pl->rope_off = static_cast<uint32_t>(header + x_bytes + static_cast<size_t>(nslots) * slot_bytes);
    if (a) {
        int S = di->sm_count / (d.B * d.Hkv);
        pl->S = S < 1 ? 1 : (S > kAttnMaxSplits ? kAttnMaxSplits : S);
    }
    // The limit is a property of the kernel, shared by every plan: set it to
    // the device maximum so that no plan's launch depends on which plan was
    // built last.
    cudaError_t e = cudaSuccess;
    switch (d.B * 2 + (a ? 1 : 0)) {
        case 2: e = set_chain_attr<1, false>(di->smem_optin); break;
        case 3: e = set_chain_attr<1, true>(di->smem_optin); break;
        case 4: e = set_chain_attr<2, false>(di->smem_optin); break;
        default: e = set_chain_attr<2, true>(di->smem_optin); break;
    }
    if (e != cudaSuccess) return WQ4_ERR_CUDA;

    uint8_t* ws = static_cast<uint8_t*>(t->workspace);
    // header (token counter) and every flagged word start at zero: epoch 0 never matches
    if (cudaMemsetAsync(ws + lay.header, 0, 256, stream) != cudaSuccess) return WQ4_ERR_CUDA;
    if (cudaMemsetAsync(ws + lay.ll_begin, 0, lay.ll_end - lay.ll_begin, stream) != cudaSuccess) return WQ4_ERR_CUDA;

    pl->table = *t;
    pl->layers.assign(t->layers, t->layers + d.L);
    pl->dims = d;
    pl->lay = lay;
    pl->device = dev;
    pl->grid = di->sm_count;
    pl->nslots = nslots;
    pl->nbars = full_bars(nslots);
    pl->slot_bytes = slot_bytes;
    pl->x_bytes = x_bytes;
    pl->smem = smem;
    pl->nw = kChainWarps;
    for (int t = 0; t < 5; ++t) pl->q[t] = q[t];
    for (int t = 0; t < 5; ++t) pl->spw[t] = spw[t];
    return WQ4_OK;
}

template <class P>
int fill_chain_params(P& p, const Plan& pl, const uint16_t* x, uint16_t* logits)
{
    uint8_t* ws = static_cast<uint8_t*>(pl.table.workspace);
    const Layout& y = pl.lay;
    for (int l = 0; l < pl.dims.L; ++l) {
        const wq4_layer& ly = pl.layers[l];
        p.mats[4 * l + 0] = {ly.qkv.W, ly.qkv.s};
        p.mats[4 * l + 1] = {ly.o.W, ly.o.s};
        p.mats[4 * l + 2] = {ly.gate_up.W, ly.gate_up.s};
        p.mats[4 * l + 3] = {ly.down.W, ly.down.s};
    }
    p.mats[4 * pl.dims.L] = {pl.table.lm_head.W, pl.table.lm_head.s};
    p.L = pl.dims.L;
    p.H = pl.dims.H;
    p.F = pl.dims.F;
    p.Nqkv = pl.dims.Nqkv;
    p.V = pl.dims.V;
    p.eps = pl.table.rms_eps;
    p.x = x;
    p.logits = logits;
    p.seq = reinterpret_cast<uint32_t*>(ws + y.header);
    p.done = reinterpret_cast<uint32_t*>(ws + y.header) + 1;
    p.abort = reinterpret_cast<uint32_t*>(ws + y.header) + 2;
    p.llA = reinterpret_cast<uint64_t*>(ws + y.llA);
    p.llX1 = reinterpret_cast<uint64_t*>(ws + y.llX1);
    p.llM = reinterpret_cast<uint64_t*>(ws + y.llM);
    p.llX = reinterpret_cast<uint64_t*>(ws + y.llX);
    p.llV = reinterpret_cast<uint64_t*>(ws + y.llV);
    {
        const uint32_t L = static_cast<uint32_t>(pl.dims.L), B = static_cast<uint32_t>(pl.dims.B);
        const uint32_t H = static_cast<uint32_t>(pl.dims.H), F = static_cast<uint32_t>(pl.dims.F);
        p.rep.A = L * B * (H / 2);
        p.rep.X1 = L * B * (H / 2);
        p.rep.M = L * B * (F / 2);
        p.rep.X = (L + 1) * B * (H / 2);
        p.rep.V = L * B * (H / 2);
    }
    p.pV = reinterpret_cast<uint16_t*>(ws + y.pV);
    p.pX2 = reinterpret_cast<uint16_t*>(ws + y.pX2);
    p.pQKV = reinterpret_cast<uint16_t*>(ws + y.pQKV);
    p.pO = reinterpret_cast<uint16_t*>(ws + y.pO);
    p.pX1 = reinterpret_cast<uint16_t*>(ws + y.pX1);
    p.pGU = reinterpret_cast<uint16_t*>(ws + y.pGU);
    p.pM = reinterpret_cast<uint16_t*>(ws + y.pM);
    p.pD = reinterpret_cast<uint16_t*>(ws + y.pD);
    p.nslots = pl.nslots;
    p.nbars = pl.nbars;
    p.slot_bytes = pl.slot_bytes;
    p.x_bytes = pl.x_bytes;
    for (int t = 0; t < 5; ++t) p.q[t] = pl.q[t];
    for (int t = 0; t < 5; ++t) p.spw[t] = pl.spw[t];
    p.err = status_word();
    if (!p.err) return WQ4_ERR_CUDA;
    p.wait_ns = g_wait_ns.load();
    p.stall_stage = g_stall_stage.load();

    return WQ4_OK;
}

int launch_chain(const Plan& pl, const uint16_t* x, uint16_t* logits, cudaStream_t stream)
{
    uint8_t* ws = static_cast<uint8_t*>(pl.table.workspace);
    const Layout& y = pl.lay;
    if (pl.graph) {
        // the graph reads the token from and writes the logits to the workspace
        uint16_t* xs = reinterpret_cast<uint16_t*>(ws + y.x_stage);
        uint16_t* ls = reinterpret_cast<uint16_t*>(ws + y.logits_stage);
        const size_t xb = static_cast<size_t>(pl.dims.B) * pl.dims.H * 2;
        const size_t lb = static_cast<size_t>(pl.dims.B) * pl.dims.V * 2;
        if (x != xs && cudaMemcpyAsync(xs, x, xb, cudaMemcpyDeviceToDevice, stream) != cudaSuccess) return WQ4_ERR_CUDA;
        if (cudaGraphLaunch(pl.graph, stream) != cudaSuccess) return WQ4_ERR_CUDA;
        if (logits != ls && cudaMemcpyAsync(logits, ls, lb, cudaMemcpyDeviceToDevice, stream) != cudaSuccess)
            return WQ4_ERR_CUDA;
        return WQ4_OK;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(pl.grid);
    cfg.blockDim = dim3((pl.nw + 1) * 32);
    cfg.dynamicSmemBytes = pl.smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeCooperative;
    attr[0].val.cooperative = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cudaError_t e;
    if (!pl.att) {
        ChainParams p = {};
        if (fill_chain_params(p, pl, x, logits) != WQ4_OK) return WQ4_ERR_CUDA;
        switch (pl.dims.B) {
            case 1: e = cudaLaunchKernelEx(&cfg, chain_kernel<1, kChainWarps, false>, p); break;
            default: e = cudaLaunchKernelEx(&cfg, chain_kernel<2, kChainWarps, false>, p); break;
        }
    } else {
        ChainParamsA p = {};
        if (fill_chain_params(p, pl, x, logits) != WQ4_OK) return WQ4_ERR_CUDA;
        const size_t L = pl.dims.L, B = pl.dims.B, H = pl.dims.H;
        p.Hkv = pl.dims.Hkv;
        p.G = pl.dims.nq / pl.dims.Hkv;
        p.P = pl.kv[0].page_size;
        p.S = pl.S;
        p.scale = pl.scale;
        p.positions = pl.positions;
        p.llK = reinterpret_cast<uint64_t*>(ws + y.llK);
        p.llVn = reinterpret_cast<uint64_t*>(ws + y.llVn);
        p.llAt = reinterpret_cast<uint64_t*>(ws + y.llAt);
        p.repAt = static_cast<uint32_t>(L * B * (H / 2));
        p.rope_off = pl.rope_off;
        p.pQr = reinterpret_cast<uint16_t*>(ws + y.pQr);
        p.pKr = reinterpret_cast<uint16_t*>(ws + y.pKr);
        p.pAt = reinterpret_cast<uint16_t*>(ws + y.pAt);
        p.apart = reinterpret_cast<float*>(ws + y.apart);
        p.acnt = reinterpret_cast<uint32_t*>(ws + y.acnt);
        fill_inv_freq(pl.theta, p.inv_freq);
        for (int l = 0; l < pl.dims.L; ++l) p.kv[l] = kv_layer(pl.kv[l]);
        switch (pl.dims.B) {
            case 1: e = cudaLaunchKernelEx(&cfg, chain_kernel<1, kChainWarps, true>, p); break;
            default: e = cudaLaunchKernelEx(&cfg, chain_kernel<2, kChainWarps, true>, p); break;
        }
    }
    return e == cudaSuccess ? WQ4_OK : WQ4_ERR_CUDA;
}

// Finds (or builds) the plan of `t`; returns a copy to launch from.  With
// no_rebuild_in_capture, a plan that would have to be (re)built while
// `stream` is capturing is refused with WQ4_ERR_UNSUPPORTED.
int get_plan(const wq4_layer_table* t, const wq4_decode_attn* a, Plan* out, cudaStream_t stream,
             bool no_rebuild_in_capture = false)
{
    if (!t) return WQ4_ERR_INVALID;
    Dims d;
    if (!table_dims(t, &d)) return WQ4_ERR_INVALID;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return WQ4_ERR_CUDA;
    std::lock_guard<std::mutex> lock(g_plan_mu);
    const std::pair<const wq4_layer_table*, bool> key(t, a != nullptr);
    auto it = g_plans.find(key);
    if (it != g_plans.end() && it->second.device == dev && same_contents(it->second, t, a)) {
        *out = it->second;
        return WQ4_OK;
    }
    if (no_rebuild_in_capture) {
        cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
        if (cudaStreamIsCapturing(stream, &cs) != cudaSuccess) return WQ4_ERR_CUDA;
        if (cs != cudaStreamCaptureStatusNone) return WQ4_ERR_UNSUPPORTED;
    }
    Plan pl;
    const int rc = build_plan(t, a, &pl, stream);
    if (rc != WQ4_OK) return rc;
    if (it != g_plans.end() && it->second.graph) {
        // a replaced graph may still run on the GPU: free it once it is done
        cudaStreamSynchronize(stream);
        cudaGraphExecDestroy(it->second.graph);
    }
    g_plans[key] = pl;
    *out = pl;
    return WQ4_OK;
}

}  // namespace
}  // namespace wq4

using namespace wq4;

extern "C" size_t wq4_chain_workspace_bytes(const wq4_layer_table* table)
{
    Dims d;
    if (!table_dims(table, &d)) return 0;
    return make_layout(d).total;
}

extern "C" int wq4_decode_chain(const wq4_layer_table* table, const uint16_t* x, uint16_t* logits, void* stream)
{
    if (!table || !x || !logits) return WQ4_ERR_INVALID;
    if (!aligned(x, 16) || !aligned(logits, 2)) return WQ4_ERR_ALIGN;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    Plan pl;
    const int rc = get_plan(table, nullptr, &pl, st);
    if (rc != WQ4_OK) return rc;
    const size_t lb = static_cast<size_t>(pl.dims.B) * pl.dims.V * 2;
    if (overlaps(logits, lb, x, static_cast<size_t>(pl.dims.B) * pl.dims.H * 2) ||
        overlaps(logits, lb, table->workspace, pl.lay.logits_stage))
        return WQ4_ERR_INVALID;
    return launch_chain(pl, x, logits, st);
}

extern "C" int wq4_decode_chain_host(const wq4_layer_table* table, const uint16_t* x_host, uint16_t* logits_host,
                                     void* stream)
{
    if (!table || !x_host || !logits_host) return WQ4_ERR_INVALID;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    Plan pl;
    int rc = get_plan(table, nullptr, &pl, st);
    if (rc != WQ4_OK) return rc;
    uint8_t* ws = static_cast<uint8_t*>(table->workspace);
    uint16_t* xd = reinterpret_cast<uint16_t*>(ws + pl.lay.x_stage);
    uint16_t* ld = reinterpret_cast<uint16_t*>(ws + pl.lay.logits_stage);
    const size_t xb = static_cast<size_t>(pl.dims.B) * pl.dims.H * 2;
    const size_t lb = static_cast<size_t>(pl.dims.B) * pl.dims.V * 2;
    if (cudaMemcpyAsync(xd, x_host, xb, cudaMemcpyHostToDevice, st) != cudaSuccess) return WQ4_ERR_CUDA;
    rc = launch_chain(pl, xd, ld, st);
    if (rc != WQ4_OK) return rc;
    if (cudaMemcpyAsync(logits_host, ld, lb, cudaMemcpyDeviceToHost, st) != cudaSuccess) return WQ4_ERR_CUDA;
    return cudaStreamSynchronize(st) == cudaSuccess ? WQ4_OK : WQ4_ERR_CUDA;
}

extern "C" int wq4_chain_plan_destroy(const wq4_layer_table* table)
{
    std::lock_guard<std::mutex> lock(g_plan_mu);
    int found = 0;
    for (bool att : {false, true}) {
        auto it = g_plans.find(std::make_pair(table, att));
        if (it == g_plans.end()) continue;
        if (it->second.graph) cudaGraphExecDestroy(it->second.graph);
        g_plans.erase(it);
        ++found;
    }
    return found ? WQ4_OK : WQ4_ERR_INVALID;
}

extern "C" int wq4_chain_path(const wq4_layer_table* table, int decode_step)
{
    std::lock_guard<std::mutex> lock(g_plan_mu);
    auto it = g_plans.find(std::make_pair(table, decode_step != 0));
    if (it == g_plans.end()) return WQ4_ERR_INVALID;
    return it->second.graph ? 2 : 1;
}

extern "C" size_t wq4_decode_step_workspace_bytes(const wq4_layer_table* table)
{
    Dims d;
    if (!table_dims(table, &d) || !attn_heads_ok(d)) return 0;
    size_t attn_ws = 0;
    if (d.B > kMaxChainBatch) {
        attn_ws = wq4_paged_attention_workspace_bytes(d.B, d.nq, d.Hkv, kAttnD);
        if (attn_ws == 0) return 0;
    }
    return make_layout(d, true, attn_ws).total;
}

extern "C" int wq4_decode_step(const wq4_layer_table* table, const wq4_decode_attn* attn, const uint16_t* x,
                               uint16_t* logits, void* stream)
{
    if (!table || !attn || !x || !logits) return WQ4_ERR_INVALID;
    if (!aligned(x, 16) || !aligned(logits, 2)) return WQ4_ERR_ALIGN;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    Plan pl;
    const int rc = get_plan(table, attn, &pl, st);
    if (rc != WQ4_OK) return rc;
    const size_t lb = static_cast<size_t>(pl.dims.B) * pl.dims.V * 2;
    if (overlaps(logits, lb, x, static_cast<size_t>(pl.dims.B) * pl.dims.H * 2) ||
        overlaps(logits, lb, table->workspace, pl.lay.total))
        return WQ4_ERR_INVALID;
    return launch_chain(pl, x, logits, st);
}

extern "C" int wq4_decode_step_host(const wq4_layer_table* table, const wq4_decode_attn* attn, const uint16_t* x_host,
                                    uint16_t* logits_host, void* stream)
{
    if (!table || !attn || !x_host || !logits_host) return WQ4_ERR_INVALID;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    Plan pl;
    int rc = get_plan(table, attn, &pl, st);
    if (rc != WQ4_OK) return rc;
    uint8_t* ws = static_cast<uint8_t*>(table->workspace);
    uint16_t* xd = reinterpret_cast<uint16_t*>(ws + pl.lay.x_stage);
    uint16_t* ld = reinterpret_cast<uint16_t*>(ws + pl.lay.logits_stage);
    const size_t xb = static_cast<size_t>(pl.dims.B) * pl.dims.H * 2;
    const size_t lb = static_cast<size_t>(pl.dims.B) * pl.dims.V * 2;
    if (cudaMemcpyAsync(xd, x_host, xb, cudaMemcpyHostToDevice, st) != cudaSuccess) return WQ4_ERR_CUDA;
    rc = launch_chain(pl, xd, ld, st);
    if (rc != WQ4_OK) return rc;
    if (cudaMemcpyAsync(logits_host, ld, lb, cudaMemcpyDeviceToHost, st) != cudaSuccess) return WQ4_ERR_CUDA;
    return cudaStreamSynchronize(st) == cudaSuccess ? WQ4_OK : WQ4_ERR_CUDA;
}

extern "C" int wq4_test_chain_waits(uint64_t wait_limit_ns, int stall_stage)
{
    if (wait_limit_ns == 0 || wait_limit_ns > kWaitTimeoutNs || stall_stage < -1) return WQ4_ERR_INVALID;
    g_wait_ns.store(wait_limit_ns);
    g_stall_stage.store(stall_stage);
    return WQ4_OK;
}

extern "C" int wq4_chain_trace_offsets(const wq4_layer_table* table, int layer, wq4_chain_trace* out)
{
    Dims d;
    if (!out || !table_dims(table, &d) || layer < 0 || layer > d.L) return WQ4_ERR_INVALID;
    const Layout y = make_layout(d);
    const size_t B = d.B, H = d.H, F = d.F, l = layer;
    std::memset(out, 0, sizeof(*out));
    out->x_in = y.pV + 2 * l * B * H;
    if (layer == d.L) return WQ4_OK;
    out->qkv = y.pQKV + 2 * l * B * d.Nqkv;
    out->o = y.pO + 2 * l * B * H;
    out->x_mid = y.pX1 + 2 * l * B * H;
    out->gate_up = y.pGU + 2 * l * B * 2 * F;
    out->act = y.pM + 2 * l * B * F;
    out->down = y.pD + 2 * l * B * H;
    out->x_out = y.pX2 + 2 * l * B * H;
    if (attn_heads_ok(d)) {
        // decode step: the attention regions come after the chain's, and their
        // offsets do not depend on the size of wq4_paged_attention's workspace
        const Layout ya = make_layout(d, true, 0);
        const size_t KD = static_cast<size_t>(d.Hkv) * kAttnD;
        out->q_rot = ya.pQr + 2 * l * B * H;
        out->k_rot = ya.pKr + 2 * l * B * KD;
        out->attn = ya.pAt + 2 * l * B * H;
    }
    return WQ4_OK;
}

// ------------------------------------------------- allocation-free variant --
//
// wq4_decode_chain_noalloc: the same persistent chain kernel, with its
// workspace in a fixed device array of this library instead of a buffer the
// caller allocates.  For callers that cannot call cudaMalloc themselves.

namespace wq4 {
namespace {

constexpr size_t kNoAllocScratchBytes = static_cast<size_t>(WQ4_NOALLOC_SCRATCH_BYTES);
constexpr int kNoAllocMaxDevices = 64;

// Every device that loads the library holds this array until the process
// exits.  Host code may not use its name as an address: the address comes
// from cudaGetSymbolAddress, once per device.
static __device__ __align__(256) uint8_t g_noalloc_scratch[kNoAllocScratchBytes];

struct NoAllocDevice {
    bool ready = false;
    void* scratch = nullptr;          // device address of g_noalloc_scratch
    wq4_layer_table table = {};       // the caller's table, pointed at the scratch
};

NoAllocDevice g_noalloc[kNoAllocMaxDevices];
std::mutex g_noalloc_mu;

}  // namespace
}  // namespace wq4

extern "C" int wq4_decode_chain_noalloc(const wq4_layer_table* table, const uint16_t* x, uint16_t* logits,
                                        void* stream)
{
    if (!table || !x || !logits) return WQ4_ERR_INVALID;
    if (!aligned(x, 16) || !aligned(logits, 2)) return WQ4_ERR_ALIGN;
    Dims d;
    if (!table_dims(table, &d)) return WQ4_ERR_INVALID;
    if (make_layout(d).total > kNoAllocScratchBytes) return WQ4_ERR_UNSUPPORTED;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return WQ4_ERR_CUDA;
    if (dev < 0 || dev >= kNoAllocMaxDevices) return WQ4_ERR_UNSUPPORTED;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    NoAllocDevice& nd = g_noalloc[dev];
    if (!nd.ready) {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr) return WQ4_ERR_CUDA;
        nd.scratch = p;
        nd.ready = true;
    }
    // One table object per device stands for "whoever uses the array now":
    // a call with another model changes its contents, so the cached plan is
    // rebuilt and the array's flags and counters are cleared again.
    nd.table = *table;
    nd.table.workspace = nd.scratch;
    nd.table.workspace_bytes = kNoAllocScratchBytes;
    Plan pl;
    const int rc = get_plan(&nd.table, nullptr, &pl, st, true);
    if (rc != WQ4_OK) return rc;
    const size_t lb = static_cast<size_t>(pl.dims.B) * pl.dims.V * 2;
    if (overlaps(logits, lb, x, static_cast<size_t>(pl.dims.B) * pl.dims.H * 2)) return WQ4_ERR_INVALID;
    return launch_chain(pl, x, logits, st);
}
