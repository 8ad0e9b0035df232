// wq4_chain.cu -- one decoded token through every projection of every layer
// and the LM head, as one persistent kernel (the per-token GPU work whose
// throughput Table 1 of Section 3 reports).
//
// Structure (GB300-first; the paper's WebGPU engine launches one compiled
// kernel per operator, Section 2.3):
//  * One CTA per SM, co-resident (cooperative launch).  Each CTA owns a fixed
//    slice of the output rows of every stage (QKV, O, gate_up, down per layer,
//    then the LM head).
//  * A producer warp walks the CTA's slices of ALL stages in order and streams
//    their packed weights through a ring of shared-memory slots with 1-D bulk
//    copies (TMA) and mbarriers.  Weights do not depend on activations, so the
//    stream runs ahead across stage boundaries and HBM keeps working while the
//    consumers wait for the next activation vector.
//  * Each layer re-feeds its input after RMS normalisation.  Every CTA
//    computes the same factor in the same order (identical bits everywhere),
//    applies it as a row factor of its projection, and publishes its slice of
//    the normalised vector for the O stage's residual add.
//  * Consumer warps stage each stage's input vector in shared memory, take
//    two-row items (four rows for gate_up: gate j, j+1 and up j, j+1)
//    round-robin, unpack in registers, accumulate in fp32, and apply the
//    fused epilogue (RMS factor, residual add, SiLU(gate) * up).
//  * Stage outputs travel between CTAs as 8-byte words {2 x fp16 data, 32-bit
//    token epoch} written with single 64-bit stores; a consumer polls the
//    words of its input until every epoch matches.  No grid-wide barrier and
//    no separate flag round trip: one L2 round trip per stage boundary.
//    Every poll is bounded in time.
//  * Plain fp16 copies of every stage output are written to the workspace for
//    inspection.
#include "wq4_device.cuh"
#include "wq4_host.h"
#include "wq4_tc_host.h"
#include "wq4.h"

#include <cuda_runtime.h>

#include <cmath>
#include <cstring>
#include <map>
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
// RMS partial sums | epoch | the residual
// words of the CTA's rows (O and down stages); then the staged input vector,
// then the weight ring.
constexpr int kHdrRed = 512;                 // float red[kMaxChainBatch][16]: per-warp sums of squares
static_assert(8 * (kFullBars + kChainMaxSlots) <= kHdrRed, "mbarriers overlap the header");
constexpr int kHdrEpoch = 768;               // uint32 epoch, then int vw0, vw1 (the CTA's slice of v)
constexpr int kHdrInfo = 784;                // StageInfo info[5], one per stage type
constexpr int kHdrWofs = 944;                // uint8 wofs[5][16]: a warp's first chunk within a stage
constexpr int kHdrRes = 1024;                // uint32 res[kMaxResWords]: prefetched residual words
constexpr int kMaxResWords = 1024;
__host__ __device__ constexpr int chain_header_bytes(int, int)
{
    return kHdrRes + 4 * kMaxResWords;
}

// Consumer warps per CTA: with the producer warp, 16 warps (128 registers a
// thread).
template <int B>
struct ChainWarps {
    static constexpr int NW = 15;
};

enum StageType { kQKV = 0, kO = 1, kGU = 2, kDOWN = 3, kLM = 4 };

struct DevMat {
    const uint32_t* W;
    const uint16_t* s;
};

struct ChainParams {
    const DevMat* mats;  // [4L + 1]: per layer qkv, o, gate_up, down; then lm_head
    int L, H, F, Nqkv, V;
    float eps;
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
};

struct Stage {
    int type, layer, N, K, rpi, items;
    const uint32_t* W;
    const uint16_t* s;
};

__device__ __forceinline__ Stage stage_at(const ChainParams& p, int st)
{
    Stage g;
    if (st == 4 * p.L) {
        g.type = kLM; g.layer = p.L; g.N = p.V; g.K = p.H; g.rpi = 4; g.items = (p.V + 3) / 4;
    } else {
        g.layer = st >> 2;
        g.type = st & 3;
        switch (g.type) {
            case kQKV: g.N = p.Nqkv; g.K = p.H; g.rpi = 2; g.items = p.Nqkv / 2; break;
            case kO: g.N = p.H; g.K = p.H; g.rpi = 2; g.items = p.H / 2; break;
            case kGU: g.N = 2 * p.F; g.K = p.H; g.rpi = 4; g.items = p.F / 2; break;
            default: g.N = p.H; g.K = p.F; g.rpi = 2; g.items = p.H / 2; break;
        }
    }
    g.W = p.mats[st].W;
    g.s = p.mats[st].s;
    return g;
}

// Byte layout of one chunk (items [ia, ib) of a stage) inside a slot.
struct ChunkLayout {
    int nrows;          // rows in the chunk (both halves for gate_up)
    int nh;             // rows per half (gate_up) / nrows otherwise
    uint32_t codes_bytes, scale_bytes;
};

__device__ __forceinline__ ChunkLayout chunk_layout(const Stage& g, int ia, int ib)
{
    ChunkLayout c;
    if (g.type == kGU) {
        c.nh = 2 * (ib - ia);
        c.nrows = 2 * c.nh;
    } else {
        const int r1 = min(g.rpi * ib, g.N);
        c.nrows = r1 - g.rpi * ia;
        c.nh = c.nrows;
    }
    c.codes_bytes = static_cast<uint32_t>(c.nrows) * (g.K / 2);
    c.scale_bytes = static_cast<uint32_t>(c.nrows) * (g.K / 16);
    return c;
}

// What one CTA does in every stage of one type, computed once per launch so
// that no stage pays for integer divisions: items [i0, i1), items per ring
// slot, the number of chunks, and that number modulo the slot and barrier
// counts (flip: parity changes of the barrier ring beyond the wrap).
struct StageInfo {
    int i0, i1, ips, nchunks, nmod_slots, nmod_bars, flip, pad;
};
static_assert(kHdrInfo + 5 * sizeof(StageInfo) <= kHdrWofs, "stage table overlaps the header");
static_assert(kHdrWofs + 5 * 16 <= kHdrRes, "warp table overlaps the header");

__device__ __forceinline__ void cta_items(int items, int* i0, int* i1)
{
    *i0 = static_cast<int>(static_cast<int64_t>(blockIdx.x) * items / gridDim.x);
    *i1 = static_cast<int>(static_cast<int64_t>(blockIdx.x + 1) * items / gridDim.x);
}

__device__ __forceinline__ int items_per_slot(const ChainParams& p, const Stage& g)
{
    const uint32_t item_bytes = static_cast<uint32_t>(g.rpi) * (g.K / 2 + g.K / 16);
    const int ips = static_cast<int>(p.slot_bytes / item_bytes);
    return ips < 1 ? 1 : ips;
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

// A wait gives up after kWaitTimeoutNs, or at once when another CTA already
// gave up on this token; the first to give up records the token in *abort.
__device__ __forceinline__ bool gave_up(uint64_t t0, uint32_t epoch, uint32_t* abort)
{
    if (*reinterpret_cast<const volatile uint32_t*>(abort) == epoch) return true;
    if (globaltimer_ns() - t0 > kWaitTimeoutNs) {
        atomicExch(abort, epoch);
        return true;
    }
    return false;
}

// Four consecutive flagged words (8 fp16 values) at a 32-byte aligned address;
// polls until all four carry `epoch`.
__device__ __forceinline__ uint4 ll_load4(const uint64_t* addr, uint32_t epoch, uint32_t* err, uint32_t* abort)
{
    uint64_t a, b, c, d;
    ll_load2_raw(addr, a, b);
    ll_load2_raw(addr + 2, c, d);
    if (static_cast<uint32_t>(a >> 32) != epoch || static_cast<uint32_t>(b >> 32) != epoch ||
        static_cast<uint32_t>(c >> 32) != epoch || static_cast<uint32_t>(d >> 32) != epoch) {
        const uint64_t t0 = globaltimer_ns();
        for (uint32_t it = 0;; ++it) {
            ll_load2_raw(addr, a, b);
            ll_load2_raw(addr + 2, c, d);
            if (static_cast<uint32_t>(a >> 32) == epoch && static_cast<uint32_t>(b >> 32) == epoch &&
                static_cast<uint32_t>(c >> 32) == epoch && static_cast<uint32_t>(d >> 32) == epoch)
                break;
            if ((it & 63) == 63 && gave_up(t0, epoch, abort)) {
                atomicOr(err, kErrFlagTimeout);
                break;
            }
        }
    }
    return make_uint4(static_cast<uint32_t>(a), static_cast<uint32_t>(b), static_cast<uint32_t>(c),
                      static_cast<uint32_t>(d));
}

__device__ __forceinline__ uint32_t ll_load(const uint64_t* addr, uint32_t epoch, uint32_t* err, uint32_t* abort)
{
    uint64_t a = ll_load1_raw(addr);
    if (static_cast<uint32_t>(a >> 32) != epoch) {
        const uint64_t t0 = globaltimer_ns();
        for (uint32_t it = 0;; ++it) {
            a = ll_load1_raw(addr);
            if (static_cast<uint32_t>(a >> 32) == epoch) break;
            if ((it & 63) == 63 && gave_up(t0, epoch, abort)) {
                atomicOr(err, kErrFlagTimeout);
                break;
            }
        }
    }
    return static_cast<uint32_t>(a);
}

__device__ __forceinline__ float lo_f(uint32_t v) { return half_bits_to_float(static_cast<uint16_t>(v & 0xFFFFu)); }
__device__ __forceinline__ float hi_f(uint32_t v) { return half_bits_to_float(static_cast<uint16_t>(v >> 16)); }
__device__ __forceinline__ uint32_t pack2(uint16_t a, uint16_t b)
{
    return static_cast<uint32_t>(a) | (static_cast<uint32_t>(b) << 16);
}
// fp16(a + b): the fp32 sum of two fp16 values rounded to fp16 equals the
// correctly rounded fp16 sum (fp32 carries more than 2 * 11 + 2 bits).
__device__ __forceinline__ uint16_t add_h(float a, float b) { return float_to_half_bits(a + b); }

// fp16(r * v_i) for the 8 fp16 values of a chunk
__device__ __forceinline__ uint4 scale8(uint4 v, float r)
{
    uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int i = 0; i < 4; ++i)
        w[i] = pack2(float_to_half_bits(r * lo_f(w[i])), float_to_half_bits(r * hi_f(w[i])));
    return make_uint4(w[0], w[1], w[2], w[3]);
}

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

// ---------------------------------------------------------- the kernel --

// One group (32 codes) of every row of an item against the staged
// activations.  crow/srow point at the lane's first group of each row, xl at
// the lane's first group of activation row 0; `off` is the group offset
// (a multiple of 32, so the lane's chunk swizzle `sw` does not change).  The
// activations are loaded once and used for every row; each row's 32 products
// go into two 16-long fp32 chains before the group's scale is applied.
template <int B, int RPI>
__device__ __forceinline__ void group_rows_dot(const uint4* const crow[4], const uint16_t* const srow[4],
                                               const uint4* xl, int cpr, int sw, int off, float acc[4][B])
{
    uint4 xv[B][4];
#pragma unroll
    for (int b = 0; b < B; ++b)
#pragma unroll
        for (int j = 0; j < 4; ++j) xv[b][j] = xl[b * cpr + 4 * off + (j ^ sw)];
#pragma unroll
    for (int r = 0; r < RPI; ++r) {
        const uint4 cw = crow[r][off];
        const float sc = half_bits_to_float(srow[r][off]);
        uint32_t q[16];
        unpack_word(cw.x, q + 0);
        unpack_word(cw.y, q + 4);
        unpack_word(cw.z, q + 8);
        unpack_word(cw.w, q + 12);
#pragma unroll
        for (int b = 0; b < B; ++b) {
            const float a01 = fma8(q + 4, xv[b][1], fma8(q + 0, xv[b][0], 0.f));
            const float a23 = fma8(q + 12, xv[b][3], fma8(q + 8, xv[b][2], 0.f));
            acc[r][b] = fmaf(sc, a01 + a23, acc[r][b]);
        }
    }
}

// Every group of the item's rows: lane l takes groups l + 32 i.  Rows of 96,
// 128 or 256 groups (K = 3072, 4096, 8192) run fully unrolled (all loads of
// the item can be issued ahead of its arithmetic); other lengths take a loop
// and a tail.
template <int B, int RPI>
__device__ __forceinline__ void item_dot(const uint4* const crow[4], const uint16_t* const srow[4],
                                         const uint4* xl, int cpr, int gpr, int lane, float acc[4][B])
{
    const int sw = (lane >> 1) & 3;
    switch (gpr) {
        case 96:
#pragma unroll
            for (int i = 0; i < 3; ++i) group_rows_dot<B, RPI>(crow, srow, xl, cpr, sw, 32 * i, acc);
            return;
        case 128:
#pragma unroll
            for (int i = 0; i < 4; ++i) group_rows_dot<B, RPI>(crow, srow, xl, cpr, sw, 32 * i, acc);
            return;
        case 256:
#pragma unroll
            for (int i = 0; i < 8; ++i) group_rows_dot<B, RPI>(crow, srow, xl, cpr, sw, 32 * i, acc);
            return;
        default: {
            const int full = gpr >> 5;
#pragma unroll 2
            for (int i = 0; i < full; ++i) group_rows_dot<B, RPI>(crow, srow, xl, cpr, sw, 32 * i, acc);
            if (lane < (gpr & 31)) group_rows_dot<B, RPI>(crow, srow, xl, cpr, sw, 32 * full, acc);
        }
    }
}

// Fused epilogue of one item for batch row b: v0..v3 are the item's row sums
// (rows 2it, 2it+1; gate_up: gate 2it, 2it+1 then up 2it, 2it+1; LM head:
// rows 4it .. 4it+3); resw is
// the item's residual word (O: the normalised layer input, down: x + o).
template <int B>
__device__ __forceinline__ void item_epilogue(const ChainParams& p, const Stage& g, int it, int b, float v0,
                                              float v1, float v2, float v3, float rf, uint32_t resw, uint32_t epoch)
{
    const int H = p.H, F = p.F, l = g.layer;
    const int n = 2 * it;
    if (g.type == kQKV) {
        const uint32_t w = pack2(float_to_half_bits(rf * v0), float_to_half_bits(rf * v1));
        *reinterpret_cast<uint32_t*>(p.pQKV + (static_cast<size_t>(l) * B + b) * p.Nqkv + n) = w;
        if (n < H) ll_store(p.llA + (static_cast<size_t>(l) * B + b) * (H / 2) + n / 2, w, epoch);
    } else if (g.type == kO) {
        const uint16_t o0 = float_to_half_bits(rf * v0);
        const uint16_t o1 = float_to_half_bits(rf * v1);
        const uint32_t x1 = pack2(add_h(lo_f(resw), half_bits_to_float(o0)), add_h(hi_f(resw), half_bits_to_float(o1)));
        const size_t off = (static_cast<size_t>(l) * B + b) * H + n;
        *reinterpret_cast<uint32_t*>(p.pO + off) = pack2(o0, o1);
        *reinterpret_cast<uint32_t*>(p.pX1 + off) = x1;
        ll_store(p.llX1 + (static_cast<size_t>(l) * B + b) * (H / 2) + n / 2, x1, epoch);
    } else if (g.type == kGU) {
        const int j = n;  // gate rows j, j+1 and up rows F+j, F+j+1
        const uint16_t g0 = float_to_half_bits(rf * v0);
        const uint16_t g1 = float_to_half_bits(rf * v1);
        const uint16_t u0 = float_to_half_bits(rf * v2);
        const uint16_t u1 = float_to_half_bits(rf * v3);
        const float gf0 = half_bits_to_float(g0), gf1 = half_bits_to_float(g1);
        const uint16_t m0 = float_to_half_bits(gf0 / (1.f + expf(-gf0)) * half_bits_to_float(u0));
        const uint16_t m1 = float_to_half_bits(gf1 / (1.f + expf(-gf1)) * half_bits_to_float(u1));
        const size_t gu = (static_cast<size_t>(l) * B + b) * (2 * F);
        *reinterpret_cast<uint32_t*>(p.pGU + gu + j) = pack2(g0, g1);
        *reinterpret_cast<uint32_t*>(p.pGU + gu + F + j) = pack2(u0, u1);
        const uint32_t mw = pack2(m0, m1);
        *reinterpret_cast<uint32_t*>(p.pM + (static_cast<size_t>(l) * B + b) * F + j) = mw;
        ll_store(p.llM + (static_cast<size_t>(l) * B + b) * (F / 2) + j / 2, mw, epoch);
    } else if (g.type == kDOWN) {
        const uint16_t d0 = float_to_half_bits(v0);
        const uint16_t d1 = float_to_half_bits(v1);
        const uint32_t x2 = pack2(add_h(lo_f(resw), half_bits_to_float(d0)), add_h(hi_f(resw), half_bits_to_float(d1)));
        *reinterpret_cast<uint32_t*>(p.pD + (static_cast<size_t>(l) * B + b) * H + n) = pack2(d0, d1);
        *reinterpret_cast<uint32_t*>(p.pX2 + (static_cast<size_t>(l) * B + b) * H + n) = x2;
        ll_store(p.llX + (static_cast<size_t>(l + 1) * B + b) * (H / 2) + n / 2, x2, epoch);
    } else {
        const int n4 = 4 * it;   // the LM head's items are 4 rows
        uint16_t* out = p.logits + static_cast<size_t>(b) * p.V + n4;
        const int nv = p.V - n4;
        out[0] = float_to_half_bits(rf * v0);
        if (nv > 1) out[1] = float_to_half_bits(rf * v1);
        if (nv > 2) out[2] = float_to_half_bits(rf * v2);
        if (nv > 3) out[3] = float_to_half_bits(rf * v3);
    }
}

template <int B, int NW>
__global__ void __launch_bounds__((NW + 1) * 32, 1) chain_kernel(const ChainParams p)
{
    extern __shared__ __align__(1024) uint8_t smem[];
    uint64_t* full = reinterpret_cast<uint64_t*>(smem);
    uint64_t* empty = full + kFullBars;
    float* red = reinterpret_cast<float*>(smem + kHdrRed);          // [NW][kMaxChainBatch]
    uint32_t* epoch_sh = reinterpret_cast<uint32_t*>(smem + kHdrEpoch);
    uint32_t* res = reinterpret_cast<uint32_t*>(smem + kHdrRes);    // [B][items of the CTA]
    StageInfo* info = reinterpret_cast<StageInfo*>(smem + kHdrInfo);
    uint8_t* wofs_tab = smem + kHdrWofs;
    constexpr int kHeader = chain_header_bytes(NW, B);
    uint4* xs = reinterpret_cast<uint4*>(smem + kHeader);
    uint8_t* slots = smem + kHeader + p.x_bytes;
    constexpr int kConsumers = NW * 32;
    constexpr int kPoll = 2;     // input chunks a thread has in flight at once

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
    if (threadIdx.x < kMaxChainBatch * 16) red[threadIdx.x] = 0.f;   // warps >= NW stay zero
    if (threadIdx.x >= 32 && threadIdx.x < 32 + 5) {
        const int t = threadIdx.x - 32;
        const Stage g = stage_at(p, stage_of_type(p, t));
        StageInfo in;
        cta_items(g.items, &in.i0, &in.i1);
        in.ips = items_per_slot(p, g);
        in.nchunks = (in.i1 - in.i0 + in.ips - 1) / in.ips;
        in.nmod_slots = in.nchunks % p.nslots;
        in.nmod_bars = in.nchunks % p.nbars;
        in.flip = (in.nchunks / p.nbars) & 1;
        in.pad = 0;
        info[t] = in;
    }
    if (threadIdx.x >= 64 && threadIdx.x < 64 + 5 * 16) {
        const int t = (threadIdx.x - 64) >> 4, w = (threadIdx.x - 64) & 15;
        wofs_tab[t * 16 + w] = static_cast<uint8_t>(w / items_per_slot(p, stage_at(p, stage_of_type(p, t))));
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
                const int i0 = in.i0, i1 = in.i1, ips = in.ips;
                const int wpr = g.K >> 3, gpr = g.K >> 5;
                for (int ia = i0; ia < i1; ia += ips, ++ord) {
                    const int ib = min(i1, ia + ips);
                    if (round > 0) mbar_wait(&empty[slot], (round - 1) & 1, p.err);
                    const ChunkLayout c = chunk_layout(g, ia, ib);
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
                        bulk_g2s(dst, g.W + static_cast<size_t>(2 * ia) * wpr, hc, fb, pol);
                        bulk_g2s(dst + hc, g.W + (up + 2 * ia) * wpr, hc, fb, pol);
                        bulk_g2s(dst + c.codes_bytes, g.s + static_cast<size_t>(2 * ia) * gpr, hs, fb, pol);
                        bulk_g2s(dst + c.codes_bytes + hs, g.s + (up + 2 * ia) * gpr, hs, fb, pol);
                    } else {
                        bulk_g2s(dst, g.W + static_cast<size_t>(g.rpi * ia) * wpr, c.codes_bytes, fb, pol);
                        bulk_g2s(dst + c.codes_bytes, g.s + static_cast<size_t>(g.rpi * ia) * gpr, c.scale_bytes,
                                 fb, pol);
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
        // slot, full barrier and barrier parity of the stage's first chunk
        int cslot = 0, cbar = 0;
        uint32_t cpar = 0;
        for (int st = 0; st < nstages; ++st) {
            const Stage g = stage_at(p, st);
            const StageInfo& in = info[g.type];
            const int i0 = in.i0, i1 = in.i1;
            if (i1 <= i0) continue;
            const int l = g.layer;
            const int K = g.K, gpr = K >> 5, cpr = K >> 3;
            const int nit = i1 - i0;

            // -- stage the input vector (all consumer warps), its RMS factor and
            //    the residual words of the CTA's rows
            named_barrier_sync(1, kConsumers);   // every warp is done with the previous xs and res
            {
                const uint64_t* ll = nullptr;
                const bool plain = (g.type == kQKV && l == 0);
                if (g.type == kQKV) ll = p.llX + static_cast<size_t>(l) * B * (H / 2);
                else if (g.type == kO) ll = p.llA + static_cast<size_t>(l) * B * (H / 2);
                else if (g.type == kGU) ll = p.llX1 + static_cast<size_t>(l) * B * (H / 2);
                else if (g.type == kDOWN) ll = p.llM + static_cast<size_t>(l) * B * (F / 2);
                else ll = p.llX + static_cast<size_t>(p.L) * B * (H / 2);
                const uint64_t* rl = nullptr;
                if (g.type == kO) rl = p.llV + static_cast<size_t>(l) * B * (H / 2);
                else if (g.type == kDOWN) rl = p.llX1 + static_cast<size_t>(l) * B * (H / 2);
                if (rl) {
#pragma unroll
                    for (int b = 0; b < B; ++b)
                        for (int k = threadIdx.x; k < nit; k += kConsumers)
                            res[b * nit + k] = ll_load(rl + static_cast<size_t>(b) * (H / 2) + i0 + k, epoch, p.err, p.abort);
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
                                for (int j = 0; j < 4; ++j) ok = ok && static_cast<uint32_t>(w[k][j] >> 32) == epoch;
                                if (ok) {
                                    v[k] = make_uint4(static_cast<uint32_t>(w[k][0]), static_cast<uint32_t>(w[k][1]),
                                                      static_cast<uint32_t>(w[k][2]), static_cast<uint32_t>(w[k][3]));
                                } else {
                                    const int b = i / cpr, c = i - b * cpr;
                                    v[k] = ll_load4(ll + static_cast<size_t>(b) * (K / 2) + 4 * c, epoch, p.err, p.abort);
                                }
                            }
                        }
                    }
#pragma unroll
                    for (int k = 0; k < kPoll; ++k) {
                        const int i = ib + k * kConsumers;
                        if (i < total) {
                            const int b = i / cpr, c = i - b * cpr;
                            xs[b * cpr + x_chunk(c >> 2, c & 3)] = v[k];
#pragma unroll
                            for (int bb = 0; bb < B; ++bb)
                                if (bb == b) ss[bb] += sum8_sq(v[k]);
                        }
                    }
                }
#pragma unroll
                for (int b = 0; b < B; ++b) {
                    const float v = warp_sum(ss[b]);
                    if (lane == 0) red[b * 16 + warp] = v;
                }
            }
            named_barrier_sync(1, kConsumers);
            float rf[B];
#pragma unroll
            for (int b = 0; b < B; ++b) {
                // the same sum, in the same order, in every warp and every CTA
                const float4* r4 = reinterpret_cast<const float4*>(red + b * 16);
                const float4 a = r4[0], c = r4[1], d = r4[2], e = r4[3];
                const float t = (((a.x + a.y) + (a.z + a.w)) + ((c.x + c.y) + (c.z + c.w))) +
                                (((d.x + d.y) + (d.z + d.w)) + ((e.x + e.y) + (e.z + e.w)));
                rf[b] = (g.type == kDOWN) ? 1.f : rsqrtf(t * (1.f / static_cast<float>(K)) + p.eps);
            }
            if (g.type == kQKV || g.type == kLM) {
                // the normalised layer input v = fp16(r * u) is kept for the
                // residual stream (and the trace): every CTA publishes its
                // slice of it; the projections below use r as a row factor
                const int w0 = static_cast<int>(epoch_sh[1]), w1 = static_cast<int>(epoch_sh[2]);
                const uint32_t* xw = reinterpret_cast<const uint32_t*>(xs);
#pragma unroll
                for (int b = 0; b < B; ++b) {
                    for (int w = w0 + threadIdx.x; w < w1; w += kConsumers) {
                        const int c = w >> 2;               // chunk of the word
                        const uint32_t u = xw[4 * (b * cpr + x_chunk(c >> 2, c & 3)) + (w & 3)];
                        const uint32_t v = pack2(float_to_half_bits(rf[b] * lo_f(u)), float_to_half_bits(rf[b] * hi_f(u)));
                        reinterpret_cast<uint32_t*>(p.pV + (static_cast<size_t>(l) * B + b) * H)[w] = v;
                        if (g.type == kQKV) ll_store(p.llV + (static_cast<size_t>(l) * B + b) * (H / 2) + w, v, epoch);
                    }
                }
            }

            // -- stream the CTA's items of this stage: item i0 + k goes to warp
            //    k % NW; a warp visits only the chunks that hold its items
            const int ips = in.ips;
            const uint4* xl = xs + 4 * lane;
            int it = i0 + warp;
            if (it < i1) {
                // the warp's first chunk: wofs chunks after the stage's first
                const int wofs = wofs_tab[g.type * 16 + warp];
                int ia = i0 + wofs * ips, ib = min(i1, ia + ips);
                int slot = cslot + wofs;
                while (slot >= p.nslots) slot -= p.nslots;
                int bar = cbar + wofs;                      // wofs < nbars
                uint32_t par = cpar;
                if (bar >= p.nbars) {
                    bar -= p.nbars;
                    par ^= 1u;
                }
                while (it < i1) {
                    while (it >= ib) {                      // next chunk
                        ia += ips;
                        ib = min(i1, ia + ips);
                        if (++slot == p.nslots) slot = 0;
                        if (++bar == p.nbars) {
                            bar = 0;
                            par ^= 1u;
                        }
                    }
                    mbar_wait(&full[bar], par, p.err);
                    const uint8_t* base = slots + static_cast<size_t>(slot) * p.slot_bytes;
                    const ChunkLayout c = chunk_layout(g, ia, ib);
                    uint32_t arrivals = (it == ia) ? kSlotRelease - static_cast<uint32_t>(ib - ia) : 0u;
                    for (; it < ib; it += NW) {
                        ++arrivals;
                        const int ii = it - ia;        // item within the chunk
                        const uint4* crow[4];
                        const uint16_t* srow[4];
                        if (g.type == kGU) {
#pragma unroll
                            for (int r = 0; r < 4; ++r) {
                                const int half = r >> 1, rr = 2 * ii + (r & 1);
                                crow[r] = reinterpret_cast<const uint4*>(base + static_cast<size_t>(half) * (c.codes_bytes / 2) +
                                                                         static_cast<size_t>(rr) * (K / 2)) + lane;
                                srow[r] = reinterpret_cast<const uint16_t*>(base + c.codes_bytes + half * (c.scale_bytes / 2) +
                                                                            rr * (K / 16)) + lane;
                            }
                        } else {
                            // rows rpi*it .. rpi*it + rpi - 1; rows past N repeat the first
                            const int nvalid = min(g.rpi, g.N - g.rpi * it);
#pragma unroll
                            for (int r = 0; r < 4; ++r) {
                                const int rr = g.rpi * ii + (r < nvalid ? r : 0);
                                crow[r] = reinterpret_cast<const uint4*>(base + static_cast<size_t>(rr) * (K / 2)) + lane;
                                srow[r] = reinterpret_cast<const uint16_t*>(base + c.codes_bytes + rr * (K / 16)) + lane;
                            }
                        }
                        float acc[4][B];
#pragma unroll
                        for (int r = 0; r < 4; ++r)
#pragma unroll
                            for (int b = 0; b < B; ++b) acc[r][b] = 0.f;
                        if (g.rpi == 4) item_dot<B, 4>(crow, srow, xl, cpr, gpr, lane, acc);
                        else item_dot<B, 2>(crow, srow, xl, cpr, gpr, lane, acc);
#pragma unroll
                        for (int r = 0; r < 4; ++r)
#pragma unroll
                            for (int b = 0; b < B; ++b)
                                if (r < g.rpi) acc[r][b] = warp_sum(acc[r][b]);
#pragma unroll
                        for (int b = 0; b < B; ++b)
                            if (lane == b)
                                item_epilogue<B>(p, g, it, b, acc[0][b], acc[1][b], acc[2][b], acc[3][b], rf[b],
                                                 (g.type == kO || g.type == kDOWN) ? res[b * nit + (it - i0)] : 0u,
                                                 epoch);
                    }
                    __syncwarp();
                    if (lane == 0) mbar_arrive_count(&empty[slot], arrivals);
                }
            }
            cslot += in.nmod_slots;
            if (cslot >= p.nslots) cslot -= p.nslots;
            cbar += in.nmod_bars;
            cpar ^= static_cast<uint32_t>(in.flip);
            if (cbar >= p.nbars) {
                cbar -= p.nbars;
                cpar ^= 1u;
            }
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

// ---------------------------------------------------------------- host --

struct Layout {
    size_t header, mats, llA, llX1, llM, llX, llV, pV, pX2, pQKV, pO, pX1, pGU, pM, pD, x_stage, logits_stage, rfac,
        xpH0, xpH1, xpF, cnt, part, total;
    size_t ll_begin, ll_end;
};

struct Dims {
    int L, H, F, Nqkv, V, B;
};

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
    return true;
}

Layout make_layout(const Dims& d)
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
    y.mats = take(sizeof(DevMat) * (4 * L + 1));
    y.ll_begin = o;
    y.llA = take(8 * L * B * (H / 2));
    y.llX1 = take(8 * L * B * (H / 2));
    y.llM = take(8 * L * B * (F / 2));
    y.llX = take(8 * (L + 1) * B * (H / 2));
    y.llV = take(8 * L * B * (H / 2));
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
    cudaGraphExec_t graph;   // graph path (batch > kMaxChainBatch), else null
};

std::mutex g_plan_mu;
std::map<const wq4_layer_table*, Plan> g_plans;

bool same_contents(const Plan& pl, const wq4_layer_table* t)
{
    if (std::memcmp(&pl.table, t, sizeof(*t)) != 0) return false;
    return std::memcmp(pl.layers.data(), t->layers, sizeof(wq4_layer) * t->num_layers) == 0;
}

bool mat_ok(const wq4_mat& m)
{
    return m.W && m.s && aligned(m.W, 16) && aligned(m.s, 16);
}

template <int B>
cudaError_t set_chain_attr(int smem)
{
    return cudaFuncSetAttribute(chain_kernel<B, ChainWarps<B>::NW>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
}

int chain_warps(int B)
{
    switch (B) {
        case 1: return ChainWarps<1>::NW;
        case 2: return ChainWarps<2>::NW;
        default: return ChainWarps<2>::NW;
    }
}


// Slot size: a multiple of 128 bytes holding at least one item of every
// stage, chosen to waste the least ring space over the chain's byte mix.
uint32_t choose_slot_bytes(const Dims& d)
{
    struct S { size_t item, bytes; };
    const size_t rowH = static_cast<size_t>(d.H) / 2 + d.H / 16, rowF = static_cast<size_t>(d.F) / 2 + d.F / 16;
    const S st[5] = {{2 * rowH, static_cast<size_t>(d.Nqkv) * rowH},
                     {2 * rowH, static_cast<size_t>(d.H) * rowH},
                     {4 * rowH, static_cast<size_t>(2) * d.F * rowH},
                     {2 * rowF, static_cast<size_t>(d.H) * rowF},
                     {4 * rowH, static_cast<size_t>(d.V) * rowH}};
    size_t max_item = 0;
    for (const S& s : st) max_item = s.item > max_item ? s.item : max_item;
    size_t lo = align_up(max_item, 128);
    if (lo < 16384) lo = 16384;
    size_t best = lo;
    double best_waste = 1e300;
    for (size_t sb = lo; sb <= lo + 8192; sb += 128) {
        double waste = 0;
        for (const S& s : st) {
            const size_t ips = sb / s.item;
            waste += static_cast<double>(s.bytes) * (1.0 - static_cast<double>(ips * s.item) / sb);
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

// True when no consumer wait on the ring can alias: for every stage,
// nslots + ceil(NW / items per slot) <= the number of full barriers.
bool ring_ok(const Dims& d, int nslots, uint32_t slot_bytes, int nw)
{
    const size_t rowH = static_cast<size_t>(d.H) / 2 + d.H / 16, rowF = static_cast<size_t>(d.F) / 2 + d.F / 16;
    const size_t items[5] = {2 * rowH, 2 * rowH, 4 * rowH, 2 * rowF, 4 * rowH};
    for (size_t item : items) {
        size_t ips = slot_bytes / item;
        if (ips < 1) ips = 1;
        if (static_cast<size_t>(nslots) + (nw + ips - 1) / ips > static_cast<size_t>(full_bars(nslots))) return false;
    }
    return true;
}

// Records one token of the graph path on `cs`: every stage kernel of every
// layer, reading the token input from the workspace staging area and writing
// the logits to the workspace logits area.
int build_graph_plan(const wq4_layer_table* t, const Dims& d, const Layout& lay, int dev, const DeviceInfo* di,
                     Plan* pl, cudaStream_t stream)
{
    uint8_t* ws = static_cast<uint8_t*>(t->workspace);
    // the split stages' arrival counters start at zero (each stage leaves them so)
    if (cudaMemsetAsync(ws + lay.cnt, 0, 4 * static_cast<size_t>(kTcCounterWords), stream) != cudaSuccess)
        return WQ4_ERR_CUDA;
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
        const int rrec = tc_record_token(tc, cs);
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

int build_plan(const wq4_layer_table* t, Plan* pl, cudaStream_t stream)
{
    Dims d;
    if (!table_dims(t, &d)) return WQ4_ERR_INVALID;
    pl->graph = nullptr;
    for (int l = 0; l < d.L; ++l) {
        const wq4_layer& ly = t->layers[l];
        if (!mat_ok(ly.qkv) || !mat_ok(ly.o) || !mat_ok(ly.gate_up) || !mat_ok(ly.down)) return WQ4_ERR_INVALID;
    }
    if (!mat_ok(t->lm_head)) return WQ4_ERR_INVALID;
    const Layout lay = make_layout(d);
    if (!t->workspace || !aligned(t->workspace, 256)) return WQ4_ERR_ALIGN;
    if (t->workspace_bytes < lay.total) return WQ4_ERR_INVALID;
    int dev = 0;
    const DeviceInfo* di = current_device_info(&dev);
    if (!di) return WQ4_ERR_CUDA;
    if (d.B > kMaxChainBatch) {
        if (d.Nqkv % 8) return WQ4_ERR_UNSUPPORTED;   // the O stage reads qkv rows with 16-byte loads
        return build_graph_plan(t, d, lay, dev, di, pl, stream);
    }
    if (!di->coop_launch) return WQ4_ERR_UNSUPPORTED;
    const uint32_t x_bytes = static_cast<uint32_t>(align_up(static_cast<size_t>(d.B) * 2 * (d.H > d.F ? d.H : d.F), 128));
    const uint32_t slot_bytes = choose_slot_bytes(d);
    const int header = chain_header_bytes(chain_warps(d.B), d.B);
    const long avail = static_cast<long>(di->smem_optin) - header - static_cast<long>(x_bytes);
    int nslots = avail > 0 ? static_cast<int>(avail / slot_bytes) : 0;
    if (nslots > kChainMaxSlots) nslots = kChainMaxSlots;
    // fewer slots give more full barriers per slot: take the deepest ring
    // whose barriers cannot alias
    while (nslots >= 2 && !ring_ok(d, nslots, slot_bytes, chain_warps(d.B))) --nslots;
    if (nslots < 2) return WQ4_ERR_UNSUPPORTED;
    const size_t smem = header + x_bytes + static_cast<size_t>(nslots) * slot_bytes;
    // The limit is a property of the kernel, shared by every plan: set it to
    // the device maximum so that no plan's launch depends on which plan was
    // built last.
    cudaError_t e = cudaSuccess;
    switch (d.B) {
        case 1: e = set_chain_attr<1>(di->smem_optin); break;
        default: e = set_chain_attr<2>(di->smem_optin); break;
    }
    if (e != cudaSuccess) return WQ4_ERR_CUDA;

    std::vector<DevMat> mats(4 * static_cast<size_t>(d.L) + 1);
    for (int l = 0; l < d.L; ++l) {
        const wq4_layer& ly = t->layers[l];
        mats[4 * l + 0] = {ly.qkv.W, ly.qkv.s};
        mats[4 * l + 1] = {ly.o.W, ly.o.s};
        mats[4 * l + 2] = {ly.gate_up.W, ly.gate_up.s};
        mats[4 * l + 3] = {ly.down.W, ly.down.s};
    }
    mats[4 * d.L] = {t->lm_head.W, t->lm_head.s};
    uint8_t* ws = static_cast<uint8_t*>(t->workspace);
    // header (token counter) and every flagged word start at zero: epoch 0 never matches
    if (cudaMemsetAsync(ws + lay.header, 0, 256, stream) != cudaSuccess) return WQ4_ERR_CUDA;
    if (cudaMemsetAsync(ws + lay.ll_begin, 0, lay.ll_end - lay.ll_begin, stream) != cudaSuccess) return WQ4_ERR_CUDA;
    // pageable source: the call returns once the bytes are staged
    if (cudaMemcpyAsync(ws + lay.mats, mats.data(), sizeof(DevMat) * mats.size(), cudaMemcpyHostToDevice, stream) !=
        cudaSuccess)
        return WQ4_ERR_CUDA;

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
    pl->nw = chain_warps(d.B);
    // the residual words of a CTA's rows must fit in shared memory
    if (static_cast<long>((d.H / 2 + pl->grid - 1) / pl->grid) * d.B > kMaxResWords) return WQ4_ERR_UNSUPPORTED;
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
    ChainParams p;
    p.mats = reinterpret_cast<const DevMat*>(ws + y.mats);
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
    p.err = status_word();
    if (!p.err) return WQ4_ERR_CUDA;

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
    switch (pl.dims.B) {
        case 1: e = cudaLaunchKernelEx(&cfg, chain_kernel<1, ChainWarps<1>::NW>, p); break;
        case 2: e = cudaLaunchKernelEx(&cfg, chain_kernel<2, ChainWarps<2>::NW>, p); break;
        default: e = cudaLaunchKernelEx(&cfg, chain_kernel<2, ChainWarps<2>::NW>, p); break;
    }
    return e == cudaSuccess ? WQ4_OK : WQ4_ERR_CUDA;
}

// Finds (or builds) the plan of `t`; returns a copy to launch from.
int get_plan(const wq4_layer_table* t, Plan* out, cudaStream_t stream)
{
    if (!t) return WQ4_ERR_INVALID;
    Dims d;
    if (!table_dims(t, &d)) return WQ4_ERR_INVALID;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return WQ4_ERR_CUDA;
    std::lock_guard<std::mutex> lock(g_plan_mu);
    auto it = g_plans.find(t);
    if (it != g_plans.end() && it->second.device == dev && same_contents(it->second, t)) {
        *out = it->second;
        return WQ4_OK;
    }
    Plan pl;
    const int rc = build_plan(t, &pl, stream);
    if (rc != WQ4_OK) return rc;
    if (it != g_plans.end() && it->second.graph) {
        // a replaced graph may still run on the GPU: free it once it is done
        cudaStreamSynchronize(stream);
        cudaGraphExecDestroy(it->second.graph);
    }
    g_plans[t] = pl;
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
    const int rc = get_plan(table, &pl, st);
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
    int rc = get_plan(table, &pl, st);
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
    auto it = g_plans.find(table);
    if (it == g_plans.end()) return WQ4_ERR_INVALID;
    if (it->second.graph) cudaGraphExecDestroy(it->second.graph);
    g_plans.erase(it);
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
    const int rc = get_plan(&nd.table, &pl, st);
    if (rc != WQ4_OK) return rc;
    const size_t lb = static_cast<size_t>(pl.dims.B) * pl.dims.V * 2;
    if (overlaps(logits, lb, x, static_cast<size_t>(pl.dims.B) * pl.dims.H * 2)) return WQ4_ERR_INVALID;
    return launch_chain(pl, x, logits, st);
}
