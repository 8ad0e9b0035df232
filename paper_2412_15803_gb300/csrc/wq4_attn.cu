// wq4_attn.cu -- decode attention over a paged key/value cache (sm_103a):
// the PagedAttention / FlashAttention step of the paper's compiled models
// (Section 2.3), one decode token per sequence, grouped-query heads.
//
// Work split.  The (sequence, kv head) pairs are laid end to end as one list
// of 16-token tiles; a persistent grid of CTAs (two per SM) takes equal
// contiguous shares of that list, so every CTA streams the same number of
// bytes whatever the length mix.  A share that covers only part of a pair's
// tiles produces a partial result (running maximum, normaliser, unnormalised
// output) in the workspace; the last CTA to finish a pair (arrival counter)
// merges the parts in their fixed order and writes the output.
//
// Inside a CTA one producer warp streams the tiles' keys and values into an
// 8-slot shared-memory ring with 2-D tensor copies (128-byte swizzle), and
// four consumer warps take the tiles round-robin.  For a tile a warp computes
// the G x 16 scores with mma.sync (query heads as the 16 rows, G <= 8 of them
// real), keeps the running maximum and normaliser per head in registers,
// rounds the weights to fp16 and accumulates weights x values (16 x 128) with
// mma.sync into fp32 registers.  The tensor cores here only keep the issue
// cost of the small contraction negligible; the kernel is bound by the HBM
// stream of keys and values (512 bytes per token and kv head).
#include "wq4.h"
#include "wq4_attn.h"
#include "wq4_device.cuh"
#include "wq4_host.h"

#include <cuda.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cstring>
#include <mutex>

namespace wq4 {
namespace {

constexpr int kD = 128;            // head_dim
constexpr int kTile = 16;          // tokens per tile
constexpr int kMaxGroup = 8;       // query heads per kv head
constexpr int kConsumers = 4;      // consumer warps
constexpr int kThreads = (kConsumers + 1) * 32;
constexpr int kSlots = 8;
constexpr int kSlotBytes = 2 * kTile * kD * 2;   // keys + values of one tile: 8 KiB
constexpr int kBoxBytes = kTile * 64 * 2;        // 16 rows x 64 dims: 2 KiB
constexpr int kPartHdr = 16;                     // floats: M[8], L[8]
constexpr int kCtasPerSm = 2;
constexpr int kMaxParts = kConsumers * kD;      // parts of one segment the merge stages: grid <= 512
constexpr int kMinShare = 16;                   // fewest tiles of a CTA's share (small batches: fewer parts to merge)

// Shared memory map (dynamic, base 1024-aligned).
constexpr int kOffRing = 0;
constexpr int kOffBars = kSlots * kSlotBytes;                     // full[S], empty[S]
constexpr int kOffMisc = kOffBars + 2 * kSlots * 8;               // ints: flags
constexpr int kOffMrow = kOffMisc + 64;                           // [W][8] floats
constexpr int kOffLrow = kOffMrow + kConsumers * kMaxGroup * 4;   // [W][8] floats
constexpr int kOffScr = kOffLrow + kConsumers * kMaxGroup * 4;    // [W][G][128] floats
constexpr int kOffPre = kOffScr + kConsumers * kMaxGroup * kD * 4;  // int [batch + 1]

size_t attn_smem_bytes(int batch)
{
    return 1024 + kOffPre + static_cast<size_t>(batch + 1) * 4;
}

struct AttnParams {
    CUtensorMap mk, mv;          // [rows = pages * kv heads * page_size][128] fp16, box 16 x 64, SW128
    const uint16_t* q;
    uint16_t* out;
    const int32_t* seq_lens;
    const int32_t* page_table;
    uint32_t* cnt;               // [batch * Hkv]
    float* part;                 // [grid + batch * Hkv][16 + G * 128]
    uint32_t* err;
    int q_stride, out_stride, pt_stride;
    int batch, Hkv, G, page_size, num_pages;
    float sl2;                   // scale * log2(e)
};

// ------------------------------------------------------------ device ---

__device__ __forceinline__ void tma_load_2d_hint(void* dst, const CUtensorMap* map, int x, int y, uint64_t* bar,
                                                 uint64_t policy)
{
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
        " [%0], [%1, {%2, %3}], [%4], %5;" ::"r"(smem_addr(dst)),
        "l"(map), "r"(x), "r"(y), "r"(smem_addr(bar)), "l"(policy)
        : "memory");
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t r[4])
{
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(addr));
}

__device__ __forceinline__ void ldsm_x4_trans(uint32_t addr, uint32_t r[4])
{
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(addr));
}

// D (16 x 8, fp32) += A (16 x 16, fp16, rows) * B (16 x 8, fp16, columns).
__device__ __forceinline__ void mma16816(float d[4], const uint32_t a[4], uint32_t b0, uint32_t b1)
{
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
        "{%0, %1, %2, %3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint32_t pack_half2(float lo, float hi)
{
    const __half2 h = __floats2half2_rn(lo, hi);
    return *reinterpret_cast<const uint32_t*>(&h);
}

__device__ __forceinline__ float2 unpack_half2(uint32_t v)
{
    return __half22float2(*reinterpret_cast<const __half2*>(&v));
}

// Byte offset of 16-byte chunk c (0..7) of row r in a 128-byte-swizzled box
// whose base is 1024-byte aligned.
__device__ __forceinline__ uint32_t sw128(int r, int c)
{
    return static_cast<uint32_t>(r * 128 + ((c ^ (r & 7)) << 4));
}

// One piece: tiles [t0, t1) of kv head h of sequence b (a contiguous run of
// one CTA's share inside one (sequence, head) segment).
struct Piece {
    int b, h, t0, t1;    // tile range within the sequence
    int seg;             // b * Hkv + h
    int npieces;         // CTAs sharing the segment
    int first;           // the first of them; piece p's partial sits in slot first + p + seg
    int slot;            // partial-result slot of this piece (unique: CTA index + segment index)
};

// Segment lookup over the tile list: pre[b] = tiles of sequences < b
// (exclusive prefix, pre[batch] = total / Hkv).  Segment (b, h) covers
// [Hkv * pre[b] + h * tiles_b, + tiles_b).
__device__ __forceinline__ Piece find_piece(const int* pre, int batch, int Hkv, int g, int end, int R, int cta)
{
    // largest b with Hkv * pre[b] <= g
    int lo = 0, hi = batch - 1;
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (Hkv * pre[mid] <= g) lo = mid;
        else hi = mid - 1;
    }
    Piece p;
    p.b = lo;
    const int tb = pre[lo + 1] - pre[lo];
    const int base = Hkv * pre[lo];
    p.h = (g - base) / tb;
    const int seg_start = base + p.h * tb;
    const int seg_end = seg_start + tb;
    const int pend = end < seg_end ? end : seg_end;
    p.t0 = g - seg_start;
    p.t1 = pend - seg_start;
    p.seg = p.b * Hkv + p.h;
    p.first = seg_start / R;
    p.npieces = (seg_end - 1) / R - p.first + 1;
    p.slot = cta + p.seg;
    return p;
}

__global__ void __launch_bounds__(kThreads, kCtasPerSm) paged_attn_kernel(const __grid_constant__ AttnParams P)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + kOffBars);
    uint64_t* empty = full + kSlots;
    volatile int* misc = reinterpret_cast<volatile int*>(smem + kOffMisc);   // [0] abort, [1] last arriver
    float* mrow = reinterpret_cast<float*>(smem + kOffMrow);
    float* lrow = reinterpret_cast<float*>(smem + kOffLrow);
    float* scr = reinterpret_cast<float*>(smem + kOffScr);
    int* pre = reinterpret_cast<int*>(smem + kOffPre);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int max_tok = P.pt_stride * P.page_size;

    // tile prefix over the batch (warp 0), barriers (thread 32)
    if (warp == 0) {
        int carry = 0;
        for (int b0 = 0; b0 < P.batch; b0 += 32) {
            const int b = b0 + lane;
            int tiles = 0;
            if (b < P.batch) {
                int T = P.seq_lens[b];
                if (T > max_tok) {
                    atomicOr(P.err, kErrSeqLen);
                    T = max_tok;
                }
                tiles = T > 0 ? (T + kTile - 1) / kTile : 0;
            }
            int incl = tiles;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int v = __shfl_up_sync(0xffffffffu, incl, o);
                if (lane >= o) incl += v;
            }
            if (b < P.batch) pre[b] = carry + incl - tiles;
            carry += __shfl_sync(0xffffffffu, incl, 31);
        }
        if (lane == 0) pre[P.batch] = carry;
    } else if (tid == 32) {
        for (int i = 0; i < kSlots; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], 1);
        }
        misc[0] = 0;
        misc[1] = 0;
        mbar_fence_init();
    }
    __syncthreads();

    const int total = P.Hkv * pre[P.batch];
    const int R = max((total + static_cast<int>(gridDim.x) - 1) / static_cast<int>(gridDim.x), kMinShare);
    const int cta = blockIdx.x;
    const int g_begin = min(total, cta * R);
    const int g_end = min(total, g_begin + R);
    const int G = P.G;

    if (warp == kConsumers) {
        // ---------------------------------------------------- producer --
        const uint64_t pol = l2_policy_evict_first();
        if (lane == 0) {
            asm volatile("prefetch.tensormap [%0];" ::"l"(&P.mk) : "memory");
            asm volatile("prefetch.tensormap [%0];" ::"l"(&P.mv) : "memory");
        }
        int i = 0;   // CTA-wide tile counter
        bool ok = true;
        for (int g = g_begin; g < g_end && ok;) {
            const Piece pc = find_piece(pre, P.batch, P.Hkv, g, g_end, R, cta);
            const int32_t* pt = P.page_table + static_cast<size_t>(pc.b) * P.pt_stride;
            for (int t = pc.t0; t < pc.t1 && ok; t += 32) {
                // page ids of up to 32 tiles, one per lane
                int mypage = -1, myrow = 0;
                const int tt = t + lane;
                if (tt < pc.t1) {
                    const int tok = tt * kTile;
                    mypage = pt[tok / P.page_size];
                    myrow = tok % P.page_size;
                }
                const int n = min(32, pc.t1 - t);
                for (int k = 0; k < n; ++k) {
                    const int page = __shfl_sync(0xffffffffu, mypage, k);
                    const int row = __shfl_sync(0xffffffffu, myrow, k);
                    if (lane == 0) {
                        const int slot = i % kSlots;
                        if (i >= kSlots && !mbar_wait(&empty[slot], ((i / kSlots) - 1) & 1, P.err)) {
                            misc[0] = 1;
                            ok = false;
                        } else {
                            int y;
                            if (page >= 0 && page < P.num_pages) {
                                y = (page * P.Hkv + pc.h) * P.page_size + row;
                            } else {
                                atomicOr(P.err, kErrPageId);
                                y = -kTile;   // wholly outside the tensor: the copy reads zeros
                            }
                            uint8_t* dst = smem + kOffRing + slot * kSlotBytes;
                            mbar_arrive_expect_tx(&full[slot], kSlotBytes);
                            tma_load_2d_hint(dst, &P.mk, 0, y, &full[slot], pol);
                            tma_load_2d_hint(dst + kBoxBytes, &P.mk, 64, y, &full[slot], pol);
                            tma_load_2d_hint(dst + 2 * kBoxBytes, &P.mv, 0, y, &full[slot], pol);
                            tma_load_2d_hint(dst + 3 * kBoxBytes, &P.mv, 64, y, &full[slot], pol);
                        }
                    }
                    ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
                    ++i;
                    if (!ok) break;
                }
            }
            g += pc.t1 - pc.t0;
        }
        // drain: the last copy issued into each slot has landed before exit
        if (lane == 0) {
            const int issued = i;
            for (int s = 0; s < kSlots && s < issued; ++s) {
                const int last = issued - 1 - ((issued - 1 - s) % kSlots);   // last tile index using slot s
                mbar_wait(&full[s], (last / kSlots) & 1, P.err);
            }
        }
        return;
    }

    // -------------------------------------------------------- consumers --
    // zero outputs of empty sequences handled by this CTA
    for (int b = cta; b < P.batch; b += gridDim.x) {
        if (pre[b + 1] == pre[b]) {
            uint16_t* ob = P.out + static_cast<size_t>(b) * P.out_stride;
            for (int e = tid; e < P.Hkv * G * kD; e += kConsumers * 32) ob[e] = 0;
        }
    }

    const int gq = lane >> 2;          // query-head row of this lane (0..7)
    const int qc = 2 * (lane & 3);     // column pair within 8
    const uint32_t ring = smem_addr(smem + kOffRing);
    int ibase = 0;                     // CTA-wide index of the piece's first tile
    for (int g = g_begin; g < g_end;) {
        const Piece pc = find_piece(pre, P.batch, P.Hkv, g, g_end, R, cta);
        const int ntile = pc.t1 - pc.t0;
        int T = P.seq_lens[pc.b];
        T = T > max_tok ? max_tok : T;

        // query fragments: rows = query heads of the group (rows >= G are 0)
        uint32_t qa[8][2];
        {
            const uint16_t* qrow = P.q + static_cast<size_t>(pc.b) * P.q_stride +
                                   static_cast<size_t>(pc.h * G + (gq < G ? gq : 0)) * kD;
#pragma unroll
            for (int ks = 0; ks < 8; ++ks) {
                const uint32_t v0 = *reinterpret_cast<const uint32_t*>(qrow + 16 * ks + qc);
                const uint32_t v1 = *reinterpret_cast<const uint32_t*>(qrow + 16 * ks + 8 + qc);
                qa[ks][0] = gq < G ? v0 : 0u;
                qa[ks][1] = gq < G ? v1 : 0u;
            }
        }
        float m = -INFINITY, l = 0.f;
        // o[j]: output dims 16j + lane/4 (0, 1) and 16j + 8 + lane/4 (2, 3) of
        // heads 2(lane&3) (0, 2) and 2(lane&3) + 1 (1, 3)
        float o[8][4];
#pragma unroll
        for (int n = 0; n < 8; ++n) o[n][0] = o[n][1] = o[n][2] = o[n][3] = 0.f;

        // tiles k of the piece with (ibase + k) % W == warp
        int k0 = (warp - ibase % kConsumers + kConsumers) % kConsumers;
        for (int k = k0; k < ntile; k += kConsumers) {
            if (misc[0]) break;
            const int i = ibase + k;
            const int slot = i % kSlots;
            if (!mbar_wait(&full[slot], (i / kSlots) & 1, P.err)) {
                misc[0] = 1;
                break;
            }
            const int tok0 = (pc.t0 + k) * kTile;
            const int valid = min(kTile, T - tok0);
            const uint32_t kb = ring + slot * kSlotBytes;
            const uint32_t vb = kb + 2 * kBoxBytes;

            // scores: s[nt] = rows gq (c0, c1) and gq + 8 (c2, c3), tokens 8 nt + qc, + 1
            float s[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
            {
                const int r = ((lane >> 4) << 3) + (lane & 7);
                const int cadd = (lane >> 3) & 1;
#pragma unroll
                for (int ks = 0; ks < 8; ++ks) {
                    uint32_t kf[4];
                    ldsm_x4(kb + (ks >> 2) * kBoxBytes + sw128(r, ((ks & 3) << 1) + cadd), kf);
                    const uint32_t a[4] = {qa[ks][0], 0u, qa[ks][1], 0u};
                    mma16816(s[0], a, kf[0], kf[1]);
                    mma16816(s[1], a, kf[2], kf[3]);
                }
            }
            // online softmax of row gq over this tile's tokens
            float x0 = qc < valid ? s[0][0] * P.sl2 : -INFINITY;
            float x1 = qc + 1 < valid ? s[0][1] * P.sl2 : -INFINITY;
            float x2 = qc + 8 < valid ? s[1][0] * P.sl2 : -INFINITY;
            float x3 = qc + 9 < valid ? s[1][1] * P.sl2 : -INFINITY;
            float mx = fmaxf(fmaxf(x0, x1), fmaxf(x2, x3));
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
            const float mnew = fmaxf(m, mx);
            const float msafe = mnew == -INFINITY ? 0.f : mnew;
            const float alpha = exp2f(m - msafe);
            m = mnew;
            const uint32_t p01 = pack_half2(exp2f(x0 - msafe), exp2f(x1 - msafe));
            const uint32_t p23 = pack_half2(exp2f(x2 - msafe), exp2f(x3 - msafe));
            const float2 f01 = unpack_half2(p01), f23 = unpack_half2(p23);
            l = l * alpha + ((f01.x + f01.y) + (f23.x + f23.y));

            // weights x values, transposed: o^T (128 dims x 8 heads) += V^T (dims x 16
            // tokens) * P^T (tokens x heads).  The score layout above leaves this
            // lane's weights of head gq, tokens qc, qc+1 and qc+8, qc+9, exactly the
            // B fragment of P^T; A = V^T comes from the value tile by a transposing
            // ldmatrix.  Output columns = heads 2(lane&3), +1: fetch their factors.
            const float al0 = __shfl_sync(0xffffffffu, alpha, 8 * (lane & 3));
            const float al1 = __shfl_sync(0xffffffffu, alpha, 8 * (lane & 3) + 4);
            // masks of the value rows past the sequence end (their contents may be anything)
            const uint32_t mlo = (qc < valid ? 0x0000FFFFu : 0u) | (qc + 1 < valid ? 0xFFFF0000u : 0u);
            const uint32_t mhi = (qc + 8 < valid ? 0x0000FFFFu : 0u) | (qc + 9 < valid ? 0xFFFF0000u : 0u);
            {
                const int mi = lane >> 3;
                const int r = ((mi >> 1) << 3) + (lane & 7);
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    uint32_t va[4];
                    ldsm_x4_trans(vb + (j >> 2) * kBoxBytes + sw128(r, ((2 * j) & 7) + (mi & 1)), va);
                    va[0] &= mlo;
                    va[1] &= mlo;
                    va[2] &= mhi;
                    va[3] &= mhi;
                    o[j][0] *= al0;
                    o[j][1] *= al1;
                    o[j][2] *= al0;
                    o[j][3] *= al1;
                    mma16816(o[j], va, p01, p23);
                }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&empty[slot]);
        }

        // ---- merge the warps' states of this piece (fixed warp order)
        l += __shfl_xor_sync(0xffffffffu, l, 1);
        l += __shfl_xor_sync(0xffffffffu, l, 2);
        {
            const int h0 = 2 * (lane & 3), dl = lane >> 2;
            float* s0 = scr + (warp * kMaxGroup + h0) * kD;
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                if (h0 < G) {
                    s0[16 * j + dl] = o[j][0];
                    s0[16 * j + 8 + dl] = o[j][2];
                }
                if (h0 + 1 < G) {
                    s0[kD + 16 * j + dl] = o[j][1];
                    s0[kD + 16 * j + 8 + dl] = o[j][3];
                }
            }
            if (gq < G && (lane & 3) == 0) {
                mrow[warp * kMaxGroup + gq] = m;
                lrow[warp * kMaxGroup + gq] = l;
            }
        }
        named_barrier_sync(1, kConsumers * 32);
        float* part = P.part + static_cast<size_t>(pc.slot) * (kPartHdr + G * kD);
        for (int e = tid; e < G * (kD / 2); e += kConsumers * 32) {
            const int gg = e / (kD / 2), d = 2 * (e % (kD / 2));
            float M = -INFINITY;
#pragma unroll
            for (int w = 0; w < kConsumers; ++w) M = fmaxf(M, mrow[w * kMaxGroup + gg]);
            const float Ms = M == -INFINITY ? 0.f : M;
            float L = 0.f, O0 = 0.f, O1 = 0.f;
#pragma unroll
            for (int w = 0; w < kConsumers; ++w) {
                const float f = exp2f(mrow[w * kMaxGroup + gg] - Ms);
                L += lrow[w * kMaxGroup + gg] * f;
                const float2 ov = *reinterpret_cast<const float2*>(scr + (w * kMaxGroup + gg) * kD + d);
                O0 += ov.x * f;
                O1 += ov.y * f;
            }
            if (pc.npieces == 1) {
                const float inv = L > 0.f ? 1.f / L : 0.f;
                uint16_t* ob = P.out + static_cast<size_t>(pc.b) * P.out_stride + static_cast<size_t>(pc.h * G + gg) * kD;
                *reinterpret_cast<uint32_t*>(ob + d) = pack_half2(O0 * inv, O1 * inv);
            } else {
                *reinterpret_cast<float2*>(part + kPartHdr + gg * kD + d) = make_float2(O0, O1);
                if (d == 0) {
                    part[gg] = M;
                    part[kMaxGroup + gg] = L;
                }
            }
        }
        if (pc.npieces > 1) {
            __threadfence();
            named_barrier_sync(1, kConsumers * 32);
            if (tid == 0) {
                const uint32_t old = atomicAdd(P.cnt + pc.seg, 1u);
                misc[1] = (old == static_cast<uint32_t>(pc.npieces - 1)) ? 1 : 0;
            }
            named_barrier_sync(1, kConsumers * 32);
            if (misc[1]) {
                __threadfence();
                // Merge parts p = 0..np-1 of this segment.  (1) per head row: 16
                // threads run the online max/normaliser merge over the parts'
                // (M_p, L_p), then a fixed shuffle tree joins them; the factors
                // 2^(M_p - M*) land in shared memory.  (2) every output element
                // sums f_p * O_p in part order, loads independent of each other.
                const int np = pc.npieces;
                const size_t pstride = kPartHdr + static_cast<size_t>(G) * kD;
                const float* pbase = P.part + static_cast<size_t>(pc.first + pc.seg) * pstride;
                float* fsm = scr;     // [np][8] (np <= kMaxParts)
                float* mls = mrow;    // M*[8], L*[8]
                {
                    const int gg = tid >> 4, sub = tid & 15;
                    float m = -INFINITY, l = 0.f;
                    if (gg < G) {
#pragma unroll 4
                        for (int p = sub; p < np; p += 16) {
                            const float Mp = __ldcg(pbase + p * pstride + gg);
                            const float Lp = __ldcg(pbase + p * pstride + kMaxGroup + gg);
                            fsm[p * kMaxGroup + gg] = Mp;
                            const float mn = fmaxf(m, Mp);
                            const float ms = mn == -INFINITY ? 0.f : mn;
                            l = l * exp2f(m - ms) + Lp * exp2f(Mp - ms);
                            m = mn;
                        }
                    }
#pragma unroll
                    for (int o = 1; o < 16; o <<= 1) {
                        const float m2 = __shfl_xor_sync(0xffffffffu, m, o);
                        const float l2 = __shfl_xor_sync(0xffffffffu, l, o);
                        const float mn = fmaxf(m, m2);
                        const float ms = mn == -INFINITY ? 0.f : mn;
                        l = l * exp2f(m - ms) + l2 * exp2f(m2 - ms);
                        m = mn;
                    }
                    if (gg < G && sub == 0) {
                        mls[gg] = m;
                        mls[kMaxGroup + gg] = l;
                    }
                    named_barrier_sync(1, kConsumers * 32);
                    if (gg < G) {
                        const float ms = mls[gg] == -INFINITY ? 0.f : mls[gg];
                        for (int p = sub; p < np; p += 16) fsm[p * kMaxGroup + gg] = exp2f(fsm[p * kMaxGroup + gg] - ms);
                    }
                    named_barrier_sync(1, kConsumers * 32);
                }
                for (int e = tid; e < G * (kD / 4); e += kConsumers * 32) {
                    const int gg = e / (kD / 4), d = 4 * (e % (kD / 4));
                    const float* po = pbase + kPartHdr + gg * kD + d;
                    float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
#pragma unroll 8
                    for (int p = 0; p < np; ++p) {
                        const float f = fsm[p * kMaxGroup + gg];
                        const float4 ov = __ldcg(reinterpret_cast<const float4*>(po + p * pstride));
                        a0 = fmaf(ov.x, f, a0);
                        a1 = fmaf(ov.y, f, a1);
                        a2 = fmaf(ov.z, f, a2);
                        a3 = fmaf(ov.w, f, a3);
                    }
                    const float L = mls[kMaxGroup + gg];
                    const float inv = L > 0.f ? 1.f / L : 0.f;
                    uint16_t* ob =
                        P.out + static_cast<size_t>(pc.b) * P.out_stride + static_cast<size_t>(pc.h * G + gg) * kD + d;
                    reinterpret_cast<uint32_t*>(ob)[0] = pack_half2(a0 * inv, a1 * inv);
                    reinterpret_cast<uint32_t*>(ob)[1] = pack_half2(a2 * inv, a3 * inv);
                }
                if (tid == 0) P.cnt[pc.seg] = 0u;
            }
        }
        named_barrier_sync(1, kConsumers * 32);   // scratch and flags free for the next piece
        ibase += ntile;
        g += ntile;
    }
}

__global__ void kv_append_kernel(const uint16_t* __restrict__ new_k, const uint16_t* __restrict__ new_v,
                                 int new_stride, uint16_t* k_cache, uint16_t* v_cache, const int32_t* page_table,
                                 int pt_stride, const int32_t* positions, int Hkv, int page_size, int num_pages,
                                 uint32_t* err)
{
    const int b = blockIdx.x;
    const int pos = positions[b];
    const int max_tok = pt_stride * page_size;
    if (pos < 0 || pos >= max_tok) {
        if (threadIdx.x == 0) atomicOr(err, kErrAppend);
        return;
    }
    const int page = page_table[static_cast<size_t>(b) * pt_stride + pos / page_size];
    if (page < 0 || page >= num_pages) {
        if (threadIdx.x == 0) atomicOr(err, kErrAppend);
        return;
    }
    const int row = pos % page_size;
    for (int e = threadIdx.x; e < Hkv * (kD / 8); e += blockDim.x) {
        const int h = e / (kD / 8), c = e % (kD / 8);
        const size_t dst = ((static_cast<size_t>(page) * Hkv + h) * page_size + row) * kD + 8 * c;
        const size_t src = static_cast<size_t>(b) * new_stride + static_cast<size_t>(h) * kD + 8 * c;
        *reinterpret_cast<uint4*>(k_cache + dst) = *reinterpret_cast<const uint4*>(new_k + src);
        *reinterpret_cast<uint4*>(v_cache + dst) = *reinterpret_cast<const uint4*>(new_v + src);
    }
}

int attn_grid(int dev, int sms)
{
    static std::mutex mu;
    static int cached[64] = {0};
    std::lock_guard<std::mutex> lock(mu);
    if (dev >= 0 && dev < 64 && cached[dev]) return cached[dev];
    int per_sm = 0;
    if (cudaFuncSetAttribute(paged_attn_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(attn_smem_bytes(WQ4_ATTN_MAX_BATCH))) != cudaSuccess)
        return 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, paged_attn_kernel, kThreads,
                                                      attn_smem_bytes(WQ4_ATTN_MAX_BATCH)) != cudaSuccess)
        return 0;
    if (per_sm < 1) return 0;
    if (per_sm > kCtasPerSm) per_sm = kCtasPerSm;
    int g = sms * per_sm;
    if (g > kMaxParts) g = kMaxParts;
    if (dev >= 0 && dev < 64) cached[dev] = g;
    return g;
}

bool check_cache(const wq4_kv_cache* c)
{
    return c && c->k && c->v && c->page_table && c->num_pages >= 1 && c->n_kv_heads >= 1 && c->page_size >= kTile &&
           c->page_size % kTile == 0 && c->page_table_stride >= 1 && c->head_dim >= 1;
}

}  // namespace
}  // namespace wq4

using namespace wq4;

extern "C" size_t wq4_paged_attention_workspace_bytes(int batch, int n_q_heads, int n_kv_heads, int head_dim)
{
    if (batch < 1 || batch > WQ4_ATTN_MAX_BATCH || n_kv_heads < 1 || n_q_heads < n_kv_heads ||
        n_q_heads % n_kv_heads || n_q_heads / n_kv_heads > kMaxGroup || head_dim != kD)
        return 0;
    int dev = 0;
    const DeviceInfo* di = current_device_info(&dev);
    if (!di) return 0;
    const int grid = attn_grid(dev, di->sm_count);
    if (grid < 1) return 0;
    const int G = n_q_heads / n_kv_heads;
    const size_t segs = static_cast<size_t>(batch) * n_kv_heads;
    const size_t cnt_bytes = align_up(segs * 4, 256);
    return cnt_bytes + (static_cast<size_t>(grid) + segs) * (kPartHdr + G * kD) * 4;
}

extern "C" int wq4_paged_attention(const wq4_kv_cache* cache, const uint16_t* q, int q_stride,
                                   const int32_t* seq_lens, uint16_t* out, int out_stride, int batch, int n_q_heads,
                                   float scale, void* workspace, size_t workspace_bytes, void* stream)
{
    if (!check_cache(cache) || !q || !seq_lens || !out || !workspace) return WQ4_ERR_INVALID;
    if (batch < 1 || batch > WQ4_ATTN_MAX_BATCH) return WQ4_ERR_INVALID;
    const int Hkv = cache->n_kv_heads;
    if (n_q_heads < Hkv || n_q_heads % Hkv) return WQ4_ERR_INVALID;
    if (cache->head_dim != kD || n_q_heads / Hkv > kMaxGroup) return WQ4_ERR_UNSUPPORTED;
    if (q_stride < n_q_heads * kD || out_stride < n_q_heads * kD) return WQ4_ERR_INVALID;
    if (!(scale == scale) || std::isinf(scale)) return WQ4_ERR_INVALID;
    if (!aligned(q, 16) || q_stride % 8 || !aligned(cache->k, 16) || !aligned(cache->v, 16) ||
        !aligned(out, 4) || out_stride % 2 || !aligned(workspace, 16) || !aligned(seq_lens, 4) ||
        !aligned(cache->page_table, 4))
        return WQ4_ERR_ALIGN;
    const int64_t rows = static_cast<int64_t>(cache->num_pages) * Hkv * cache->page_size;
    if (rows >= (int64_t(1) << 31)) return WQ4_ERR_UNSUPPORTED;
    if (static_cast<int64_t>(cache->page_table_stride) * cache->page_size >= (int64_t(1) << 30))
        return WQ4_ERR_UNSUPPORTED;
    // the tile list (every sequence at its page table's capacity) is indexed in int
    const int64_t max_tiles = (static_cast<int64_t>(cache->page_table_stride) * cache->page_size + kTile - 1) / kTile;
    if (max_tiles * batch * Hkv >= (int64_t(1) << 31)) return WQ4_ERR_UNSUPPORTED;
    const size_t need = wq4_paged_attention_workspace_bytes(batch, n_q_heads, Hkv, kD);
    if (need == 0) return WQ4_ERR_CUDA;
    if (workspace_bytes < need) return WQ4_ERR_INVALID;
    const size_t cache_bytes = static_cast<size_t>(rows) * kD * 2;
    const size_t out_bytes = (static_cast<size_t>(batch - 1) * out_stride + static_cast<size_t>(n_q_heads) * kD) * 2;
    if (overlaps(cache->k, cache_bytes, cache->v, cache_bytes) || overlaps(out, out_bytes, cache->k, cache_bytes) ||
        overlaps(out, out_bytes, cache->v, cache_bytes) || overlaps(out, out_bytes, workspace, need) ||
        overlaps(out, out_bytes, q, (static_cast<size_t>(batch - 1) * q_stride + n_q_heads * kD) * 2))
        return WQ4_ERR_INVALID;

    int dev = 0;
    const DeviceInfo* di = current_device_info(&dev);
    if (!di) return WQ4_ERR_CUDA;
    const int grid = attn_grid(dev, di->sm_count);
    if (grid < 1) return WQ4_ERR_CUDA;

    AttnParams p;
    std::memset(&p, 0, sizeof(p));
    if (!encode_tensor_map_2d(&p.mk, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, cache->k, kD, static_cast<uint64_t>(rows), kD * 2,
                              64, kTile, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !encode_tensor_map_2d(&p.mv, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, cache->v, kD, static_cast<uint64_t>(rows), kD * 2,
                              64, kTile, CU_TENSOR_MAP_SWIZZLE_128B))
        return WQ4_ERR_CUDA;
    const size_t segs = static_cast<size_t>(batch) * Hkv;
    p.q = q;
    p.out = out;
    p.seq_lens = seq_lens;
    p.page_table = cache->page_table;
    p.cnt = static_cast<uint32_t*>(workspace);
    p.part = reinterpret_cast<float*>(static_cast<uint8_t*>(workspace) + align_up(segs * 4, 256));
    p.err = status_word();
    p.q_stride = q_stride;
    p.out_stride = out_stride;
    p.pt_stride = cache->page_table_stride;
    p.batch = batch;
    p.Hkv = Hkv;
    p.G = n_q_heads / Hkv;
    p.page_size = cache->page_size;
    p.num_pages = cache->num_pages;
    p.sl2 = static_cast<float>(static_cast<double>(scale) * 1.4426950408889634);
    if (!p.err) return WQ4_ERR_CUDA;
    paged_attn_kernel<<<grid, kThreads, attn_smem_bytes(batch), static_cast<cudaStream_t>(stream)>>>(p);
    return cudaGetLastError() == cudaSuccess ? WQ4_OK : WQ4_ERR_CUDA;
}

extern "C" int wq4_kv_append(const wq4_kv_cache* cache, const uint16_t* new_k, const uint16_t* new_v, int new_stride,
                             const int32_t* positions, int batch, void* stream)
{
    if (!check_cache(cache) || !new_k || !new_v || !positions || batch < 1) return WQ4_ERR_INVALID;
    if (cache->head_dim != kD) return WQ4_ERR_UNSUPPORTED;
    if (new_stride < cache->n_kv_heads * kD) return WQ4_ERR_INVALID;
    if (!aligned(new_k, 16) || !aligned(new_v, 16) || new_stride % 8 || !aligned(cache->k, 16) ||
        !aligned(cache->v, 16) || !aligned(positions, 4) || !aligned(cache->page_table, 4))
        return WQ4_ERR_ALIGN;
    if (static_cast<int64_t>(cache->page_table_stride) * cache->page_size >= (int64_t(1) << 30))
        return WQ4_ERR_UNSUPPORTED;
    uint32_t* err = status_word();
    if (!err) return WQ4_ERR_CUDA;
    kv_append_kernel<<<batch, 256, 0, static_cast<cudaStream_t>(stream)>>>(
        new_k, new_v, new_stride, cache->k, cache->v, cache->page_table, cache->page_table_stride, positions,
        cache->n_kv_heads, cache->page_size, cache->num_pages, err);
    return cudaGetLastError() == cudaSuccess ? WQ4_OK : WQ4_ERR_CUDA;
}
