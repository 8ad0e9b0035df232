// wq4_gemv.cu -- the fused dequantize x GEMV of one decode step and the
// C-ABI entry points that do not belong to the chain.
//
// y[b][n] = fp16( sum_k (q(n,k) - 7) * s[n][k/32] * x[b][k] ), the projection
// every decoded token applies to every 4-bit weight matrix (Section 3,
// Table 1).  Two kernels:
//
//  * gemv_mma_kernel<B> (batch B <= 2, K % 256 == 0, 16-byte aligned scales):
//    the persistent decode chain's weight stream for one projection.  A
//    producer warp streams the CTA's word rows (pairs of rows) through a
//    ring of shared-memory slots with 1-D bulk copies; 15 consumer warps take
//    work items (superpair of row pairs, K part) round-robin in ring order
//    and run them on the legacy tensor path (wq4_items.cuh: exact fp16
//    q - 7, eight groups of x as the MMA's columns, scales in fp32 on the
//    diagonal); K parts are added in part order in shared memory.
//  * gemv_tma_kernel<B> (batch B <= 4, K % 256 == 0): one persistent CTA per
//    SM.  A producer warp streams the CTA's contiguous block of rows through a
//    ring of shared-memory slots with 1-D bulk copies (TMA) and mbarriers;
//    consumer warps take rows round-robin, unpack in registers and accumulate
//    in fp32 against the activations staged once in shared memory ("GEMM
//    tiling" and "kernel fusion" of Section 2.3, by hand).
//  * gemv_generic_kernel<BT> (any K % 32 == 0, batch up to 32, scales of any
//    2-byte alignment): warp per row, weights loaded straight into registers,
//    activations read through L1.
#include "wq4_device.cuh"
#include "wq4_items.cuh"
#include "wq4_host.h"
#include "wq4.h"

#include <cuda_runtime.h>

#include <atomic>
#include <mutex>

namespace wq4 {

__device__ uint32_t g_status_word;

// Programmatic dependent launch: wait for the previous grid of the stream
// (complete, memory visible) / let the next one launch.  No effect when the
// launch did not ask for it.
__device__ __forceinline__ void grid_dependency_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void grid_dependents_launch() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

constexpr int kGemvConsumerWarps = 8;
constexpr int kGemvThreads = (kGemvConsumerWarps + 1) * 32;
constexpr int kMaxSlots = 32;
constexpr int kHeaderBytes = 1024;              // mbarriers (2 * kMaxSlots * 8 B) + pad
constexpr int kTargetSlotBytes = 16 * 1024;

struct GemvTmaParams {
    const uint32_t* W;
    const uint16_t* s;
    const uint16_t* x;
    uint16_t* y;
    int N, K;
    int rows_per_slot;
    int nslots;
    uint32_t slot_bytes;       // stride between slots (128-byte multiple)
    uint32_t scales_offset;    // offset of the scales region inside a slot
    uint32_t x_bytes;          // bytes reserved for staged activations
    uint32_t* err;
};

template <int B>
__global__ void __launch_bounds__(kGemvThreads, 1) gemv_tma_kernel(const GemvTmaParams p)
{
    extern __shared__ __align__(1024) uint8_t smem[];
    uint64_t* full = reinterpret_cast<uint64_t*>(smem);
    uint64_t* empty = full + kMaxSlots;
    uint4* xs = reinterpret_cast<uint4*>(smem + kHeaderBytes);
    uint8_t* slots = smem + kHeaderBytes + p.x_bytes;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int n0 = static_cast<int>(static_cast<int64_t>(blockIdx.x) * p.N / gridDim.x);
    const int n1 = static_cast<int>(static_cast<int64_t>(blockIdx.x + 1) * p.N / gridDim.x);
    const int R = n1 - n0;
    const int rps = p.rows_per_slot;
    const int nchunks = (R + rps - 1) / rps;
    const int wpr = p.K >> 3;   // words per row
    const int gpr = p.K >> 5;   // groups per row

    if (threadIdx.x == 0) {
        for (int i = 0; i < p.nslots; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], kGemvConsumerWarps);
        }
        mbar_fence_init();
    }
    __syncthreads();
    grid_dependents_launch();     // the next launch in the stream may start its set-up

    if (warp == kGemvConsumerWarps) {
        // ---------------- producer: one elected lane issues the bulk copies
        if (lane == 0) {
            const uint64_t pol = l2_policy_evict_first();
            for (int ch = 0; ch < nchunks; ++ch) {
                const int slot = ch % p.nslots;
                const int round = ch / p.nslots;
                if (round > 0) mbar_wait(&empty[slot], (round - 1) & 1, p.err);
                const int r0 = ch * rps;
                const int nr = min(rps, R - r0);
                const uint32_t cb = static_cast<uint32_t>(nr) * (p.K / 2);
                const uint32_t sb = static_cast<uint32_t>(nr) * (p.K / 16);
                uint8_t* dst = slots + static_cast<size_t>(slot) * p.slot_bytes;
                mbar_arrive_expect_tx(&full[slot], cb + sb);
                bulk_g2s(dst, p.W + static_cast<size_t>(n0 + r0) * wpr, cb, &full[slot], pol);
                bulk_g2s(dst + p.scales_offset, p.s + static_cast<size_t>(n0 + r0) * gpr, sb, &full[slot], pol);
            }
            // no copy may still be in flight when the CTA exits
            const int first = nchunks > p.nslots ? nchunks - p.nslots : 0;
            for (int ch = first; ch < nchunks; ++ch)
                mbar_wait(&full[ch % p.nslots], (ch / p.nslots) & 1, p.err);
        }
        return;
    }

    // ---------------- consumers: stage x (swizzled) once, after the previous
    // grid in the stream is complete (programmatic dependent launch: the
    // producer's weight copies may start earlier)
    grid_dependency_wait();
    {
        const uint4* xg = reinterpret_cast<const uint4*>(p.x);
        const int chunks_per_row = p.K >> 3;
        for (int i = threadIdx.x; i < B * chunks_per_row; i += kGemvConsumerWarps * 32) {
            const int b = i / chunks_per_row, c = i - b * chunks_per_row;
            xs[b * chunks_per_row + x_chunk(c >> 2, c & 3)] = xg[i];
        }
        named_barrier_sync(1, kGemvConsumerWarps * 32);
    }

    for (int ch = 0; ch < nchunks; ++ch) {
        const int slot = ch % p.nslots;
        mbar_wait(&full[slot], (ch / p.nslots) & 1, p.err);
        const uint8_t* base = slots + static_cast<size_t>(slot) * p.slot_bytes;
        const int r0 = ch * rps, r1 = min(R, r0 + rps);
        int i = r0 + ((warp - r0 % kGemvConsumerWarps) + kGemvConsumerWarps) % kGemvConsumerWarps;
        for (; i < r1; i += kGemvConsumerWarps) {
            const uint4* crow = reinterpret_cast<const uint4*>(base) + static_cast<size_t>(i - r0) * gpr;
            const uint16_t* srow = reinterpret_cast<const uint16_t*>(base + p.scales_offset) + (i - r0) * gpr;
            float racc[B];
#pragma unroll
            for (int b = 0; b < B; ++b) racc[b] = 0.f;
#pragma unroll 2
            for (int g = lane; g < gpr; g += 32)
                group_dot_smem<B>(crow[g], half_bits_to_float(srow[g]), xs, p.K >> 3, g, racc);
#pragma unroll
            for (int b = 0; b < B; ++b) {
                const float v = warp_sum(racc[b]);
                if (lane == b) p.y[static_cast<size_t>(b) * p.N + n0 + i] = float_to_half_bits(v);
            }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&empty[slot]);
    }
}

// Generic path: warp per row, batch processed in tiles of BT rows of x.
// ------------------------------------------------------ gemv_mma_kernel --

constexpr int kMmaWarps = 15;                         // consumer warps
constexpr int kMmaThreads = (kMmaWarps + 1) * 32;     // + the producer warp
constexpr int kMmaMaxSlots = 16;
constexpr int kMmaFullBars = 48;                      // full barriers: nbars = (48 / nslots) * nslots
constexpr uint32_t kMmaRelease = 1024;                // arrivals that release a slot (see below)
constexpr int kMmaMaxPart = 384;                      // float4 partial sums [superpair][part][batch]
constexpr int kMmaHdrPart = 8 * (kMmaFullBars + kMmaMaxSlots);
constexpr int kMmaHeader = kMmaHdrPart + 16 * kMmaMaxPart;
static_assert(kMmaHdrPart % 16 == 0 && kMmaHeader % 128 == 0, "header alignment");

struct GemvMmaParams {
    const uint32_t* W;
    const uint16_t* s;
    const uint16_t* x;
    uint16_t* y;
    int N, K;
    int nslots, nbars;
    uint32_t slot_bytes, x_bytes;
    int spw;         // words (row pairs) per superpair: 1 or 2
    int q;           // K parts per superpair (divides K / 256)
    uint32_t* err;
};

// Chunk c of a CTA's words lives in slot c % nslots and lands on full barrier
// c % nbars; a slot is released after kMmaRelease arrivals: one per item
// consumed from it plus (kMmaRelease - items) from the warp that took its
// first item.  A warp waits only on the chunks holding its items; the plan
// keeps nslots + ceil(15 / items per chunk) <= nbars so that no parity wait
// can alias, as in the chain kernel.
template <int B>
__global__ void __launch_bounds__(kMmaThreads, 1) gemv_mma_kernel(const GemvMmaParams p)
{
    extern __shared__ __align__(1024) uint8_t smem[];
    uint64_t* full = reinterpret_cast<uint64_t*>(smem);
    uint64_t* empty = full + kMmaFullBars;
    float4* part = reinterpret_cast<float4*>(smem + kMmaHdrPart);
    uint4* xs = reinterpret_cast<uint4*>(smem + kMmaHeader);
    uint8_t* slots = smem + kMmaHeader + p.x_bytes;
    constexpr int kConsumers = kMmaWarps * 32;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int N = p.N, K = p.K, cpr = K >> 3, wpr = K >> 3, gpr = K >> 5;
    const int nw = (N + 1) / 2;
    const int w0 = static_cast<int>(static_cast<int64_t>(blockIdx.x) * nw / gridDim.x);
    const int w1 = static_cast<int>(static_cast<int64_t>(blockIdx.x + 1) * nw / gridDim.x);
    const int nwd = w1 - w0;
    const int spw = p.spw, q = p.q;
    const uint32_t word_bytes = 2u * static_cast<uint32_t>(K / 2 + K / 16);
    const int wps = max(spw, static_cast<int>(p.slot_bytes / word_bytes) / spw * spw);
    const int nch = (nwd + wps - 1) / wps;

    if (threadIdx.x == 0) {
        for (int i = 0; i < p.nbars; ++i) mbar_init(&full[i], 1);
        for (int i = 0; i < p.nslots; ++i) mbar_init(&empty[i], kMmaRelease);
        mbar_fence_init();
    }
    __syncthreads();
    grid_dependents_launch();     // the next launch in the stream may start its set-up

    if (warp == kMmaWarps) {
        // ---------------- producer: one lane issues the bulk copies
        if (lane == 0) {
            const uint64_t pol = l2_policy_evict_first();
            int slot = 0, round = 0, fbi = 0;
            for (int k = 0; k < nch; ++k) {
                const int wa = w0 + k * wps, wb = min(w1, wa + wps);
                if (round > 0) mbar_wait(&empty[slot], (round - 1) & 1, p.err);
                const int nrows = min(2 * wb, N) - 2 * wa;
                const uint32_t cb = static_cast<uint32_t>(nrows) * (K / 2);
                const uint32_t sb = static_cast<uint32_t>(nrows) * (K / 16);
                uint8_t* dst = slots + static_cast<size_t>(slot) * p.slot_bytes;
                uint64_t* fb = &full[fbi];
                if (++slot == p.nslots) {
                    slot = 0;
                    ++round;
                }
                if (++fbi == p.nbars) fbi = 0;
                mbar_arrive_expect_tx(fb, cb + sb);
                bulk_g2s(dst, p.W + static_cast<size_t>(2 * wa) * wpr, cb, fb, pol);
                bulk_g2s(dst + cb, p.s + static_cast<size_t>(2 * wa) * gpr, sb, fb, pol);
            }
            // the chunks before the last nslots were consumed, so have landed:
            // wait for the rest before the CTA's shared memory goes away
            const int first = nch > p.nslots ? nch - p.nslots : 0;
            for (int o = first; o < nch; ++o) mbar_wait(&full[o % p.nbars], (o / p.nbars) & 1, p.err);
        }
        return;
    }

    // ---------------- consumers: x once, in the MMA's pair-permuted order,
    // after the previous grid in the stream is complete
    grid_dependency_wait();
    {
        const uint4* xg = reinterpret_cast<const uint4*>(p.x);
        for (int i = threadIdx.x; i < B * cpr; i += kConsumers) xs[i] = pair_permute(xg[i]);
        named_barrier_sync(1, kConsumers);
    }
    const int J = K >> 8, upp = J / q;
    const int nsp = (nwd + spw - 1) / spw, nitems = nsp * q;
    const int sps = spw - 1;
    const int ips = (wps >> sps) * q;                          // items per chunk
    const uint32_t xsa = smem_addr(xs);
    const FDiv fq = fdiv_make(q), fips = fdiv_make(ips), fns = fdiv_make(p.nslots), fnb = fdiv_make(p.nbars);
    int it = warp;
    if (it < nitems) {
        int k = fdiv(it, fips);
        int ia = k * ips, ib = min(nitems, ia + ips);
        int slot = k - fdiv(k, fns) * p.nslots;
        const int qb = fdiv(k, fnb);
        int bar = k - qb * p.nbars;
        uint32_t par = static_cast<uint32_t>(qb) & 1u;
        while (it < nitems) {
            while (it >= ib) {                                 // next chunk holding one of the warp's items
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
            const int kw0 = k * wps;
            const int nrows = min(2 * min(w1, w0 + kw0 + wps), N) - 2 * (w0 + kw0);
            const uint32_t cbase = smem_addr(slots + static_cast<size_t>(slot) * p.slot_bytes);
            const uint32_t sbase = cbase + static_cast<uint32_t>(nrows) * (K / 2);
            uint32_t arrivals = (it == ia) ? kMmaRelease - static_cast<uint32_t>(ib - ia) : 0u;
            for (; it < ib; it += kMmaWarps) {
                ++arrivals;
                const int sl = fdiv(it, fq);
                const int pt = it - sl * q;
                const int jb = pt * upp, je = jb + upp;
                const int sw0 = sl << sps;                     // the superpair's first word (CTA-relative)
                const int wl = sw0 - kw0;                      // ... within the chunk
                // pairs (2w, 2w + 1) of words w, w + 1 (a missing second word
                // repeats the first, not stored; a missing last row repeats
                // the row before, not stored)
                uint32_t ca[2], cb2[2], sa[2], sb2[2];
#pragma unroll
                for (int pr = 0; pr < 2; ++pr) {
                    const int wr = (sw0 + pr < nwd) ? wl + pr : wl;
                    const uint32_t ra = 2 * wr;
                    const uint32_t rb = (2 * (w0 + kw0 + wr) + 1 < N) ? 2 * wr + 1 : 2 * wr;
                    ca[pr] = cbase + ra * (K / 2);
                    cb2[pr] = cbase + rb * (K / 2);
                    sa[pr] = sbase + ra * (K / 16);
                    sb2[pr] = sbase + rb * (K / 16);
                }
                float acc[2][B];
#pragma unroll
                for (int pr = 0; pr < 2; ++pr)
#pragma unroll
                    for (int b = 0; b < B; ++b) acc[pr][b] = 0.f;
                if (spw == 2) {
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
                if (q == 1) {
                    // whole superpairs: lane 0 writes rows 2w (and 2w + 2), lane 16
                    // rows 2w + 1 (and 2w + 3)
                    const int n0 = 2 * (w0 + sw0) + (lane == 16 ? 1 : 0);
                    if (lane == 0 || lane == 16) {
#pragma unroll
                        for (int b = 0; b < B; ++b) {
                            uint16_t* out = p.y + static_cast<size_t>(b) * N;
                            if (n0 < N) out[n0] = float_to_half_bits(acc[0][b]);
                            if (spw == 2 && sw0 + 1 < nwd && n0 + 2 < N) out[n0 + 2] = float_to_half_bits(acc[1][b]);
                        }
                    }
                } else {
                    float* pf = reinterpret_cast<float*>(part + (sl * q + pt) * B);
#pragma unroll
                    for (int b = 0; b < B; ++b) {
                        if (lane == 0) {
                            pf[4 * b + 0] = acc[0][b];
                            pf[4 * b + 2] = acc[1][b];
                        }
                        if (lane == 16) {
                            pf[4 * b + 1] = acc[0][b];
                            pf[4 * b + 3] = acc[1][b];
                        }
                    }
                }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive_count(&empty[slot], arrivals);
        }
    }
    if (q > 1) {
        // every part is in: add them in part order, one thread per (superpair, row)
        named_barrier_sync(1, kConsumers);
        for (int e = threadIdx.x; e < nsp * B; e += kConsumers) {
            const int sl = e / B, b = e - sl * B;
            const float4* pp = part + sl * q * B + b;
            float4 sum = pp[0];
            for (int r = 1; r < q; ++r) {
                const float4 t = pp[r * B];
                sum.x += t.x;
                sum.y += t.y;
                sum.z += t.z;
                sum.w += t.w;
            }
            const int n = 2 * (w0 + (sl << sps));
            uint16_t* out = p.y + static_cast<size_t>(b) * N;
            out[n] = float_to_half_bits(sum.x);
            if (n + 1 < N) out[n + 1] = float_to_half_bits(sum.y);
            if (spw == 2 && (sl << sps) + 1 < nwd) {
                out[n + 2] = float_to_half_bits(sum.z);
                if (n + 3 < N) out[n + 3] = float_to_half_bits(sum.w);
            }
        }
    }
}

template <int BT>
__global__ void __launch_bounds__(256) gemv_generic_kernel(const uint32_t* __restrict__ W,
                                                           const uint16_t* __restrict__ s,
                                                           const uint16_t* __restrict__ x,
                                                           uint16_t* __restrict__ y, int N, int K,
                                                           int batch)
{
    const int lane = threadIdx.x & 31;
    const int gw = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    const int nw = gridDim.x * (blockDim.x >> 5);
    const int gpr = K >> 5;
    for (int n = gw; n < N; n += nw) {
        const uint4* crow = reinterpret_cast<const uint4*>(W + static_cast<size_t>(n) * (K >> 3));
        const uint16_t* srow = s + static_cast<size_t>(n) * gpr;
        for (int b0 = 0; b0 < batch; b0 += BT) {
            float acc[BT];
#pragma unroll
            for (int b = 0; b < BT; ++b) acc[b] = 0.f;
            for (int g = lane; g < gpr; g += 32) {
                const uint4 cw = __ldg(crow + g);
                const float sc = half_bits_to_float(__ldg(srow + g));
                uint32_t pq[16];
                unpack_word(cw.x, pq + 0);
                unpack_word(cw.y, pq + 4);
                unpack_word(cw.z, pq + 8);
                unpack_word(cw.w, pq + 12);
#pragma unroll
                for (int b = 0; b < BT; ++b) {
                    if (b0 + b < batch) {
                        const uint4* xb =
                            reinterpret_cast<const uint4*>(x + static_cast<size_t>(b0 + b) * K) + g * 4;
                        const float a0 = fma8(pq + 0, __ldg(xb + 0), 0.f);
                        const float a1 = fma8(pq + 4, __ldg(xb + 1), 0.f);
                        const float a2 = fma8(pq + 8, __ldg(xb + 2), 0.f);
                        const float a3 = fma8(pq + 12, __ldg(xb + 3), 0.f);
                        acc[b] = fmaf(sc, (a0 + a1) + (a2 + a3), acc[b]);
                    }
                }
            }
#pragma unroll
            for (int b = 0; b < BT; ++b) {
                const float v = warp_sum(acc[b]);
                if (lane == b && b0 + b < batch) y[static_cast<size_t>(b0 + b) * N + n] = float_to_half_bits(v);
            }
        }
    }
}

// Unpack test hook: the GEMV's own unpack, written out.
__global__ void unpack_debug_kernel(const uint32_t* __restrict__ W, const uint16_t* __restrict__ s,
                                    float* __restrict__ w_out, uint8_t* __restrict__ q_out, int N, int K)
{
    const int64_t words = static_cast<int64_t>(N) * (K >> 3);
    const int wpr = K >> 3;
    for (int64_t t = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; t < words;
         t += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t n = t / wpr;
        const int j = static_cast<int>(t - n * wpr);
        uint32_t pq[4];
        unpack_word(W[t], pq);
        const float sc = half_bits_to_float(s[n * (K >> 5) + (j >> 2)]);
        const int64_t base = n * K + 8 * j;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float vlo = __half2float(__ushort_as_half(static_cast<uint16_t>(pq[i] & 0xFFFFu)));
            const float vhi = __half2float(__ushort_as_half(static_cast<uint16_t>(pq[i] >> 16)));
            if (q_out) {
                q_out[base + i] = static_cast<uint8_t>(static_cast<int>(vlo) + 7);
                q_out[base + i + 4] = static_cast<uint8_t>(static_cast<int>(vhi) + 7);
            }
            if (w_out) {
                w_out[base + i] = vlo * sc;
                w_out[base + i + 4] = vhi * sc;
            }
        }
    }
}

// --------------------------------------------------------------- host --

namespace {

constexpr int kMaxDevices = 64;
DeviceInfo g_info[kMaxDevices];
bool g_info_ready[kMaxDevices];
uint32_t* g_status_ptr[kMaxDevices];
std::mutex g_mu;

template <int B>
bool set_tma_attr(int smem)
{
    return cudaFuncSetAttribute(gemv_tma_kernel<B>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) ==
           cudaSuccess;
}

template <int B>
bool set_mma_attr(int smem)
{
    return cudaFuncSetAttribute(gemv_mma_kernel<B>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) ==
           cudaSuccess;
}

}  // namespace

const DeviceInfo* current_device_info(int* device_out)
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
    if (device_out) *device_out = dev;
    std::lock_guard<std::mutex> lock(g_mu);
    if (!g_info_ready[dev]) {
        DeviceInfo d;
        if (cudaDeviceGetAttribute(&d.sm_count, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return nullptr;
        if (cudaDeviceGetAttribute(&d.smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess)
            return nullptr;
        if (cudaDeviceGetAttribute(&d.coop_launch, cudaDevAttrCooperativeLaunch, dev) != cudaSuccess) return nullptr;
        if (!set_tma_attr<1>(d.smem_optin) || !set_tma_attr<2>(d.smem_optin) || !set_tma_attr<3>(d.smem_optin) ||
            !set_tma_attr<4>(d.smem_optin) || !set_mma_attr<1>(d.smem_optin) || !set_mma_attr<2>(d.smem_optin))
            return nullptr;
        void* ptr = nullptr;
        if (cudaGetSymbolAddress(&ptr, g_status_word) != cudaSuccess) return nullptr;
        g_status_ptr[dev] = static_cast<uint32_t*>(ptr);
        g_info[dev] = d;
        g_info_ready[dev] = true;
    }
    return &g_info[dev];
}

uint32_t* status_word()
{
    int dev = 0;
    if (!current_device_info(&dev)) return nullptr;
    return g_status_ptr[dev];
}

namespace {

// The launch shape of gemv_mma_kernel, or false when the matrix does not fit
// it (then the CUDA-core kernels run).  Superpairs of two words unless that
// is more than 20 KB of weights; slots of whole superpairs near 20 KB; K
// parts from the chain's cost model: rounds of items over the 15 warps times
// (units per item x unit cost + ~1200 cycles per item), with the first
// round's chunks inside the ring and no aliased barrier phase.
struct MmaPlan {
    int grid, nslots, nbars, spw, q;
    uint32_t slot_bytes, x_bytes;
    size_t smem;
};

bool plan_mma(const DeviceInfo* di, int N, int K, int B, MmaPlan* pl)
{
    const int nw = (N + 1) / 2;
    const int grid = nw < di->sm_count ? nw : di->sm_count;
    const int nwc = (nw + grid - 1) / grid;                       // most words of a CTA
    const size_t word_bytes = 2 * (static_cast<size_t>(K) / 2 + static_cast<size_t>(K) / 16);
    const int spw = (2 * word_bytes <= 20 * 1024 && nwc >= 2) ? 2 : 1;
    const size_t sp_bytes = spw * word_bytes;
    const size_t x_bytes = align_up(static_cast<size_t>(B) * K * 2, 128);
    if (static_cast<size_t>(di->smem_optin) < kMmaHeader + x_bytes) return false;
    const size_t avail = static_cast<size_t>(di->smem_optin) - kMmaHeader - x_bytes;
    size_t per = sp_bytes < 20 * 1024 ? (20 * 1024) / sp_bytes : 1;
    size_t slot_bytes = align_up(per * sp_bytes, 128);
    while (avail / slot_bytes < 4 && per > 1) {
        --per;
        slot_bytes = align_up(per * sp_bytes, 128);
    }
    int nslots = static_cast<int>(avail / slot_bytes);
    if (nslots > kMmaMaxSlots) nslots = kMmaMaxSlots;
    if (nslots < 3) return false;
    const int nbars = (kMmaFullBars / nslots) * nslots;
    const int J = K / 256;
    const int nsp = (nwc + spw - 1) / spw;
    const int sp_per_chunk = static_cast<int>((slot_bytes / word_bytes) / spw);
    const double unit = (spw == 2 ? 300.0 : 200.0) * (1.0 + 0.5 * (B - 1));
    int best_q = 0;
    double best = 0.0;
    for (int qq = 1; qq <= J; ++qq) {
        if (J % qq) continue;
        if (qq > 1 && nsp * qq * B > kMmaMaxPart) continue;
        const int ips = sp_per_chunk * qq;
        const int first_chunks = (kMmaWarps + ips - 1) / ips;
        if (first_chunks > nslots - 2 || nslots + first_chunks > nbars) continue;
        const int rounds = (nsp * qq + kMmaWarps - 1) / kMmaWarps;
        const double cost = rounds * ((J / qq) * unit + 1200.0);
        if (best_q == 0 || cost <= best) {
            best = cost;
            best_q = qq;
        }
    }
    if (best_q == 0) return false;
    pl->grid = grid;
    pl->nslots = nslots;
    pl->nbars = nbars;
    pl->spw = spw;
    pl->q = best_q;
    pl->slot_bytes = static_cast<uint32_t>(slot_bytes);
    pl->x_bytes = static_cast<uint32_t>(x_bytes);
    pl->smem = kMmaHeader + x_bytes + static_cast<size_t>(nslots) * slot_bytes;
    return true;
}

// Which batch 1-2 kernel a call takes (wq4_test_gemv_path): 0 the size rule,
// 1 the legacy-tensor-path kernel wherever it applies, 2 the CUDA-core one.
std::atomic<int> g_gemv_path{0};

// Below ~12 M weights a launch is bound by its fixed costs (x staging, the
// first chunk's round trip, the epilogue), which the smaller CUDA-core
// kernel pays less of; above it the legacy-tensor-path kernel streams
// faster.  Measured per launch in a graph of launches over rotated copies,
// batch 1 (legacy tensor path / CUDA cores, us): 2048 x 2048 3.34 / 2.72,
// 3072 x 3072 4.11 / 3.85, 5120 x 3072 5.02 / 5.21, 3072 x 8192 6.21 / 6.62,
// 16384 x 3072 8.69 / 12.20, 128256 x 3072 45.1 / 75.1.
constexpr int64_t kMmaMinWeights = int64_t(12) << 20;

int launch_gemv(const uint32_t* W, const uint16_t* s, const uint16_t* x, uint16_t* y, int N, int K, int batch,
                cudaStream_t stream)
{
    int dev = 0;
    const DeviceInfo* di = current_device_info(&dev);
    if (!di) return WQ4_ERR_CUDA;
    MmaPlan mp;
    const int path = g_gemv_path.load();
    const bool big = static_cast<int64_t>(N) * K >= kMmaMinWeights;
    if (path != 2 && (big || path == 1) && batch <= 2 && (K % 256) == 0 && aligned(s, 16) &&
        plan_mma(di, N, K, batch, &mp)) {
        GemvMmaParams p;
        p.W = W;
        p.s = s;
        p.x = x;
        p.y = y;
        p.N = N;
        p.K = K;
        p.nslots = mp.nslots;
        p.nbars = mp.nbars;
        p.slot_bytes = mp.slot_bytes;
        p.x_bytes = mp.x_bytes;
        p.spw = mp.spw;
        p.q = mp.q;
        p.err = status_word();
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[0].val.programmaticStreamSerializationAllowed = 1;
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(mp.grid);
        cfg.blockDim = dim3(kMmaThreads);
        cfg.dynamicSmemBytes = mp.smem;
        cfg.stream = stream;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        const cudaError_t e = batch == 1 ? cudaLaunchKernelEx(&cfg, gemv_mma_kernel<1>, p)
                                         : cudaLaunchKernelEx(&cfg, gemv_mma_kernel<2>, p);
        return e == cudaSuccess ? WQ4_OK : WQ4_ERR_CUDA;
    }
    const size_t row_bytes = static_cast<size_t>(K) / 2 + static_cast<size_t>(K) / 16;
    const size_t x_bytes = align_up(static_cast<size_t>(batch) * K * 2, 128);
    const bool fast = batch <= 4 && (K % 256) == 0 && aligned(s, 16) &&
                      kHeaderBytes + x_bytes + 2 * align_up(row_bytes, 128) <= static_cast<size_t>(di->smem_optin);
    if (fast) {
        const int grid = N < di->sm_count ? N : di->sm_count;
        const int rows_per_cta = (N + grid - 1) / grid;
        int rps = static_cast<int>(kTargetSlotBytes / row_bytes);
        if (rps < 1) rps = 1;
        if (rps > rows_per_cta) rps = rows_per_cta;
        size_t slot_bytes = align_up(rps * row_bytes, 128);
        const size_t avail = static_cast<size_t>(di->smem_optin) - kHeaderBytes - x_bytes;
        int nslots = static_cast<int>(avail / slot_bytes);
        while (nslots < 2 && rps > 1) {  // very long rows: fewer rows per slot
            --rps;
            slot_bytes = align_up(rps * row_bytes, 128);
            nslots = static_cast<int>(avail / slot_bytes);
        }
        if (nslots > kMaxSlots) nslots = kMaxSlots;
        GemvTmaParams p;
        p.W = W;
        p.s = s;
        p.x = x;
        p.y = y;
        p.N = N;
        p.K = K;
        p.rows_per_slot = rps;
        p.nslots = nslots;
        p.slot_bytes = static_cast<uint32_t>(slot_bytes);
        p.scales_offset = static_cast<uint32_t>(static_cast<size_t>(rps) * (K / 2));
        p.x_bytes = static_cast<uint32_t>(x_bytes);
        p.err = status_word();
        const size_t smem = kHeaderBytes + x_bytes + static_cast<size_t>(nslots) * slot_bytes;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[0].val.programmaticStreamSerializationAllowed = 1;
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(grid);
        cfg.blockDim = dim3(kGemvThreads);
        cfg.dynamicSmemBytes = smem;
        cfg.stream = stream;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        cudaError_t e;
        switch (batch) {
            case 1: e = cudaLaunchKernelEx(&cfg, gemv_tma_kernel<1>, p); break;
            case 2: e = cudaLaunchKernelEx(&cfg, gemv_tma_kernel<2>, p); break;
            case 3: e = cudaLaunchKernelEx(&cfg, gemv_tma_kernel<3>, p); break;
            default: e = cudaLaunchKernelEx(&cfg, gemv_tma_kernel<4>, p); break;
        }
        if (e != cudaSuccess) return WQ4_ERR_CUDA;
    } else {
        const int warps_per_block = 8;
        int grid = (N + warps_per_block - 1) / warps_per_block;
        const int cap = di->sm_count * 8;
        if (grid > cap) grid = cap;
        if (batch == 1)
            gemv_generic_kernel<1><<<grid, 256, 0, stream>>>(W, s, x, y, N, K, batch);
        else if (batch == 2)
            gemv_generic_kernel<2><<<grid, 256, 0, stream>>>(W, s, x, y, N, K, batch);
        else if (batch <= 4)
            gemv_generic_kernel<4><<<grid, 256, 0, stream>>>(W, s, x, y, N, K, batch);
        else
            gemv_generic_kernel<8><<<grid, 256, 0, stream>>>(W, s, x, y, N, K, batch);
    }
    return cudaGetLastError() == cudaSuccess ? WQ4_OK : WQ4_ERR_CUDA;
}

int check_matrix_args(const uint32_t* W, const uint16_t* s, int N, int K)
{
    if (!W || !s) return WQ4_ERR_INVALID;
    if (N < 1 || K < 32 || (K % 32) != 0) return WQ4_ERR_INVALID;
    if (static_cast<int64_t>(N) * K / 8 > (static_cast<int64_t>(1) << 40)) return WQ4_ERR_INVALID;
    if (!aligned(W, 16) || !aligned(s, 2)) return WQ4_ERR_ALIGN;
    return WQ4_OK;
}

}  // namespace
}  // namespace wq4

using namespace wq4;

extern "C" int wq4_gemv(const uint32_t* W_packed, const uint16_t* scales, const uint16_t* x, uint16_t* y, int N,
                        int K, int batch, void* stream)
{
    int rc = check_matrix_args(W_packed, scales, N, K);
    if (rc != WQ4_OK) return rc;
    if (!x || !y || batch < 1 || batch > WQ4_MAX_BATCH) return WQ4_ERR_INVALID;
    if (!aligned(x, 16) || !aligned(y, 2)) return WQ4_ERR_ALIGN;
    const size_t yb = static_cast<size_t>(batch) * N * 2, xb = static_cast<size_t>(batch) * K * 2;
    const size_t wb = static_cast<size_t>(N) * K / 2, sb = static_cast<size_t>(N) * K / 16;
    if (overlaps(y, yb, x, xb) || overlaps(y, yb, W_packed, wb) || overlaps(y, yb, scales, sb))
        return WQ4_ERR_INVALID;
    return launch_gemv(W_packed, scales, x, y, N, K, batch, static_cast<cudaStream_t>(stream));
}

extern "C" int wq4_test_gemv_path(int path)
{
    if (path < 0 || path > 2) return WQ4_ERR_INVALID;
    g_gemv_path.store(path);
    return WQ4_OK;
}

extern "C" int wq4_unpack_debug(const uint32_t* W_packed, const uint16_t* scales, float* w_out, uint8_t* q_out,
                                int N, int K, void* stream)
{
    int rc = check_matrix_args(W_packed, scales, N, K);
    if (rc != WQ4_OK) return rc;
    if (!w_out && !q_out) return WQ4_ERR_INVALID;
    if (w_out && !aligned(w_out, 4)) return WQ4_ERR_ALIGN;
    int dev = 0;
    const DeviceInfo* di = current_device_info(&dev);
    if (!di) return WQ4_ERR_CUDA;
    const int64_t words = static_cast<int64_t>(N) * (K / 8);
    int64_t blocks = (words + 255) / 256;
    if (blocks > static_cast<int64_t>(di->sm_count) * 16) blocks = static_cast<int64_t>(di->sm_count) * 16;
    unpack_debug_kernel<<<static_cast<int>(blocks), 256, 0, static_cast<cudaStream_t>(stream)>>>(W_packed, scales,
                                                                                                  w_out, q_out, N, K);
    return cudaGetLastError() == cudaSuccess ? WQ4_OK : WQ4_ERR_CUDA;
}

extern "C" int wq4_pack_host(const uint8_t* q_host, uint32_t* W_host, int N, int K)
{
    if (!q_host || !W_host || N < 1 || K < 8 || (K % 8) != 0) return WQ4_ERR_INVALID;
    for (int64_t n = 0; n < N; ++n) {
        for (int j = 0; j < K / 8; ++j) {
            uint32_t word = 0;
            for (int i = 0; i < 8; ++i) {
                const uint8_t q = q_host[n * K + 8 * j + i];
                if (q > 15) return WQ4_ERR_INVALID;
                word |= static_cast<uint32_t>(q) << (4 * i);
            }
            W_host[n * (K / 8) + j] = word;
        }
    }
    return WQ4_OK;
}

extern "C" const char* wq4_status_string(int status)
{
    switch (status) {
        case WQ4_OK: return "ok";
        case WQ4_ERR_INVALID: return "invalid argument";
        case WQ4_ERR_ALIGN: return "misaligned pointer";
        case WQ4_ERR_UNSUPPORTED: return "unsupported configuration";
        case WQ4_ERR_CUDA: return "CUDA runtime error";
        case WQ4_ERR_TIMEOUT: return "device-side wait timed out";
        default: return "unknown status";
    }
}

extern "C" int wq4_device_status(void* stream, int* flags_out)
{
    uint32_t* w = status_word();
    if (!w) return WQ4_ERR_CUDA;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    uint32_t v = 0;
    if (cudaMemcpyAsync(&v, w, sizeof(v), cudaMemcpyDeviceToHost, st) != cudaSuccess) return WQ4_ERR_CUDA;
    if (cudaMemsetAsync(w, 0, sizeof(uint32_t), st) != cudaSuccess) return WQ4_ERR_CUDA;
    if (cudaStreamSynchronize(st) != cudaSuccess) return WQ4_ERR_CUDA;
    if (flags_out) *flags_out = static_cast<int>(v);
    return v ? WQ4_ERR_TIMEOUT : WQ4_OK;
}
