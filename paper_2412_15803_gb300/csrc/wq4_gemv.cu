// wq4_gemv.cu -- the fused dequantize x GEMV of one decode step and the
// C-ABI entry points that do not belong to the chain.
//
// y[b][n] = fp16( sum_k (q(n,k) - 7) * s[n][k/32] * x[b][k] ), the projection
// every decoded token applies to every 4-bit weight matrix (Section 3,
// Table 1).  Two kernels:
//
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
#include "wq4_host.h"
#include "wq4.h"

#include <cuda_runtime.h>

#include <mutex>

namespace wq4 {

__device__ uint32_t g_status_word;

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

    // ---------------- consumers: stage x (swizzled) once
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
            !set_tma_attr<4>(d.smem_optin))
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

int launch_gemv(const uint32_t* W, const uint16_t* s, const uint16_t* x, uint16_t* y, int N, int K, int batch,
                cudaStream_t stream)
{
    int dev = 0;
    const DeviceInfo* di = current_device_info(&dev);
    if (!di) return WQ4_ERR_CUDA;
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
        switch (batch) {
            case 1: gemv_tma_kernel<1><<<grid, kGemvThreads, smem, stream>>>(p); break;
            case 2: gemv_tma_kernel<2><<<grid, kGemvThreads, smem, stream>>>(p); break;
            case 3: gemv_tma_kernel<3><<<grid, kGemvThreads, smem, stream>>>(p); break;
            default: gemv_tma_kernel<4><<<grid, kGemvThreads, smem, stream>>>(p); break;
        }
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
