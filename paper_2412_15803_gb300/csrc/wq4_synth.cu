// wq4_synth.cu -- device-side seeded generator of synthetic packed weights.
//
// Not part of the method: it draws the same counter-based SplitMix64 bits as
// the host generator (Steele, Lea and Flood, OOPSLA 2014) so that multi-GB
// synthetic models can be created directly in device memory.  Each output
// element depends only on (seed, stream id, index).
#include "wq4_synth.h"

#include <cuda_runtime.h>

#include <cstdint>

namespace {

constexpr uint64_t kGamma = 0x9E3779B97F4A7C15ull;
constexpr uint64_t kSidMul = 0xD1B54A32D192ED03ull;

__host__ __device__ __forceinline__ uint64_t mix64(uint64_t z)
{
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

uint64_t stream_key(uint64_t seed, uint64_t sid)
{
    return mix64(seed * kGamma + sid * kSidMul);
}

// Every 4-bit field equal to 15 becomes 7 (bit 3 cleared where all four bits
// are set): codes 0..14 with mean 7.
__device__ __forceinline__ uint32_t fold15(uint32_t w)
{
    const uint32_t m = w & (w >> 1) & (w >> 2) & (w >> 3) & 0x11111111u;
    return w ^ (m << 3);
}

__global__ void codes_kernel(uint32_t* __restrict__ W, int64_t pair_start, int64_t npairs, uint64_t key,
                             int symmetric)
{
    for (int64_t t = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; t < npairs;
         t += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const uint64_t v = mix64(key + static_cast<uint64_t>(pair_start + t + 1) * kGamma);
        uint32_t lo = static_cast<uint32_t>(v), hi = static_cast<uint32_t>(v >> 32);
        if (symmetric) {
            lo = fold15(lo);
            hi = fold15(hi);
        }
        reinterpret_cast<uint2*>(W)[t] = make_uint2(lo, hi);
    }
}

__global__ void scales_kernel(uint16_t* __restrict__ s, int64_t start, int64_t n, uint64_t key, double lo,
                              double span)
{
    for (int64_t t = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; t < n;
         t += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const uint64_t v = mix64(key + static_cast<uint64_t>(start + t + 1) * kGamma);
        const double u = static_cast<double>(v >> 11) * 0x1.0p-53;
        const double x = __dadd_rn(lo, __dmul_rn(span, u));   // no contraction into an fma
        unsigned short h;
        asm("cvt.rn.f16.f64 %0, %1;" : "=h"(h) : "d"(x));   // one rounding, to nearest even
        s[t] = h;
    }
}

// sum4: fp16_RNE((a + b + c + d - 131070) * 2^-15), a..d the four 16-bit
// fields of u64(key, i); integer arithmetic then a single rounding.
__global__ void sum4_kernel(uint16_t* __restrict__ out, int64_t start, int64_t n, uint64_t key)
{
    for (int64_t t = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; t < n;
         t += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const uint64_t v = mix64(key + static_cast<uint64_t>(start + t + 1) * kGamma);
        const int64_t c = static_cast<int64_t>((v & 0xFFFF) + ((v >> 16) & 0xFFFF) + ((v >> 32) & 0xFFFF) + (v >> 48)) -
                          131070;
        const double x = static_cast<double>(c) * 0x1.0p-15;   // exact
        unsigned short h;
        asm("cvt.rn.f16.f64 %0, %1;" : "=h"(h) : "d"(x));
        out[t] = h;
    }
}

int grid_for(int64_t n)
{
    int64_t b = (n + 255) / 256;
    if (b > 65536) b = 65536;
    return b < 1 ? 1 : static_cast<int>(b);
}

}  // namespace

extern "C" int wq4_synth_codes(uint32_t* W, int64_t word_start, int64_t nwords, uint64_t seed, uint64_t sid,
                               int symmetric, void* stream)
{
    if (!W || word_start < 0 || nwords < 0 || (word_start % 2) || (nwords % 2)) return -1;
    if (reinterpret_cast<uintptr_t>(W) % 8) return -1;
    if (nwords == 0) return 0;
    const int64_t npairs = nwords / 2;
    codes_kernel<<<grid_for(npairs), 256, 0, static_cast<cudaStream_t>(stream)>>>(W, word_start / 2, npairs,
                                                                                  stream_key(seed, sid), symmetric);
    return cudaGetLastError() == cudaSuccess ? 0 : -4;
}

extern "C" int wq4_synth_scales(uint16_t* s, int64_t start, int64_t n, uint64_t seed, uint64_t sid, double lo,
                                double hi, void* stream)
{
    if (!s || start < 0 || n < 0 || !(hi >= lo)) return -1;
    if (n == 0) return 0;
    scales_kernel<<<grid_for(n), 256, 0, static_cast<cudaStream_t>(stream)>>>(s, start, n, stream_key(seed, sid),
                                                                               lo, hi - lo);
    return cudaGetLastError() == cudaSuccess ? 0 : -4;
}

extern "C" int wq4_synth_sum4(uint16_t* out, int64_t start, int64_t n, uint64_t seed, uint64_t sid, void* stream)
{
    if (!out || start < 0 || n < 0) return -1;
    if (n == 0) return 0;
    sum4_kernel<<<grid_for(n), 256, 0, static_cast<cudaStream_t>(stream)>>>(out, start, n, stream_key(seed, sid));
    return cudaGetLastError() == cudaSuccess ? 0 : -4;
}
