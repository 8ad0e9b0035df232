// wq4_device.cuh -- device building blocks of the weight-streaming kernels
// (sm_103a): mbarrier / bulk-copy PTX, the in-register int4 unpack and the
// fp16 x fp16 -> fp32 multiply-accumulate.
//
// The decode step of a 4-bit model (Section 3, Table 1) reads every packed
// weight once; what this header provides is the register path of one packed
// word: 8 codes -> 8 exact fp16 values (q - 7) -> 8 products with x
// accumulated in fp32.  Dequantization never touches memory: that is the
// "kernel fusion" of Section 2.3 done by hand.
#pragma once

#include <cstdint>
#include <cuda_fp16.h>

namespace wq4 {

// Bits of the library's device status word.
constexpr uint32_t kErrPipeTimeout = 1u;   // an mbarrier wait gave up
constexpr uint32_t kErrFlagTimeout = 2u;   // a wait on another CTA's data gave up
constexpr uint32_t kErrSeqLen = 8u;        // attention: a length beyond the page table (clamped)
constexpr uint32_t kErrPageId = 16u;       // attention: a page id outside the pool (zeros read)
constexpr uint32_t kErrAppend = 32u;       // append: bad position or page id (row not written)
constexpr uint32_t kErrScale = 64u;        // a scale beyond +-8188 met an fp16 dequantized-weight path

// Largest fp16 scale magnitude whose dequantized weights (q - 7) s, |q - 7|
// <= 8, stay finite in fp16 (8 * 8188 = 65504, the fp16 maximum; the next
// fp16 value, 8192, overflows).  As the bits of |s|: 0x6FFF.
constexpr uint32_t kMaxFp16ScaleBits = 0x6FFFu;

// Every spin-wait gives up after this long (a legitimate wait lasts
// microseconds); the kernel then records the error and runs to its end.
constexpr unsigned long long kWaitTimeoutNs = 500ull * 1000ull * 1000ull;

__device__ __forceinline__ uint64_t globaltimer_ns()
{
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

__device__ __forceinline__ uint32_t smem_addr(const void* p)
{
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// ------------------------------------------------------------- mbarrier --

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count) : "memory");
}

// Makes barrier initialisation visible to the bulk-copy (async) proxy.
__device__ __forceinline__ void mbar_fence_init()
{
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes)
{
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;"
                 ::"r"(smem_addr(bar)), "r"(bytes) : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar)
{
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(bar)) : "memory");
}

__device__ __forceinline__ void mbar_arrive_count(uint64_t* bar, uint32_t count)
{
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity)
{
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_addr(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}

// Waits for the phase of `bar` with the given parity to complete.  Bounded:
// after kWaitTimeoutNs it sets kErrPipeTimeout in *err and returns false.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, uint32_t* err)
{
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = globaltimer_ns();
    for (;;) {
        if (mbar_try_wait(bar, parity)) return true;
        if (globaltimer_ns() - t0 > kWaitTimeoutNs) {
            atomicOr(err, kErrPipeTimeout);
            return false;
        }
    }
}

// ------------------------------------------------------------ bulk copy --

// L2 policy for data read exactly once per token (the weights): evict first,
// so the stream does not push activations and flags out of L2.
__device__ __forceinline__ uint64_t l2_policy_evict_first()
{
    uint64_t pol;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
    return pol;
}

// One-dimensional bulk copy global -> shared (TMA unit), completing `bytes`
// transactions on `bar`.  dst, src 16-byte aligned; bytes a multiple of 16.
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar,
                                         uint64_t policy)
{
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
        " [%0], [%1], %2, [%3], %4;" ::"r"(smem_addr(dst)),
        "l"(src), "r"(bytes), "r"(smem_addr(bar)), "l"(policy)
        : "memory");
}

__device__ __forceinline__ void named_barrier_sync(int id, int nthreads)
{
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}

// --------------------------------------------------------------- unpack --

__device__ __forceinline__ uint32_t lop3_and_or(uint32_t a, uint32_t b, uint32_t c)
{
    uint32_t d;  // (a & b) | c
    asm("lop3.b32 %0, %1, %2, %3, 0xEA;" : "=r"(d) : "r"(a), "r"(b), "r"(c));
    return d;
}

__device__ __forceinline__ uint32_t hsub2_u32(uint32_t a, uint32_t b)
{
    uint32_t d;
    asm("sub.rn.f16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
    return d;
}

__device__ __forceinline__ uint32_t hfma2_u32(uint32_t a, uint32_t b, uint32_t c)
{
    uint32_t d;
    asm("fma.rn.f16x2 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(c));
    return d;
}

// One packed word (codes k = 0..7 of the word, lowest nibble first) to four
// fp16x2 registers holding the exact values q - 7:
//   p[0] = (k0, k4)   p[1] = (k1, k5)   p[2] = (k2, k6)   p[3] = (k3, k7)
// The 0x6400 exponent makes a nibble OR-ed into the mantissa read as 1024 + q
// (mask 0x000F) or 1024 + 16q (mask 0x00F0); one subtraction or one fma
// (x/16 - 71) then gives q - 7 exactly.  5 integer ops + 4 fp16x2 ops for 8
// weights.
__device__ __forceinline__ void unpack_word(uint32_t w, uint32_t p[4])
{
    constexpr uint32_t kMagic = 0x64006400u;   // 1024.0 in both halves
    constexpr uint32_t k1031 = 0x64076407u;    // 1031.0 = 1024 + 7
    constexpr uint32_t kSixteenth = 0x2C002C00u;  // 1/16
    constexpr uint32_t kMinus71 = 0xD470D470u;    // -71 = -(1024/16) - 7
    const uint32_t lo0 = lop3_and_or(w, 0x000F000Fu, kMagic);
    const uint32_t hi0 = lop3_and_or(w, 0x00F000F0u, kMagic);
    const uint32_t w8 = w >> 8;
    const uint32_t lo1 = lop3_and_or(w8, 0x000F000Fu, kMagic);
    const uint32_t hi1 = lop3_and_or(w8, 0x00F000F0u, kMagic);
    p[0] = hsub2_u32(lo0, k1031);
    p[1] = hfma2_u32(hi0, kSixteenth, kMinus71);
    p[2] = hsub2_u32(lo1, k1031);
    p[3] = hfma2_u32(hi1, kSixteenth, kMinus71);
}

// acc + sum_{i<8} (q_i - 7) * x_i with p from unpack_word and xv = x[0..7]
// (fp16, consecutive).  Each product of two fp16 values is exact in fp32 and
// is added in fp32 (mixed-precision fma, sm_100+): no fp16 rounding of
// products or partial sums.
__device__ __forceinline__ float fma8(const uint32_t p[4], uint4 xv, float acc)
{
    asm("{\n\t.reg .f16 a0, a1, a2, a3, a4, a5, a6, a7, x0, x1, x2, x3, x4, x5, x6, x7;\n\t"
        "mov.b32 {a0, a4}, %1;\n\t"
        "mov.b32 {a1, a5}, %2;\n\t"
        "mov.b32 {a2, a6}, %3;\n\t"
        "mov.b32 {a3, a7}, %4;\n\t"
        "mov.b32 {x0, x1}, %5;\n\t"
        "mov.b32 {x2, x3}, %6;\n\t"
        "mov.b32 {x4, x5}, %7;\n\t"
        "mov.b32 {x6, x7}, %8;\n\t"
        "fma.rn.f32.f16 %0, a0, x0, %0;\n\t"
        "fma.rn.f32.f16 %0, a1, x1, %0;\n\t"
        "fma.rn.f32.f16 %0, a2, x2, %0;\n\t"
        "fma.rn.f32.f16 %0, a3, x3, %0;\n\t"
        "fma.rn.f32.f16 %0, a4, x4, %0;\n\t"
        "fma.rn.f32.f16 %0, a5, x5, %0;\n\t"
        "fma.rn.f32.f16 %0, a6, x6, %0;\n\t"
        "fma.rn.f32.f16 %0, a7, x7, %0;\n\t}"
        : "+f"(acc)
        : "r"(p[0]), "r"(p[1]), "r"(p[2]), "r"(p[3]), "r"(xv.x), "r"(xv.y), "r"(xv.z), "r"(xv.w));
    return acc;
}

// Position (in uint4 units) of the 8-element chunk j (0..3) of group g of an
// activation row staged in shared memory.  The chunk index is XOR-swizzled
// with (g >> 1) & 3 so that 8 lanes reading 8 consecutive groups hit 8
// distinct 16-byte bank quads.
__device__ __forceinline__ int x_chunk(int g, int j)
{
    return g * 4 + (j ^ ((g >> 1) & 3));
}

// Dot product of one group (32 codes in cw, scale sc) with B activation rows
// staged (swizzled) in shared memory at xs (uint4 units, row stride K/8).
// racc[b] += sc * sum_{i<32} (q_i - 7) x_b[i].
template <int B>
__device__ __forceinline__ void group_dot_smem(uint4 cw, float sc, const uint4* xs, int row_stride_u4,
                                               int g, float racc[B])
{
    uint32_t p[16];
    unpack_word(cw.x, p + 0);
    unpack_word(cw.y, p + 4);
    unpack_word(cw.z, p + 8);
    unpack_word(cw.w, p + 12);
#pragma unroll
    for (int b = 0; b < B; ++b) {
        const uint4* xb = xs + b * row_stride_u4;
        const float a0 = fma8(p + 0, xb[x_chunk(g, 0)], 0.f);
        const float a1 = fma8(p + 4, xb[x_chunk(g, 1)], 0.f);
        const float a2 = fma8(p + 8, xb[x_chunk(g, 2)], 0.f);
        const float a3 = fma8(p + 12, xb[x_chunk(g, 3)], 0.f);
        racc[b] = fmaf(sc, (a0 + a1) + (a2 + a3), racc[b]);
    }
}

// ------------------------------------------------ legacy tensor-core path --

// Two 8x8 b16 matrices from shared memory: lane t (t < 16) supplies the
// address of row t & 7 of matrix t >> 3 (16-byte aligned); lane (g, c) =
// (lane >> 2, lane & 3) receives bytes 4c..4c+3 of row g of each matrix.
__device__ __forceinline__ void ldsm_x2(uint32_t addr, uint32_t& r0, uint32_t& r1)
{
    asm volatile("ldmatrix.sync.aligned.m8n8.x2.shared.b16 {%0, %1}, [%2];" : "=r"(r0), "=r"(r1) : "r"(addr) : "memory");
}

__device__ __forceinline__ uint32_t lds_u32(uint32_t addr)
{
    uint32_t v;
    asm volatile("ld.shared.b32 %0, [%1];" : "=r"(v) : "r"(addr) : "memory");
    return v;
}

__device__ __forceinline__ uint4 lds_v4(uint32_t addr)
{
    uint4 v;
    asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(addr) : "memory");
    return v;
}

// D = A (16x16, fp16, row-major fragment a[0..3]) * B (16x8, fp16, column
// fragment b0, b1) + C, fp32 accumulation.  Fragments of lane (g, c):
// a = {A[g][2c..2c+1], A[g+8][2c..2c+1], A[g][2c+8..2c+9], A[g+8][2c+8..2c+9]},
// b0 = B[2c..2c+1][g], b1 = B[2c+8..2c+9][g],
// d = {D[g][2c], D[g][2c+1], D[g+8][2c], D[g+8][2c+1]}.
// fp16 x fp16 products are exact in fp32.
__device__ __forceinline__ void mma_16816(float d[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3, uint32_t b0,
                                          uint32_t b1, const float c[4])
{
    asm("mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%10,%11,%12,%13};"
        : "=f"(d[0]), "=f"(d[1]), "=f"(d[2]), "=f"(d[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1), "f"(c[0]), "f"(c[1]), "f"(c[2]), "f"(c[3]));
}

__device__ __forceinline__ float warp_sum(float v)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

__device__ __forceinline__ float half_bits_to_float(uint16_t h)
{
    return __half2float(__ushort_as_half(h));
}

__device__ __forceinline__ uint16_t float_to_half_bits(float f)
{
    return __half_as_ushort(__float2half_rn(f));
}

}  // namespace wq4
