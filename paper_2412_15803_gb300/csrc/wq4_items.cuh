// wq4_items.cuh -- the work item of the batch 1-2 weight stream on the legacy
// tensor path (mma.sync m16n8k16), shared by the persistent decode chain
// (wq4_chain.cu) and the single-projection GEMV (wq4_gemv.cu).
//
// A work item multiplies row pairs (codes and scales staged in shared memory)
// by the activations staged once per projection in the MMA's pair-permuted
// order: exact fp16 (q - 7) as the A operand, eight 32-code groups of x as
// the eight B columns, the wanted sums on the diagonal, scaled by the group
// scales in fp32.
#pragma once

#include "wq4_device.cuh"

namespace wq4 {

// Exact floor(n / d) for 0 <= n, d < 2^24 from a float reciprocal: the
// product is within 2^-9 of n / d for the quotients used here (< 2^14), so
// one correction step gives the floor.  No integer division on the path.
struct FDiv {
    float r;
    int d;
};
__device__ __forceinline__ FDiv fdiv_make(int d)
{
    FDiv f;
    f.d = d;
    f.r = __frcp_rn(static_cast<float>(d));
    return f;
}
__device__ __forceinline__ int fdiv(int n, const FDiv& f)
{
    int q = __float2int_rz(static_cast<float>(n) * f.r);
    if (q * f.d > n) --q;
    else if ((q + 1) * f.d <= n) ++q;
    return q;
}

__device__ __forceinline__ float lo_f(uint32_t v) { return half_bits_to_float(static_cast<uint16_t>(v & 0xFFFFu)); }
__device__ __forceinline__ float hi_f(uint32_t v) { return half_bits_to_float(static_cast<uint16_t>(v >> 16)); }
__device__ __forceinline__ uint32_t pack2(uint16_t a, uint16_t b)
{
    return static_cast<uint32_t>(a) | (static_cast<uint32_t>(b) << 16);
}

// Eight consecutive activations x0..x7 (four words of two) in the order the
// MMA's B fragment takes them: (x0, x4), (x1, x5), (x2, x6), (x3, x7) -- the
// pairing of unpack_word's outputs.
__device__ __forceinline__ uint4 pair_permute(uint4 v)
{
    return make_uint4(__byte_perm(v.x, v.z, 0x5410), __byte_perm(v.x, v.z, 0x7632), __byte_perm(v.y, v.w, 0x5410),
                      __byte_perm(v.y, v.w, 0x7632));
}

// The units of one item for NP row pairs (smem code rows ca[], cb[], scale
// rows sa[], sb[]): for each group set j (256 codes) in [j0, j1), two
// m16n8k16 MMAs per pair over its 16 (row, group) combinations and the eight
// groups' activations (loaded once for all pairs), then the scaled diagonal
// into acc[pair][b] (lanes 0, 5, 10, 15 hold row a's partial sums, lanes 16,
// 21, 26, 31 row b's).
//
// Lane (g, c) = (lane >> 2, lane & 3).  A row m of the MMA is (row, group
// 8j + sigma): m = g < 4: (a, 2g); m = g + 8 < 12: (a, 2g + 1); m = g >= 4:
// (b, 2g - 7); m = g + 8 >= 12: (b, 2g - 8).  The pairing of rows a and b with
// odd and even groups puts the eight 16-byte rows of each ldmatrix on
// distinct bank quads.  B column sigma holds group 8j + sigma of x, so the
// wanted sums sit on the diagonal D[m][sigma(m)]: lanes 5g (g < 4) hold them
// in d0 (even group) and d3 (odd group), lanes 5g - 4 (g >= 4) in d2 and d1.
template <int B, int NP>
__device__ __forceinline__ void item_units(const uint32_t (&ca)[NP], const uint32_t (&cb)[NP], const uint32_t (&sa)[NP],
                                           const uint32_t (&sb)[NP], uint32_t xs, int cpr, int j0, int j1,
                                           float (&acc)[NP][B])
{
    const int lane = threadIdx.x & 31;
    const int g = lane >> 2, c = lane & 3;
    const bool hi = g >= 4;
    // this lane's ldmatrix row address: matrix lane >> 3 (0: A rows g, 1: A rows g + 8)
    const int t = lane & 7, mi = (lane >> 3) & 1;
    const int goff = (t < 4) ? (2 * t + mi) : (2 * (t - 4) + 1 - mi);
    uint32_t lb[NP], sbs[NP];
#pragma unroll
    for (int pr = 0; pr < NP; ++pr) {
        lb[pr] = ((t < 4) ? ca[pr] : cb[pr]) + 16 * goff;
        sbs[pr] = (hi ? sb[pr] : sa[pr]) + 4 * c;
    }
    const uint32_t xbase = xs + 16 * lane;
    const float zero[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll(B == 1 || NP == 1 ? 2 : 1)   // two group sets an iteration at batch 1 (measured ~1 % faster), not at 2
    for (int j = j0; j < j1; ++j) {
        uint4 xv[B];
#pragma unroll
        for (int b = 0; b < B; ++b) xv[b] = lds_v4(xbase + 16 * (b * cpr + 32 * j));
        uint32_t r0[NP], r1[NP], sw[NP];
#pragma unroll
        for (int pr = 0; pr < NP; ++pr) {
            ldsm_x2(lb[pr] + 128 * j, r0[pr], r1[pr]);
            sw[pr] = lds_u32(sbs[pr] + 16 * j);
        }
#pragma unroll
        for (int pr = 0; pr < NP; ++pr) {
            uint32_t pa[4], pb[4];
            unpack_word(r0[pr], pa);
            unpack_word(r1[pr], pb);
            const float se = lo_f(sw[pr]), so = hi_f(sw[pr]);
#pragma unroll
            for (int b = 0; b < B; ++b) {
                float d[4];
                mma_16816(d, pa[0], pb[0], pa[1], pb[1], xv[b].x, xv[b].y, zero);
                mma_16816(d, pa[2], pb[2], pa[3], pb[3], xv[b].z, xv[b].w, d);
                const float ve = hi ? d[2] : d[0];
                const float vo = hi ? d[1] : d[3];
                acc[pr][b] = fmaf(se, ve, fmaf(so, vo, acc[pr][b]));
            }
        }
    }
}

// Row sums of a row pair from item_units: lane 0 gets row a, lane 16 row b.
__device__ __forceinline__ float pair_reduce(float v)
{
    v += __shfl_down_sync(0xffffffffu, v, 5);
    v += __shfl_down_sync(0xffffffffu, v, 10);
    return v;
}

}  // namespace wq4
