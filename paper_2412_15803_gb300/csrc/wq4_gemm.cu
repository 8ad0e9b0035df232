// wq4_gemm.cu -- the 4-bit dequantize-and-multiply for many activation rows
// (prefill-shaped M: a prompt's tokens through one projection), on the
// tcgen05 tensor cores of sm_103a.
//
// Y[m][n] = fp16( sum_k x[m][k] * fp16((q(n,k) - 7) * s(n, k/32)) ), fp32 sums.
//
// A persistent grid walks (128 weight rows x T tokens) tiles, T = 128, 192 or
// 256 chosen per call (pick_tok), row tile major so that the CTAs running at
// one time share a weight tile through L2.  Per 64-wide K chunk a producer
// warp brings the tile's codes and scales (2-D tensor copies) and the T x 64
// activation block (one 128-byte swizzled box) into a ring of 4-6 slots
// (small slots, so that copies stay in flight while the MMAs of earlier
// chunks run); eight dequant warps write the 128 x 64 weights, dequantized to
// fp16 in natural K order, into one of three 32-column A buffers in tensor
// memory (lane = weight row); one thread issues 4 tcgen05.mma (kind::f16,
// M = 128, N = T tokens, K = 16: at T = 256 the tensor-core rate, ~128 cycles
// each, so the dequant warps keep up) into a T-column fp32 accumulator; four
// epilogue warps move a finished accumulator into a shared-memory transpose
// buffer, release it, and store T tokens x 128 outputs with 16-byte stores
// while the next tile's MMAs run.  Every weight is rounded to fp16 once
// (relative error <= 2^-11, accumulated in fp32): within the library's
// accuracy contract.
#include "wq4.h"
#include "wq4_device.cuh"
#include "wq4_host.h"
#include "wq4_tc.cuh"

#include <cuda.h>
#include <cuda_runtime.h>

#include <cstring>
#include <mutex>

namespace wq4 {
namespace {

constexpr int kGThreads = 448;        // warps 0-7 dequant, 8 producer, 9 MMA, 10-13 epilogue
constexpr int kGProducer = 8, kGIssuer = 9;
constexpr int kGCodes = 128 * 32;     // 128 rows x 64 codes (32-byte rows, 32-byte swizzle)
constexpr int kGScales = 128 * 16;    // 128 rows x 8 fp16 scales (the 256-wide K block of the chunk)
constexpr int kGABufs = 3;            // 32-column A buffers
constexpr int kGDCol = 256;           // accumulator: TOK columns
constexpr int kGT = 1024;             // transpose buffer: TOK tokens x 128 outputs fp16
constexpr int kGTmemCols = 512;

// Tile of TOK tokens (MMA N = 128, 192 or 256).
template <int TOK>
struct GCfg {
    static constexpr int kSlots = TOK == 256 ? 4 : (TOK == 192 ? 5 : 6);
    static constexpr int kX = TOK * 64 * 2;                // activation block: TOK tokens x 64 K fp16
    static constexpr int kSlot = kX + kGCodes + kGScales;  // a multiple of 1024
    static constexpr int kRing = kGT + TOK * 128 * 2;
    static constexpr int kSmem = kRing + kSlots * kSlot;
    static_assert(kSmem <= 227 * 1024, "shared memory");
};

struct GemmArgs {
    uint16_t* y;
    int N, K, M, rtiles, ttiles;
    uint32_t* err;
};

__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t sel)
{
    uint32_t d;
    asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(sel));
    return d;
}

__device__ __forceinline__ bool g_wait(uint64_t* bar, uint32_t parity, uint32_t* err)
{
    return mbar_wait(bar, parity, err);
}

template <int TOK>
__global__ void __launch_bounds__(kGThreads, 1)
    gemm_kernel(const __grid_constant__ CUtensorMap tm_codes, const __grid_constant__ CUtensorMap tm_scales,
                const __grid_constant__ CUtensorMap tm_x, const GemmArgs a)
{
    using C = GCfg<TOK>;
    constexpr int kGSlots = C::kSlots, kGX = C::kX, kGSlot = C::kSlot, kGRing = C::kRing, kGTok = TOK;
    extern __shared__ __align__(1024) uint8_t smem[];
    uint64_t* full = reinterpret_cast<uint64_t*>(smem);      // codes, scales, activations landed
    uint64_t* empty = full + kGSlots;
    uint64_t* afull = empty + kGSlots;
    uint64_t* aempty = afull + kGABufs;
    uint64_t* dfull = aempty + kGABufs;
    uint64_t* dempty = dfull + 1;
    uint64_t* drain = dempty + 1;                            // ends at byte (2 slots + 9) * 8 <= 240
    uint32_t* tbase_sh = reinterpret_cast<uint32_t*>(smem + 240);
    uint16_t* tbuf = reinterpret_cast<uint16_t*>(smem + kGT);
    uint8_t* ring = smem + kGRing;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nch = a.K >> 6;   // 64-wide K chunks
    const int tiles = a.rtiles * a.ttiles;
    uint32_t* err = a.err;

    if (threadIdx.x == 0) {
        for (int i = 0; i < kGSlots; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], 9);   // 8 dequant warps + the MMA commit
        }
        for (int i = 0; i < kGABufs; ++i) {
            mbar_init(&afull[i], 8);
            mbar_init(&aempty[i], 1);
        }
        mbar_init(dfull, 1);
        mbar_init(dempty, 4);
        mbar_init(drain, 1);
        mbar_fence_init();
    }
    if (warp == kGIssuer) tc::tmem_alloc(tbase_sh, kGTmemCols);
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    const uint32_t tbase = *tbase_sh;

    if (warp == kGProducer) {
        // ---------------------------------------------------- producer
        if (lane == 0) {
            tc::prefetch_map(&tm_codes);
            tc::prefetch_map(&tm_scales);
            tc::prefetch_map(&tm_x);
            int it = 0;
            bool ok = true;
            for (int u = blockIdx.x; u < tiles && ok; u += gridDim.x) {
                const int n0 = (u / a.ttiles) * 128, m0 = (u % a.ttiles) * kGTok;
                for (int c = 0; c < nch; ++c, ++it) {
                    const int slot = it % kGSlots;
                    if (it >= kGSlots && !g_wait(&empty[slot], ((it / kGSlots) - 1) & 1, err)) {
                        ok = false;
                        break;
                    }
                    uint8_t* base = ring + static_cast<size_t>(slot) * kGSlot;
                    mbar_arrive_expect_tx(&full[slot], kGSlot);
                    tc::tma_load_2d(base, &tm_x, c * 64, m0, &full[slot]);
                    tc::tma_load_2d(base + kGX, &tm_codes, c * 32, n0, &full[slot]);
                    tc::tma_load_2d(base + kGX + 64 * 32, &tm_codes, c * 32, n0 + 64, &full[slot]);
                    tc::tma_load_2d(base + kGX + kGCodes, &tm_scales, (c >> 2) * 8, n0, &full[slot]);
                    tc::tma_load_2d(base + kGX + kGCodes + 64 * 16, &tm_scales, (c >> 2) * 8, n0 + 64, &full[slot]);
                }
            }
            // every copy issued has landed before the CTA's memory goes away
            const int first = it > kGSlots ? it - kGSlots : 0;
            for (int i = first; i < it; ++i) g_wait(&full[i % kGSlots], (i / kGSlots) & 1, err);
        }
    } else if (warp == kGIssuer) {
        // ---------------------------------------------------- MMA issuer
        if (lane == 0) {
            constexpr uint32_t idesc = tc::idesc_f16_f32(128, kGTok);
            int it = 0, dit = 0;
            bool ok = true;
            const uint32_t dt = tbase + kGDCol;
            for (int u = blockIdx.x; u < tiles && ok; u += gridDim.x, ++dit) {
                if (dit >= 1 && !g_wait(dempty, (dit - 1) & 1, err)) break;
                tc::fence_after_sync();
                for (int c = 0; c < nch; ++c, ++it) {
                    const int slot = it % kGSlots, abuf = it % kGABufs;
                    if (!g_wait(&full[slot], (it / kGSlots) & 1, err) ||
                        !g_wait(&afull[abuf], (it / kGABufs) & 1, err)) {
                        ok = false;
                        break;
                    }
                    tc::fence_after_sync();
                    const uint32_t xs = smem_addr(ring + static_cast<size_t>(slot) * kGSlot);
#pragma unroll
                    for (int s = 0; s < 4; ++s) {
                        const uint64_t bd = tc::sw128_kmajor_desc(xs + 32 * s);
                        tc::mma_f16_ts(dt, tbase + 32 * abuf + 8 * s, bd, idesc, (c > 0 || s > 0) ? 1u : 0u);
                    }
                    tc::commit(&aempty[abuf]);
                    tc::commit(&empty[slot]);
                }
                if (!ok) break;
                tc::commit(dfull);
            }
            // all MMAs issued have completed before tensor memory is released
            tc::commit(drain);
            g_wait(drain, 0, err);
        }
    } else if (warp < 8) {
        // ---------------------------------------------------- dequant
        // warp w: rows 32 (w % 4) + lane (its tensor-memory lanes), group
        // w / 4 of each 64-wide chunk, written in natural K order
        const int row = 32 * (warp & 3) + lane;
        const int jg = warp >> 2;
        const uint32_t lane_base = tbase + (static_cast<uint32_t>(32 * (warp & 3)) << 16);
        int it = 0;
        bool ok = true;
        for (int u = blockIdx.x; u < tiles && ok; u += gridDim.x) {
            for (int c = 0; c < nch; ++c, ++it) {
                const int slot = it % kGSlots, abuf = it % kGABufs;
                if (!g_wait(&full[slot], (it / kGSlots) & 1, err) ||
                    (it >= kGABufs && !g_wait(&aempty[abuf], ((it / kGABufs) - 1) & 1, err))) {
                    ok = false;
                    break;
                }
                const uint8_t* base = ring + static_cast<size_t>(slot) * kGSlot + kGX;
                const uint8_t* crow = base + row * 32;
                // scale of group 2 (c & 3) + jg of the 8 loaded for this 256-wide block
                const uint32_t sh = *reinterpret_cast<const uint16_t*>(base + kGCodes + row * 16 + 4 * (c & 3) + 2 * jg);
                // (q - 7) s is rounded to fp16 below: a larger scale would overflow
                if ((sh & 0x7FFFu) > kMaxFp16ScaleBits) atomicOr(err, kErrScale);
                {
                    const int j = jg;   // 16-byte chunk of the 32-byte row, 32-byte swizzle
                    const uint4 cw = *reinterpret_cast<const uint4*>(crow + ((j ^ ((row >> 2) & 1)) << 4));
                    const uint32_t s2 = sh | (sh << 16);
                    const uint32_t words[4] = {cw.x, cw.y, cw.z, cw.w};
                    uint32_t q[16];
#pragma unroll
                    for (int w = 0; w < 4; ++w) {
                        uint32_t p[4];   // (k, k+4) pairs of the word
                        unpack_word(words[w], p);
                        q[4 * w + 0] = tc::hmul2_u32(prmt(p[0], p[1], 0x5410u), s2);   // k0 k1
                        q[4 * w + 1] = tc::hmul2_u32(prmt(p[2], p[3], 0x5410u), s2);   // k2 k3
                        q[4 * w + 2] = tc::hmul2_u32(prmt(p[0], p[1], 0x7632u), s2);   // k4 k5
                        q[4 * w + 3] = tc::hmul2_u32(prmt(p[2], p[3], 0x7632u), s2);   // k6 k7
                    }
                    tc::st16(lane_base + 32 * abuf + 16 * j, q);
                }
                tc::st_wait();
                tc::fence_before_sync();
                __syncwarp();
                if (lane == 0) {
                    mbar_arrive(&empty[slot]);
                    mbar_arrive(&afull[abuf]);
                }
            }
        }
    } else {
        // ---------------------------------------------------- epilogue warps
        // warp w reads tensor-memory lanes 32 (w % 4) .. + 31 (weight rows)
        const int quad = warp & 3;
        const int row = 32 * quad + lane;
        const int tid = 32 * quad + lane;   // 0..127 over the four warps
        const uint32_t lane_base = tbase + (static_cast<uint32_t>(32 * quad) << 16);
        int dit = 0;
        for (int u = blockIdx.x; u < tiles; u += gridDim.x, ++dit) {
            const int n0 = (u / a.ttiles) * 128, m0 = (u % a.ttiles) * kGTok;
            if (!g_wait(dfull, dit & 1, err)) break;
            tc::fence_after_sync();
            // accumulator (row, token) -> transpose buffer [token][row], fp16;
            // the accumulator is free for the next tile's MMAs right after
#pragma unroll 4
            for (int h = 0; h < kGTok / 16; ++h) {
                uint32_t d[16];
                tc::ld16(lane_base + kGDCol + 16 * h, d);
                tc::ld_wait();
#pragma unroll
                for (int i = 0; i < 16; ++i)
                    tbuf[(16 * h + i) * 128 + row] = float_to_half_bits(__uint_as_float(d[i]));
            }
            tc::fence_before_sync();
            __syncwarp();
            if (lane == 0) mbar_arrive(dempty);
            named_barrier_sync(3, 128);
            // 256 tokens x 256 bytes out, 16 bytes per store
#pragma unroll 4
            for (int i = 0; i < kGTok / 8; ++i) {
                const int chunk = tid + 128 * i;
                const int tok = chunk >> 4, seg = chunk & 15;
                const int m = m0 + tok, n = n0 + 8 * seg;
                if (m < a.M && n < a.N)
                    *reinterpret_cast<uint4*>(a.y + static_cast<size_t>(m) * a.N + n) =
                        *reinterpret_cast<const uint4*>(tbuf + tok * 128 + 8 * seg);
            }
            named_barrier_sync(3, 128);   // the buffer is free for the next tile
        }
    }

    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    if (warp == kGIssuer) tc::tmem_dealloc(tbase, kGTmemCols);
}

template <int TOK>
int gemm_attr()
{
    static std::once_flag once;
    static int rc = -1;
    std::call_once(once, [] {
        rc = cudaFuncSetAttribute(gemm_kernel<TOK>, cudaFuncAttributeMaxDynamicSharedMemorySize, GCfg<TOK>::kSmem) ==
                     cudaSuccess
                 ? 0
                 : 1;
    });
    return rc;
}

// Token tile: the width whose grid rounds (tiles over the SMs, rounded up)
// times its cost relative to a 256-token tile is least; a 128-token tile
// costs well over half of a 256-token one, a 192-token tile more than 6/7 of
// one (measured: 7 rounds of 192 ran slower than 6 of 256), so 0.6 and 0.9.
// Ties go to the wider tile.  128 when the prompt has at most 128 tokens.
int pick_tok(int N, int M, int sms)
{
    if (M <= 128) return 128;
    const int rt = (N + 127) / 128;
    const int toks[3] = {256, 192, 128};
    const double cost[3] = {1.0, 0.9, 0.6};
    int best = 256;
    double best_c = 1e300;
    for (int i = 0; i < 3; ++i) {
        const int64_t tiles = static_cast<int64_t>(rt) * ((M + toks[i] - 1) / toks[i]);
        const double c = static_cast<double>((tiles + sms - 1) / sms) * cost[i];
        if (c < best_c - 1e-9) {
            best_c = c;
            best = toks[i];
        }
    }
    return best;
}

}  // namespace
}  // namespace wq4

using namespace wq4;

extern "C" int wq4_gemm(const uint32_t* W_packed, const uint16_t* scales, const uint16_t* x, uint16_t* y, int N, int K,
                        int M, void* stream)
{
    if (!W_packed || !scales || !x || !y) return WQ4_ERR_INVALID;
    if (N < 1 || K < 32 || M < 1 || (K % 32) != 0) return WQ4_ERR_INVALID;
    if ((K % 256) != 0 || (N % 8) != 0) return WQ4_ERR_UNSUPPORTED;
    if (static_cast<int64_t>(N) * K / 8 > (static_cast<int64_t>(1) << 40)) return WQ4_ERR_INVALID;
    if (!aligned(W_packed, 16) || !aligned(scales, 16) || !aligned(x, 16) || !aligned(y, 16)) return WQ4_ERR_ALIGN;
    const size_t yb = static_cast<size_t>(M) * N * 2, xb = static_cast<size_t>(M) * K * 2;
    const size_t wb = static_cast<size_t>(N) * K / 2, sb = static_cast<size_t>(N) * K / 16;
    if (overlaps(y, yb, x, xb) || overlaps(y, yb, W_packed, wb) || overlaps(y, yb, scales, sb)) return WQ4_ERR_INVALID;
    int dev = 0;
    const DeviceInfo* di = current_device_info(&dev);
    if (!di) return WQ4_ERR_CUDA;
    const int tok = pick_tok(N, M, di->sm_count);
    if ((tok == 256 ? gemm_attr<256>() : tok == 192 ? gemm_attr<192>() : gemm_attr<128>()) != 0) return WQ4_ERR_CUDA;
    CUtensorMap mc, ms, mx;
    if (!encode_tensor_map_2d(&mc, CU_TENSOR_MAP_DATA_TYPE_UINT8, W_packed, static_cast<uint64_t>(K) / 2,
                              static_cast<uint64_t>(N), static_cast<uint64_t>(K) / 2, 32, 64,
                              CU_TENSOR_MAP_SWIZZLE_32B) ||
        !encode_tensor_map_2d(&ms, CU_TENSOR_MAP_DATA_TYPE_UINT16, scales, static_cast<uint64_t>(K) / 32,
                              static_cast<uint64_t>(N), static_cast<uint64_t>(K) / 16, 8, 64,
                              CU_TENSOR_MAP_SWIZZLE_NONE) ||
        !encode_tensor_map_2d(&mx, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, x, static_cast<uint64_t>(K), static_cast<uint64_t>(M),
                              static_cast<uint64_t>(K) * 2, 64, tok, CU_TENSOR_MAP_SWIZZLE_128B))
        return WQ4_ERR_CUDA;
    GemmArgs a;
    a.y = y;
    a.N = N;
    a.K = K;
    a.M = M;
    a.rtiles = (N + 127) / 128;
    a.ttiles = (M + tok - 1) / tok;
    a.err = status_word();
    if (!a.err) return WQ4_ERR_CUDA;
    const int64_t tiles = static_cast<int64_t>(a.rtiles) * a.ttiles;
    if (tiles > (static_cast<int64_t>(1) << 30)) return WQ4_ERR_UNSUPPORTED;
    const int grid = static_cast<int>(tiles < di->sm_count ? tiles : di->sm_count);
    if (tok == 256)
        gemm_kernel<256><<<grid, kGThreads, GCfg<256>::kSmem, static_cast<cudaStream_t>(stream)>>>(mc, ms, mx, a);
    else if (tok == 192)
        gemm_kernel<192><<<grid, kGThreads, GCfg<192>::kSmem, static_cast<cudaStream_t>(stream)>>>(mc, ms, mx, a);
    else
        gemm_kernel<128><<<grid, kGThreads, GCfg<128>::kSmem, static_cast<cudaStream_t>(stream)>>>(mc, ms, mx, a);
    return cudaGetLastError() == cudaSuccess ? WQ4_OK : WQ4_ERR_CUDA;
}
