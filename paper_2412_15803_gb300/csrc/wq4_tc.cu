// wq4_tc.cu -- batched decode chain on the tensor cores (batch 5-32).
//
// Above batch 4 the per-weight FMA work of the CUDA-core path grows with the
// batch while the weight stream does not; here every projection becomes a
// dequantize + tcgen05 GEMM: y[b][n] = sum_k w[n][k] x[b][k] with
// w = fp16((q - 7) s) (one rounding per weight, at most 2^-11 relative, then
// fp32 accumulation in tensor memory: within the GEMV tolerance of
// Section 3's 4-bit decode), M = 128 weight rows per tile, N = the batch
// padded to 16 or 32, K in chunks of 256.
//
// One stage kernel per projection, persistent over (row tile, K part) units:
//   warp 4 lane 0   TMA producer: packed codes (128 rows x 128 B, 128-byte
//                   swizzle), scales (128 rows x 16 B) and the chunk's input
//                   columns (NB rows x 4 x 64 fp16, 128-byte swizzle) into a
//                   4-slot shared-memory ring;
//   warps 0-3       dequantize their 32 rows (lane = tensor-memory lane) into
//                   one of two 128-column A buffers in tensor memory, then
//                   read the unit's accumulator out as fp32 partial sums;
//   warp 5 lane 0   issues 16 MMAs per chunk (A from tensor memory, B from
//                   shared memory) into one of two accumulators.
// The unpack pairs codes (k, k + 4) of each packed word, so the input is kept
// in a matching permuted order (xp): logical position 8w + l holds element
// 8w + perm[l], perm = 0 4 1 5 2 6 3 7.  The epilogue kernels (one CTA per
// batch row) sum the K parts in order, apply the chain's row factors,
// residual adds and SiLU (same formulas as the persistent kernel), write the
// stage traces, the next stage's permuted input and its RMS factor.
#include "wq4_host.h"
#include "wq4_tc.cuh"
#include "wq4_tc_host.h"

#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cstring>
#include <mutex>
#include <vector>

namespace wq4 {
namespace {

constexpr int kTcStages = 4;          // ring slots
constexpr int kTcThreads = 192;       // warps 0-3 dequant, 4 producer, 5 MMA
constexpr int kTcCodes = 128 * 128;   // one chunk of codes: 128 rows x 256 codes
constexpr int kTcScales = 128 * 16;   // 128 rows x 8 fp16 scales
constexpr int kTcTmemCols = 512;      // A: 2 x 128 columns, D: 2 x 32 columns at 256

template <int NB>
struct TcSmem {
    static constexpr int kX = NB * 512;                       // 4 slabs x NB rows x 128 B
    static constexpr int kSlot = kTcCodes + kX + kTcScales;   // multiple of 1024
    static constexpr int kBytes = 1024 + kTcStages * kSlot;
};

__device__ __forceinline__ bool tc_wait(uint64_t* bar, uint32_t parity, uint32_t* err)
{
    return mbar_wait(bar, parity, err);
}

template <int NB>
__global__ void __launch_bounds__(kTcThreads, 1)
    tc_stage_kernel(const __grid_constant__ CUtensorMap tm_codes, const __grid_constant__ CUtensorMap tm_scales,
                    const __grid_constant__ CUtensorMap tm_x, int N, int K, int B, int P, int units,
                    float* __restrict__ part, uint32_t* err)
{
    using L = TcSmem<NB>;
    extern __shared__ __align__(1024) uint8_t smem[];
    uint64_t* full = reinterpret_cast<uint64_t*>(smem);
    uint64_t* empty = full + kTcStages;
    uint64_t* afull = empty + kTcStages;
    uint64_t* aempty = afull + 2;
    uint64_t* dfull = aempty + 2;
    uint64_t* dempty = dfull + 2;
    uint64_t* drain = dempty + 2;
    uint32_t* tbase_sh = reinterpret_cast<uint32_t*>(smem + 256);
    uint8_t* ring = smem + 1024;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nch = K >> 8;   // chunks of 256 along K

    if (threadIdx.x == 0) {
        for (int i = 0; i < kTcStages; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], 5);   // 4 dequant warps + the MMA commit
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&afull[i], 4);
            mbar_init(&aempty[i], 1);
            mbar_init(&dfull[i], 1);
            mbar_init(&dempty[i], 4);
        }
        mbar_init(drain, 1);
        mbar_fence_init();
    }
    if (warp == 5) tc::tmem_alloc(tbase_sh, kTcTmemCols);
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    const uint32_t tbase = *tbase_sh;

    if (warp == 4) {
        // ---------------------------------------------------- producer
        if (lane == 0) {
            tc::prefetch_map(&tm_codes);
            tc::prefetch_map(&tm_scales);
            tc::prefetch_map(&tm_x);
            int it = 0;
            bool ok = true;
            for (int u = blockIdx.x; u < units && ok; u += gridDim.x) {
                const int tile = u / P, pt = u - tile * P;
                const int c0 = pt * nch / P, c1 = (pt + 1) * nch / P;
                for (int c = c0; c < c1; ++c, ++it) {
                    const int slot = it % kTcStages;
                    if (it >= kTcStages && !tc_wait(&empty[slot], ((it / kTcStages) - 1) & 1, err)) {
                        ok = false;
                        break;
                    }
                    uint8_t* base = ring + static_cast<size_t>(slot) * L::kSlot;
                    mbar_arrive_expect_tx(&full[slot], kTcCodes + L::kX + kTcScales);
                    tc::tma_load_2d(base, &tm_codes, c * 128, tile * 128, &full[slot]);
                    tc::tma_load_2d(base + kTcCodes + L::kX, &tm_scales, c * 8, tile * 128, &full[slot]);
#pragma unroll
                    for (int j = 0; j < 4; ++j)
                        tc::tma_load_2d(base + kTcCodes + j * NB * 128, &tm_x, c * 256 + 64 * j, 0, &full[slot]);
                }
            }
            // every copy issued has landed before the CTA's memory goes away
            const int first = it > kTcStages ? it - kTcStages : 0;
            for (int i = first; i < it; ++i) tc_wait(&full[i % kTcStages], (i / kTcStages) & 1, err);
        }
    } else if (warp == 5) {
        // ---------------------------------------------------- MMA issuer
        if (lane == 0) {
            constexpr uint32_t idesc = tc::idesc_f16_f32(128, NB);
            int it = 0, ait = 0, dit = 0;
            bool ok = true;
            for (int u = blockIdx.x; u < units && ok; u += gridDim.x) {
                const int tile = u / P, pt = u - tile * P;
                const int c0 = pt * nch / P, c1 = (pt + 1) * nch / P;
                const int dbuf = dit & 1;
                if (dit >= 2 && !tc_wait(&dempty[dbuf], ((dit >> 1) - 1) & 1, err)) break;
                const uint32_t dt = tbase + 256 + 32 * dbuf;
                for (int c = c0; c < c1; ++c, ++it, ++ait) {
                    const int slot = it % kTcStages, abuf = ait & 1;
                    if (!tc_wait(&full[slot], (it / kTcStages) & 1, err) || !tc_wait(&afull[abuf], (ait >> 1) & 1, err)) {
                        ok = false;
                        break;
                    }
                    tc::fence_after_sync();
                    const uint32_t xs = smem_addr(ring + static_cast<size_t>(slot) * L::kSlot + kTcCodes);
#pragma unroll
                    for (int s = 0; s < 16; ++s) {
                        const uint64_t bd = tc::sw128_kmajor_desc(xs + (s >> 2) * NB * 128 + 32 * (s & 3));
                        tc::mma_f16_ts(dt, tbase + 128 * abuf + 8 * s, bd, idesc, (c > c0 || s > 0) ? 1u : 0u);
                    }
                    tc::commit(&aempty[abuf]);
                    tc::commit(&empty[slot]);
                }
                if (!ok) break;
                tc::commit(&dfull[dbuf]);
                ++dit;
            }
            // all MMAs issued have completed before tensor memory is released
            tc::commit(drain);
            tc_wait(drain, 0, err);
        }
    } else {
        // ---------------------------------------------------- dequant + readout
        const int row = 32 * warp + lane;            // tile row = tensor-memory lane
        const uint32_t lane_base = tbase + (static_cast<uint32_t>(32 * warp) << 16);
        int it = 0, ait = 0, dit = 0;
        bool ok = true;
        for (int u = blockIdx.x; u < units && ok; u += gridDim.x) {
            const int tile = u / P, pt = u - tile * P;
            const int c0 = pt * nch / P, c1 = (pt + 1) * nch / P;
            for (int c = c0; c < c1; ++c, ++it, ++ait) {
                const int slot = it % kTcStages, abuf = ait & 1;
                if (!tc_wait(&full[slot], (it / kTcStages) & 1, err) ||
                    (ait >= 2 && !tc_wait(&aempty[abuf], ((ait >> 1) - 1) & 1, err))) {
                    ok = false;
                    break;
                }
                const uint8_t* base = ring + static_cast<size_t>(slot) * L::kSlot;
                const uint8_t* crow = base + row * 128;
                const uint4 sv = *reinterpret_cast<const uint4*>(base + kTcCodes + L::kX + row * 16);
                const uint32_t sw[4] = {sv.x, sv.y, sv.z, sv.w};
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    const uint4 cw = *reinterpret_cast<const uint4*>(crow + ((j ^ (row & 7)) << 4));
                    const uint32_t sh = (j & 1) ? (sw[j >> 1] >> 16) : (sw[j >> 1] & 0xFFFFu);
                    const uint32_t s2 = sh | (sh << 16);
                    uint32_t q[16];
                    unpack_word(cw.x, q + 0);
                    unpack_word(cw.y, q + 4);
                    unpack_word(cw.z, q + 8);
                    unpack_word(cw.w, q + 12);
#pragma unroll
                    for (int i = 0; i < 16; ++i) q[i] = tc::hmul2_u32(q[i], s2);
                    tc::st16(lane_base + 128 * abuf + 16 * j, q);
                }
                tc::st_wait();
                tc::fence_before_sync();
                __syncwarp();
                if (lane == 0) {
                    mbar_arrive(&empty[slot]);
                    mbar_arrive(&afull[abuf]);
                }
            }
            if (!ok) break;
            const int dbuf = dit & 1;
            if (!tc_wait(&dfull[dbuf], (dit >> 1) & 1, err)) break;
            tc::fence_after_sync();
            uint32_t d[32];
            tc::ld16(lane_base + 256 + 32 * dbuf, d);
            if (NB > 16) tc::ld16(lane_base + 256 + 32 * dbuf + 16, d + 16);
            tc::ld_wait();
            const int n = tile * 128 + row;
            if (n < N) {
                float* pb = part + static_cast<size_t>(pt) * B * N + n;
#pragma unroll
                for (int b = 0; b < NB; ++b)
                    if (b < B) pb[static_cast<size_t>(b) * N] = __uint_as_float(d[b]);
            }
            tc::fence_before_sync();
            __syncwarp();
            if (lane == 0) mbar_arrive(&dempty[dbuf]);
            ++dit;
        }
    }

    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    if (warp == 5) tc::tmem_dealloc(tbase, kTcTmemCols);
}

// ------------------------------------------------------------ epilogues --

__device__ __forceinline__ int perm8(int l) { return (l & 1) ? (l >> 1) + 4 : (l >> 1); }

// fp16(a + b) for fp16 operands: the fp32 sum rounded once to fp16.
__device__ __forceinline__ uint16_t add_h(float a, float b) { return float_to_half_bits(a + b); }

// Sum of squares of vec[0, n) in a fixed order (same bits on every run).
__device__ float block_sumsq(const uint16_t* vec, int n, float* red)
{
    float s = 0.f;
    for (int k = threadIdx.x; k < n; k += blockDim.x) {
        const float t = half_bits_to_float(vec[k]);
        s = fmaf(t, t, s);
    }
    s = warp_sum(s);
    __syncthreads();
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = s;
    __syncthreads();
    float t = 0.f;
    for (int w = 0; w < static_cast<int>(blockDim.x >> 5); ++w) t += red[w];
    return t;
}

// xp[8w + l] = vec[8w + perm8(l)]
__device__ void write_perm(const uint16_t* vec, int n, uint16_t* xp)
{
    for (int w = threadIdx.x; w < (n >> 3); w += blockDim.x) {
        uint16_t o[8];
#pragma unroll
        for (int l = 0; l < 8; ++l) o[l] = vec[8 * w + perm8(l)];
        uint4 v;
        v.x = o[0] | (static_cast<uint32_t>(o[1]) << 16);
        v.y = o[2] | (static_cast<uint32_t>(o[3]) << 16);
        v.z = o[4] | (static_cast<uint32_t>(o[5]) << 16);
        v.w = o[6] | (static_cast<uint32_t>(o[7]) << 16);
        reinterpret_cast<uint4*>(xp)[w] = v;
    }
}

__device__ __forceinline__ float rms_factor(float sumsq, int n, float eps)
{
    return rsqrtf(sumsq * (1.f / static_cast<float>(n)) + eps);
}

// Token start (one CTA per batch row): r = r(u), v = fp16(r u), xp = perm(u).
__global__ void __launch_bounds__(1024) tc_prologue_kernel(const uint16_t* __restrict__ u, int H, float eps,
                                                           float* __restrict__ r_out, uint16_t* __restrict__ v_out,
                                                           uint16_t* __restrict__ xp)
{
    __shared__ float red[32];
    const int b = blockIdx.x;
    const uint16_t* ub = u + static_cast<size_t>(b) * H;
    const float r = rms_factor(block_sumsq(ub, H, red), H, eps);
    if (threadIdx.x == 0) r_out[b] = r;
    for (int k = threadIdx.x; k < H; k += blockDim.x)
        v_out[static_cast<size_t>(b) * H + k] = float_to_half_bits(r * half_bits_to_float(ub[k]));
    write_perm(ub, H, xp + static_cast<size_t>(b) * H);
}

// One stage's epilogue for batch row b = blockIdx.x; vec (shared memory) holds
// the next stage's input.
__global__ void __launch_bounds__(1024) tc_epilogue_kernel(TcEpi e)
{
    extern __shared__ __align__(16) uint16_t vec[];
    __shared__ float red[32];
    const int b = blockIdx.x, B = e.B, N = e.N, H = e.H, F = e.F;
    auto ysum = [&](int n) {
        float t = 0.f;
        for (int p = 0; p < e.P; ++p) t += e.part[(static_cast<size_t>(p) * B + b) * N + n];
        return t;
    };
    const float r = e.r_in ? e.r_in[b] : 1.f;
    int nvec = 0;
    switch (e.type) {
        case kTcQKV:
            for (int n = threadIdx.x; n < N; n += blockDim.x) {
                const uint16_t q = float_to_half_bits(r * ysum(n));
                e.y[static_cast<size_t>(b) * N + n] = q;
                if (n < H) vec[n] = q;
            }
            nvec = H;
            break;
        case kTcO:
            for (int n = threadIdx.x; n < H; n += blockDim.x) {
                const uint16_t o = float_to_half_bits(r * ysum(n));
                const uint16_t x1 = add_h(half_bits_to_float(e.v_in[static_cast<size_t>(b) * H + n]), half_bits_to_float(o));
                e.y[static_cast<size_t>(b) * H + n] = o;
                e.y2[static_cast<size_t>(b) * H + n] = x1;
                vec[n] = x1;
            }
            nvec = H;
            break;
        case kTcGU:
            for (int j = threadIdx.x; j < F; j += blockDim.x) {
                const uint16_t g = float_to_half_bits(r * ysum(j));
                const uint16_t uu = float_to_half_bits(r * ysum(F + j));
                const float gf = half_bits_to_float(g);
                const uint16_t m = float_to_half_bits(gf / (1.f + expf(-gf)) * half_bits_to_float(uu));
                e.y[static_cast<size_t>(b) * 2 * F + j] = g;
                e.y[static_cast<size_t>(b) * 2 * F + F + j] = uu;
                e.y2[static_cast<size_t>(b) * F + j] = m;
                vec[j] = m;
            }
            nvec = F;
            break;
        case kTcDOWN:
            for (int n = threadIdx.x; n < H; n += blockDim.x) {
                const uint16_t d = float_to_half_bits(ysum(n));
                const uint16_t x2 = add_h(half_bits_to_float(e.v_in[static_cast<size_t>(b) * H + n]), half_bits_to_float(d));
                e.y[static_cast<size_t>(b) * H + n] = d;
                e.y2[static_cast<size_t>(b) * H + n] = x2;
                vec[n] = x2;
            }
            nvec = H;
            break;
        default:   // LM head
            for (int n = threadIdx.x; n < N; n += blockDim.x)
                e.y[static_cast<size_t>(b) * N + n] = float_to_half_bits(r * ysum(n));
            return;
    }
    __syncthreads();
    if (e.r_out) {
        const float rn = rms_factor(block_sumsq(vec, nvec, red), nvec, e.eps);
        if (threadIdx.x == 0) e.r_out[b] = rn;
        if (e.v_out)
            for (int k = threadIdx.x; k < nvec; k += blockDim.x)
                e.v_out[static_cast<size_t>(b) * nvec + k] = float_to_half_bits(rn * half_bits_to_float(vec[k]));
    }
    write_perm(vec, nvec, e.xp + static_cast<size_t>(b) * nvec);
}

// ----------------------------------------------------------------- host --

PFN_cuTensorMapEncodeTiled_v12000 encode_fn()
{
    static std::once_flag once;
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    std::call_once(once, [] {
        cudaDriverEntryPointQueryResult q;
        void* p = nullptr;
        if (cudaGetDriverEntryPoint("cuTensorMapEncodeTiled", &p, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    });
    return fn;
}

bool encode_2d(CUtensorMap* m, CUtensorMapDataType dt, const void* base, uint64_t inner, uint64_t outer,
               uint64_t row_bytes, uint32_t box_inner, uint32_t box_outer, CUtensorMapSwizzle swz)
{
    PFN_cuTensorMapEncodeTiled_v12000 enc = encode_fn();
    if (!enc) return false;
    cuuint64_t dims[2] = {inner, outer};
    cuuint64_t strides[1] = {row_bytes};
    cuuint32_t box[2] = {box_inner, box_outer};
    cuuint32_t es[2] = {1, 1};
    return enc(m, dt, 2, const_cast<void*>(base), dims, strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, swz,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

struct TcMatMaps {
    CUtensorMap codes, scales;
    int N, K;
};

template <int NB>
int set_stage_attr()
{
    static int rc = -1;
    static std::mutex mu;
    std::lock_guard<std::mutex> lock(mu);
    if (rc < 0)
        rc = cudaFuncSetAttribute(tc_stage_kernel<NB>, cudaFuncAttributeMaxDynamicSharedMemorySize, TcSmem<NB>::kBytes) ==
                     cudaSuccess
                 ? 0
                 : 1;
    return rc;
}

}  // namespace

struct TcPlan {
    std::vector<TcMatMaps> mats;   // [4L + 1]
    CUtensorMap xH, xF;
    TcBuffers buf;
    int L, H, F, Nqkv, V, B, NB, sms;
    float eps;
    uint32_t* err;
};

size_t tc_part_floats(int L, int H, int F, int Nqkv, int V, int B, int sms)
{
    (void)L;
    auto pn = [&](int N, int K) {
        const int tiles = (N + 127) / 128, nch = K / 256;
        int P = sms / tiles;
        if (P < 1) P = 1;
        if (P > nch) P = nch;
        return static_cast<size_t>(P) * N;
    };
    size_t m = pn(Nqkv, H);
    m = std::max(m, pn(H, H));
    m = std::max(m, pn(2 * F, H));
    m = std::max(m, pn(H, F));
    m = std::max(m, pn(V, H));
    return m * B;
}

int tc_plan_create(const wq4_layer_table* t, int H, int F, int Nqkv, int V, int B, const TcBuffers& buf, int sms,
                   uint32_t* err, TcPlan** out)
{
    *out = nullptr;
    if (B > 32 || H % 256 || F % 256 || !encode_fn()) return WQ4_ERR_UNSUPPORTED;
    TcPlan* p = new TcPlan();
    p->L = t->num_layers;
    p->H = H;
    p->F = F;
    p->Nqkv = Nqkv;
    p->V = V;
    p->B = B;
    p->NB = B > 16 ? 32 : 16;
    p->sms = sms;
    p->eps = t->rms_eps;
    p->buf = buf;
    p->err = err;
    auto add = [&](const wq4_mat& m, int N, int K) {
        TcMatMaps mm;
        mm.N = N;
        mm.K = K;
        const bool ok = encode_2d(&mm.codes, CU_TENSOR_MAP_DATA_TYPE_UINT8, m.W, K / 2, N, K / 2, 128, 128,
                                  CU_TENSOR_MAP_SWIZZLE_128B) &&
                        encode_2d(&mm.scales, CU_TENSOR_MAP_DATA_TYPE_UINT16, m.s, K / 32, N, K / 16, 8, 128,
                                  CU_TENSOR_MAP_SWIZZLE_NONE);
        p->mats.push_back(mm);
        return ok;
    };
    bool ok = true;
    for (int l = 0; l < p->L && ok; ++l) {
        const wq4_layer& ly = t->layers[l];
        ok = add(ly.qkv, Nqkv, H) && add(ly.o, H, H) && add(ly.gate_up, 2 * F, H) && add(ly.down, H, F);
    }
    ok = ok && add(t->lm_head, V, H);
    ok = ok && encode_2d(&p->xH, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, buf.xpH, H, p->NB, static_cast<uint64_t>(H) * 2, 64,
                         p->NB, CU_TENSOR_MAP_SWIZZLE_128B);
    ok = ok && encode_2d(&p->xF, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, buf.xpF, F, p->NB, static_cast<uint64_t>(F) * 2, 64,
                         p->NB, CU_TENSOR_MAP_SWIZZLE_128B);
    ok = ok && set_stage_attr<16>() == 0 && set_stage_attr<32>() == 0;
    if (!ok) {
        delete p;
        return WQ4_ERR_CUDA;
    }
    *out = p;
    return WQ4_OK;
}

void tc_plan_destroy(TcPlan* p) { delete p; }

// Records one token on `cs` (inside a stream capture).
void tc_record_token(const TcPlan* p, cudaStream_t cs)
{
    const int B = p->B, H = p->H, F = p->F, L = p->L;
    const TcBuffers& u = p->buf;
    const size_t LH = static_cast<size_t>(B) * H;
    auto stage = [&](const TcMatMaps& m, const CUtensorMap& xmap) {
        const int tiles = (m.N + 127) / 128, nch = m.K / 256;
        int P = p->sms / tiles;
        if (P < 1) P = 1;
        if (P > nch) P = nch;
        const int units = tiles * P;
        const int grid = units < p->sms ? units : p->sms;
        if (p->NB == 16)
            tc_stage_kernel<16><<<grid, kTcThreads, TcSmem<16>::kBytes, cs>>>(m.codes, m.scales, xmap, m.N, m.K, B, P,
                                                                             units, u.part, p->err);
        else
            tc_stage_kernel<32><<<grid, kTcThreads, TcSmem<32>::kBytes, cs>>>(m.codes, m.scales, xmap, m.N, m.K, B, P,
                                                                             units, u.part, p->err);
        return P;
    };
    auto epi = [&](TcEpi e, int nvec_max) {
        e.B = B;
        e.H = H;
        e.F = F;
        e.eps = p->eps;
        e.part = u.part;
        tc_epilogue_kernel<<<B, 1024, 2 * nvec_max, cs>>>(e);
    };
    float* rf = u.rf;   // [L + 1][3][B]
    tc_prologue_kernel<<<B, 1024, 0, cs>>>(u.x_stage, H, p->eps, rf, u.pV, u.xpH);
    for (int l = 0; l < L; ++l) {
        float* r = rf + static_cast<size_t>(3 * l) * B;
        const TcMatMaps* m = &p->mats[4 * static_cast<size_t>(l)];
        TcEpi e{};
        e.type = kTcQKV;
        e.N = p->Nqkv;
        e.P = stage(m[0], p->xH);
        e.r_in = r;
        e.y = u.pQKV + static_cast<size_t>(l) * B * p->Nqkv;
        e.r_out = r + B;
        e.xp = u.xpH;
        epi(e, H);

        e = TcEpi{};
        e.type = kTcO;
        e.N = H;
        e.P = stage(m[1], p->xH);
        e.r_in = r + B;
        e.v_in = u.pV + static_cast<size_t>(l) * LH;
        e.y = u.pO + static_cast<size_t>(l) * LH;
        e.y2 = u.pX1 + static_cast<size_t>(l) * LH;
        e.r_out = r + 2 * B;
        e.xp = u.xpH;
        epi(e, H);

        e = TcEpi{};
        e.type = kTcGU;
        e.N = 2 * F;
        e.P = stage(m[2], p->xH);
        e.r_in = r + 2 * B;
        e.y = u.pGU + static_cast<size_t>(l) * B * 2 * F;
        e.y2 = u.pM + static_cast<size_t>(l) * B * F;
        e.xp = u.xpF;
        epi(e, F);

        e = TcEpi{};
        e.type = kTcDOWN;
        e.N = H;
        e.P = stage(m[3], p->xF);
        e.v_in = u.pX1 + static_cast<size_t>(l) * LH;
        e.y = u.pD + static_cast<size_t>(l) * LH;
        e.y2 = u.pX2 + static_cast<size_t>(l) * LH;
        e.r_out = r + 3 * B;                                   // next layer's (or the LM head's) factor
        e.v_out = u.pV + static_cast<size_t>(l + 1) * LH;
        e.xp = u.xpH;
        epi(e, H);
    }
    TcEpi e{};
    e.type = kTcLM;
    e.N = p->V;
    e.P = stage(p->mats[4 * static_cast<size_t>(L)], p->xH);
    e.r_in = rf + static_cast<size_t>(3 * L) * B;
    e.y = u.logits;
    epi(e, 0);
}

}  // namespace wq4
