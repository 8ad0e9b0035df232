// wq4_tc.cu -- batched decode chain on the tensor cores (batch 3-32).
//
// Above batch 2 the per-weight FMA work of the CUDA-core path grows with the
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
constexpr int kTcThreads = 480;       // warps 0-7 dequant, 8 producer, 9 and 14 MMA, 10-13 epilogue
constexpr int kTcProducer = 8, kTcIssuer = 9, kTcIssuer2 = 14;
constexpr int kTcCodes = 128 * 128;   // one chunk of codes: 128 rows x 256 codes
constexpr int kTcScales = 128 * 16;   // 128 rows x 8 fp16 scales
constexpr int kTcMaxParts = 8;        // K parts of a split stage (bounds the epilogue's loads in flight)
constexpr int kTcABufs = 3;           // dequantized A buffers (128 columns each)
constexpr int kTcDCol = 128 * kTcABufs;  // accumulators: 2 buffers x 2 issuers x 32 columns
constexpr int kTcTmemCols = 512;

template <int NB>
struct TcSmem {
    static_assert(256 + 4 * (192 + 128 * 33) <= 18432, "epilogue scratch overlaps the ring");
    static constexpr int kX = NB * 512;                       // 4 slabs x NB rows x 128 B
    static constexpr int kSlot = kTcCodes + kX + kTcScales;   // multiple of 1024
    static constexpr int kRing = 18432;                        // header + epilogue scratch, then the ring
    static constexpr int kBytes = kRing + kTcStages * kSlot;
};

__device__ __forceinline__ bool tc_wait_ok(uint64_t* bar, uint32_t parity, uint32_t* err)
{
    return mbar_wait(bar, parity, err);
}

// Kernel arguments besides the tensor maps.  A stage's "tile" is 128 weight
// rows: rows [128 t, 128 t + 128), or for gate_up gate rows [64 t, 64 t + 64)
// followed by the matching up rows [F + 64 t, F + 64 t + 64), so that one tile
// holds both halves of SiLU(gate) * up.
struct TcArgs {
    int type, N, K, B, P, units, tiles, H, F;
    float eps;
    float* part;            // [P][B][N] partial sums (P > 1)
    uint32_t* cnt;          // [tiles] arrival counters (P > 1), zero between stages
    const float* sq_in;     // per-tile sums of squares of this stage's input [H/128][B]; null: factor 1
    const float* sq_u;      // O: sums of squares of the layer input u
    const uint16_t* res;    // O: the layer input u; down: x1
    uint16_t* y;            // QKV: qkv, O: o, gate_up: gate|up, down: d, LM: logits
    uint16_t* y2;           // O: x1, gate_up: m, down: x2
    uint16_t* y3;           // O: v = fp16(r(u) u)
    float* sq_out;          // per-tile sums of squares of the next stage's input [H/128][B]
    uint16_t* xp;           // next stage's permuted input [32][ldxp]
    int ldxp;
    uint32_t* err;
};

__device__ __forceinline__ void grid_dep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void grid_dep_launch() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// fp16(a + b) for fp16 operands: the fp32 sum rounded once to fp16.
__device__ __forceinline__ uint16_t add_h(float a, float b) { return float_to_half_bits(a + b); }

// Logical position, within its 8-block, of element p (0..7) of a packed
// word: the unpack pairs (p, p + 4), so logical order is 0 4 1 5 2 6 3 7.
__device__ __forceinline__ int perm_pos(int p) { return p < 4 ? 2 * p : 2 * (p - 4) + 1; }

// r = 1/sqrt(mean + eps) from per-tile sums of squares, summed in tile order
// (up to 32 loads issued at once, then the rest).
__device__ __forceinline__ float rms_of(const float* sq, int ntiles, int B, int b, int n, float eps)
{
    float v[32];
#pragma unroll
    for (int k = 0; k < 32; ++k) v[k] = k < ntiles ? __ldcg(sq + k * B + b) : 0.f;
    float t = 0.f;
#pragma unroll
    for (int k = 0; k < 32; ++k)
        if (k < ntiles) t += v[k];
    for (int i = 32; i < ntiles; ++i) t += __ldcg(sq + i * B + b);
    return rsqrtf(t * (1.f / static_cast<float>(n)) + eps);
}

// Epilogue of one tile by the 128 epilogue threads (row = 32 quad + lane):
// v[b] the row's sums over K for batch row b, resv the row's residual
// inputs (O, down, LM head) as fp16 pairs, already loaded when NB is 16.  ep: shared scratch whose first
// 64 floats hold the RMS factors r_in[b] and r_u[b] of the stage.
template <int NB>
__device__ void tile_epilogue(const TcArgs& a, int tile, int row, const float v[NB], const uint32_t resv[NB / 2],
                              float* ep)
{
    const int n_row = 128 * tile + row;
    auto res_b = [&](int b) {
        return NB == 16 ? half_bits_to_float(static_cast<uint16_t>(resv[b >> 1] >> (16 * (b & 1))))
                        : half_bits_to_float(a.res[static_cast<size_t>(b) * a.H + n_row]);
    };
    const float* r_in = ep;    // [32]
    const float* r_u = ep + 32;
    float* red = ep + 64;      // [4][32]
    float* sqs = ep + 192;     // [128][33] squares of the next input (padded rows), ends before the ring
    uint16_t* upart = reinterpret_cast<uint16_t*>(ep + 192);   // [64][32] up values of gate_up (aliases sqs)
    const int B = a.B, H = a.H, F = a.F;
    float nxt[NB];              // value of the next stage's input at this row (if any)
    bool has_next = false;
    int nidx = 0;               // its index in the next input
    if (a.type == kTcGU) {
        const bool up = row >= 64;
        const int j = 64 * tile + (row & 63);
        if (up) {
#pragma unroll
            for (int b = 0; b < NB; ++b)
                if (b < B) {
                    const uint16_t uu = float_to_half_bits(r_in[b] * v[b]);
                    a.y[static_cast<size_t>(b) * 2 * F + F + j] = uu;
                    upart[(row - 64) * 32 + b] = uu;
                }
        }
        named_barrier_sync(3, 128);
        if (!up) {
#pragma unroll
            for (int b = 0; b < NB; ++b)
                if (b < B) {
                    const uint16_t g = float_to_half_bits(r_in[b] * v[b]);
                    const float gf = half_bits_to_float(g);
                    const uint16_t m =
                        float_to_half_bits(gf / (1.f + expf(-gf)) * half_bits_to_float(upart[row * 32 + b]));
                    a.y[static_cast<size_t>(b) * 2 * F + j] = g;
                    a.y2[static_cast<size_t>(b) * F + j] = m;
                    a.xp[static_cast<size_t>(b) * a.ldxp + (j & ~7) + perm_pos(j & 7)] = m;
                }
        }
        return;
    }
    const int n = 128 * tile + row;
    if (n < a.N) {
        switch (a.type) {
            case kTcQKV:
#pragma unroll
                for (int b = 0; b < NB; ++b)
                    if (b < B) {
                        const uint16_t q = float_to_half_bits(r_in[b] * v[b]);
                        a.y[static_cast<size_t>(b) * a.N + n] = q;
                        nxt[b] = half_bits_to_float(q);
                    }
                has_next = n < H;
                nidx = n;
                break;
            case kTcO:
#pragma unroll
                for (int b = 0; b < NB; ++b)
                    if (b < B) {
                        const uint16_t o = float_to_half_bits(r_in[b] * v[b]);
                        const uint16_t vn = float_to_half_bits(r_u[b] * res_b(b));
                        const uint16_t x1 = add_h(half_bits_to_float(vn), half_bits_to_float(o));
                        a.y[static_cast<size_t>(b) * H + n] = o;
                        a.y2[static_cast<size_t>(b) * H + n] = x1;
                        a.y3[static_cast<size_t>(b) * H + n] = vn;
                        nxt[b] = half_bits_to_float(x1);
                    }
                has_next = true;
                nidx = n;
                break;
            case kTcDOWN:
#pragma unroll
                for (int b = 0; b < NB; ++b)
                    if (b < B) {
                        const uint16_t d = float_to_half_bits(v[b]);
                        const uint16_t x2 = add_h(res_b(b), half_bits_to_float(d));
                        a.y[static_cast<size_t>(b) * H + n] = d;
                        a.y2[static_cast<size_t>(b) * H + n] = x2;
                        nxt[b] = half_bits_to_float(x2);
                    }
                has_next = true;
                nidx = n;
                break;
            default:   // LM head; its first H / 128 tiles also keep v = fp16(r x_L)
#pragma unroll
                for (int b = 0; b < NB; ++b)
                    if (b < B) {
                        a.y[static_cast<size_t>(b) * a.N + n] = float_to_half_bits(r_in[b] * v[b]);
                        if (n < H)
                            a.y3[static_cast<size_t>(b) * H + n] =
                                float_to_half_bits(r_in[b] * res_b(b));
                    }
                break;
        }
    }
    if (a.type == kTcLM) return;
    // the next stage's permuted input and, per tile of its rows, its sum of squares
    if (has_next) {
#pragma unroll
        for (int b = 0; b < NB; ++b)
            if (b < B) a.xp[static_cast<size_t>(b) * a.ldxp + (nidx & ~7) + perm_pos(nidx & 7)] = float_to_half_bits(nxt[b]);
    }
    if (tile < H / 128) {
        // sum over the tile's 128 rows per batch row, in a fixed order:
        // 32-row runs, then the four runs
#pragma unroll
        for (int b = 0; b < NB; ++b)
            if (b < B) sqs[row * 33 + b] = has_next ? nxt[b] * nxt[b] : 0.f;
        named_barrier_sync(3, 128);
        {
            const int b = row & 31, run = row >> 5;
            float t = 0.f;
            if (b < B)
                for (int k = 0; k < 32; ++k) t += sqs[(32 * run + k) * 33 + b];
            red[run * 32 + b] = t;
        }
        named_barrier_sync(3, 128);
        if (row < B) a.sq_out[tile * B + row] = ((red[row] + red[32 + row]) + red[64 + row]) + red[96 + row];
    }
}

template <int NB>
__global__ void __launch_bounds__(kTcThreads, 1)
    tc_stage_kernel(const __grid_constant__ CUtensorMap tm_codes, const __grid_constant__ CUtensorMap tm_scales,
                    const __grid_constant__ CUtensorMap tm_x, const TcArgs a)
{
    using L = TcSmem<NB>;
    extern __shared__ __align__(1024) uint8_t smem[];
    uint64_t* fullw = reinterpret_cast<uint64_t*>(smem);   // codes + scales landed
    uint64_t* fullx = fullw + kTcStages;                     // input columns landed
    uint64_t* empty = fullx + kTcStages;
    uint64_t* afull = empty + kTcStages;
    uint64_t* aempty = afull + kTcABufs;
    uint64_t* dfull = aempty + kTcABufs;
    uint64_t* dempty = dfull + 2;
    uint64_t* drain = dempty + 2;
    static_assert((3 * kTcStages + 2 * kTcABufs + 5) * 8 <= 240, "barriers overlap the tensor-memory base word");
    static_assert(kTcDCol + 128 <= kTcTmemCols, "tensor memory overflow");
    uint32_t* tbase_sh = reinterpret_cast<uint32_t*>(smem + 240);
    uint32_t* last_sh = tbase_sh + 1;
    float* ep = reinterpret_cast<float*>(smem + 256);        // epilogue scratch: 768 B + 128 x 33 floats
    uint8_t* ring = smem + L::kRing;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nch = a.K >> 8;   // chunks of 256 along K
    const int P = a.P, units = a.units;
    uint32_t* err = a.err;

    if (threadIdx.x == 0) {
        for (int i = 0; i < kTcStages; ++i) {
            mbar_init(&fullw[i], 1);
            mbar_init(&fullx[i], 1);
            mbar_init(&empty[i], 9);   // 8 dequant warps + the MMA commit
        }
        for (int i = 0; i < kTcABufs; ++i) {
            mbar_init(&afull[i], 8);
            mbar_init(&aempty[i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&dfull[i], 2);   // one commit per issuer
            mbar_init(&dempty[i], 4);
        }
        mbar_init(drain, 2);
        mbar_fence_init();
    }
    if (warp == kTcIssuer) tc::tmem_alloc(tbase_sh, kTcTmemCols);
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    const uint32_t tbase = *tbase_sh;
    // the next stage may start its set-up and weight stream now; it reads our
    // outputs only after this grid has completed
    grid_dep_launch();

    auto tile_rows = [&](int tile, int half) {   // first weight row of a 64-row half tile
        return a.type == kTcGU ? (half ? a.F : 0) + 64 * tile : 128 * tile + 64 * half;
    };

    if (warp == kTcProducer) {
        // ---------------------------------------------------- producer
        if (lane == 0) {
            tc::prefetch_map(&tm_codes);
            tc::prefetch_map(&tm_scales);
            tc::prefetch_map(&tm_x);
            int it = 0;
            bool ok = true, waited = false;
            int pend_c[kTcStages];   // chunks whose input columns wait for the previous stage
            int npend = 0;
            for (int u = blockIdx.x; u < units && ok; u += gridDim.x) {
                const int tile = u / P, pt = u - tile * P;
                const int c0 = pt * nch / P, c1 = (pt + 1) * nch / P;
                for (int c = c0; c < c1; ++c, ++it) {
                    const int slot = it % kTcStages;
                    if (it >= kTcStages) {
                        if (!waited) {
                            grid_dep_wait();
                            waited = true;
                            for (int i = 0; i < npend; ++i) {
                                uint8_t* pb = ring + static_cast<size_t>(i) * L::kSlot;
                                mbar_arrive_expect_tx(&fullx[i], L::kX);
#pragma unroll
                                for (int j = 0; j < 4; ++j)
                                    tc::tma_load_2d(pb + kTcCodes + j * NB * 128, &tm_x, pend_c[i] * 256 + 64 * j, 0, &fullx[i]);
                            }
                        }
                        if (!tc_wait_ok(&empty[slot], ((it / kTcStages) - 1) & 1, err)) {
                            ok = false;
                            break;
                        }
                    }
                    uint8_t* base = ring + static_cast<size_t>(slot) * L::kSlot;
                    mbar_arrive_expect_tx(&fullw[slot], kTcCodes + kTcScales);
                    tc::tma_load_2d(base, &tm_codes, c * 128, tile_rows(tile, 0), &fullw[slot]);
                    tc::tma_load_2d(base + 64 * 128, &tm_codes, c * 128, tile_rows(tile, 1), &fullw[slot]);
                    tc::tma_load_2d(base + kTcCodes + L::kX, &tm_scales, c * 8, tile_rows(tile, 0), &fullw[slot]);
                    tc::tma_load_2d(base + kTcCodes + L::kX + 64 * 16, &tm_scales, c * 8, tile_rows(tile, 1), &fullw[slot]);
                    if (waited) {
                        mbar_arrive_expect_tx(&fullx[slot], L::kX);
#pragma unroll
                        for (int j = 0; j < 4; ++j)
                            tc::tma_load_2d(base + kTcCodes + j * NB * 128, &tm_x, c * 256 + 64 * j, 0, &fullx[slot]);
                    } else {
                        pend_c[npend++] = c;
                    }
                }
            }
            if (!waited) {
                grid_dep_wait();
                for (int i = 0; i < npend; ++i) {
                    uint8_t* pb = ring + static_cast<size_t>(i) * L::kSlot;
                    mbar_arrive_expect_tx(&fullx[i], L::kX);
#pragma unroll
                    for (int j = 0; j < 4; ++j)
                        tc::tma_load_2d(pb + kTcCodes + j * NB * 128, &tm_x, pend_c[i] * 256 + 64 * j, 0, &fullx[i]);
                }
            }
            // every copy issued has landed before the CTA's memory goes away
            const int first = it > kTcStages ? it - kTcStages : 0;
            for (int i = first; i < it; ++i) {
                tc_wait_ok(&fullw[i % kTcStages], (i / kTcStages) & 1, err);
                tc_wait_ok(&fullx[i % kTcStages], (i / kTcStages) & 1, err);
            }
        }
    } else if (warp == kTcIssuer || warp == kTcIssuer2) {
        // ---------------------------------------------------- MMA issuers
        // Two issuing warps: chunk ait goes to issuer ait & 1 (own
        // accumulator) from A buffer ait % 3.  One thread issues a
        // tcgen05.mma only every ~45 cycles at these shapes, so a second
        // issuer doubles the rate; the epilogue adds the two accumulators.
        // The third A buffer lets the dequant warps run a chunk ahead.
        const int iss = warp == kTcIssuer ? 0 : 1;
        if (lane == 0) {
            constexpr uint32_t idesc = tc::idesc_f16_f32(128, NB);
            int it = 0, ait = 0, dit = 0;
            bool ok = true;
            for (int u = blockIdx.x; u < units && ok; u += gridDim.x) {
                const int tile = u / P, pt = u - tile * P;
                const int c0 = pt * nch / P, c1 = (pt + 1) * nch / P;
                (void)tile;
                const int dbuf = dit & 1;
                if (dit >= 2 && !tc_wait_ok(&dempty[dbuf], ((dit >> 1) - 1) & 1, err)) break;
                const uint32_t dt = tbase + kTcDCol + 64 * dbuf + 32 * iss;
                bool first = true;
                for (int c = c0; c < c1; ++c, ++it, ++ait) {
                    if ((ait & 1) != iss) continue;          // the other issuer's chunk
                    const int slot = it % kTcStages, abuf = ait % kTcABufs;
                    if (!tc_wait_ok(&fullx[slot], (it / kTcStages) & 1, err) ||
                        !tc_wait_ok(&afull[abuf], (ait / kTcABufs) & 1, err)) {
                        ok = false;
                        break;
                    }
                    tc::fence_after_sync();
                    const uint32_t xs = smem_addr(ring + static_cast<size_t>(slot) * L::kSlot + kTcCodes);
#pragma unroll
                    for (int s = 0; s < 16; ++s) {
                        const uint64_t bd = tc::sw128_kmajor_desc(xs + (s >> 2) * NB * 128 + 32 * (s & 3));
                        tc::mma_f16_ts(dt, tbase + 128 * abuf + 8 * s, bd, idesc, (!first || s > 0) ? 1u : 0u);
                    }
                    first = false;
                    tc::commit(&aempty[abuf]);
                    tc::commit(&empty[slot]);
                }
                if (!ok) break;
                tc::commit(&dfull[dbuf]);   // arrives at once if this issuer had no chunk here
                ++dit;
            }
            // all MMAs issued have completed before tensor memory is released
            tc::commit(drain);
            tc_wait_ok(drain, 0, err);
        }
    } else if (warp < 8) {
        // ---------------------------------------------------- dequant
        // warp w: rows 32 (w % 4) + lane (its tensor-memory lanes), groups
        // 4 (w / 4) .. + 3 of each chunk
        const int row = 32 * (warp & 3) + lane;
        const int jg = 4 * (warp >> 2);
        const uint32_t lane_base = tbase + (static_cast<uint32_t>(32 * (warp & 3)) << 16);
        int it = 0, ait = 0;
        bool ok = true;
        for (int u = blockIdx.x; u < units && ok; u += gridDim.x) {
            const int tile = u / P, pt = u - tile * P;
            const int c0 = pt * nch / P, c1 = (pt + 1) * nch / P;
            for (int c = c0; c < c1; ++c, ++it, ++ait) {
                const int slot = it % kTcStages, abuf = ait % kTcABufs;
                if (!tc_wait_ok(&fullw[slot], (it / kTcStages) & 1, err) ||
                    (ait >= kTcABufs && !tc_wait_ok(&aempty[abuf], ((ait / kTcABufs) - 1) & 1, err))) {
                    ok = false;
                    break;
                }
                const uint8_t* base = ring + static_cast<size_t>(slot) * L::kSlot;
                const uint8_t* crow = base + row * 128;
                const uint2 sv = *reinterpret_cast<const uint2*>(base + kTcCodes + L::kX + row * 16 + 2 * jg);
                const uint32_t sw[2] = {sv.x, sv.y};
#pragma unroll
                for (int jj = 0; jj < 4; ++jj) {
                    const int j = jg + jj;
                    const uint4 cw = *reinterpret_cast<const uint4*>(crow + ((j ^ (row & 7)) << 4));
                    const uint32_t sh = (jj & 1) ? (sw[jj >> 1] >> 16) : (sw[jj >> 1] & 0xFFFFu);
                    const uint32_t s2 = sh | (sh << 16);
                    // (q - 7) s is rounded to fp16 here: a larger scale would overflow
                    if ((sh & 0x7FFFu) > kMaxFp16ScaleBits) atomicOr(err, kErrScale);
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
        }
    } else {
        // ---------------------------------------------------- epilogue warps
        // warp w reads tensor-memory lanes 32 (w % 4) .. + 31
        const int quad = warp & 3;
        const int row = 32 * quad + lane;
        const uint32_t lane_base = tbase + (static_cast<uint32_t>(32 * quad) << 16);
        int dit = 0, ait = 0;
        // the previous stage's outputs are complete and visible from here on;
        // the stage's RMS factors are computed while the MMAs run
        grid_dep_wait();
        if (quad == 0 && lane < a.B)
            ep[lane] = a.sq_in ? rms_of(a.sq_in, a.H / 128, a.B, lane, a.H, a.eps) : 1.f;
        if (quad == 1 && lane < a.B && a.sq_u) ep[32 + lane] = rms_of(a.sq_u, a.H / 128, a.B, lane, a.H, a.eps);
        named_barrier_sync(3, 128);
        for (int u = blockIdx.x; u < units; u += gridDim.x) {
            const int tile = u / P, pt = u - tile * P;
            const int dbuf = dit & 1;
            // this row's residual input, loaded before the accumulator is ready
            uint32_t resv[NB / 2];   // fp16 pairs: batch rows 2i (low half), 2i + 1
            {
                const int n = 128 * tile + row;
                // (batch > 16: loaded in the epilogue instead, registers are short)
                const bool need = NB == 16 && a.res && a.type != kTcGU && n < a.N && (a.type != kTcLM || n < a.H);
#pragma unroll
                for (int i = 0; i < NB / 2; ++i) {
                    const uint32_t lo = (need && 2 * i < a.B) ? __ldcg(a.res + static_cast<size_t>(2 * i) * a.H + n) : 0u;
                    const uint32_t hi = (need && 2 * i + 1 < a.B) ? __ldcg(a.res + static_cast<size_t>(2 * i + 1) * a.H + n) : 0u;
                    resv[i] = lo | (hi << 16);
                }
            }
            // which issuers accumulated this unit: both unless it has one chunk
            const int nchk = (pt + 1) * nch / P - pt * nch / P;
            const bool has0 = nchk >= 2 || (ait & 1) == 0, has1 = nchk >= 2 || (ait & 1) == 1;
            ait += nchk;
            if (!tc_wait_ok(&dfull[dbuf], (dit >> 1) & 1, err)) break;
            tc::fence_after_sync();
            // the two issuers' accumulators, 16 columns at a time, added in issuer order
            float v[NB];
#pragma unroll
            for (int h = 0; h < NB / 16; ++h) {
                uint32_t d[16], d1[16];
                tc::ld16(lane_base + kTcDCol + 64 * dbuf + 16 * h, d);
                tc::ld16(lane_base + kTcDCol + 64 * dbuf + 32 + 16 * h, d1);
                tc::ld_wait();
#pragma unroll
                for (int b = 0; b < 16; ++b)
                    v[16 * h + b] = (has0 ? __uint_as_float(d[b]) : 0.f) + (has1 ? __uint_as_float(d1[b]) : 0.f);
            }
            tc::fence_before_sync();
            __syncwarp();
            if (lane == 0) mbar_arrive(&dempty[dbuf]);
            ++dit;
            if (P > 1) {
                // K is split over units: publish this part; the last part of
                // the tile sums all parts in order and runs the epilogue
                const int nrow = a.type == kTcGU ? tile_rows(tile, row >> 6) + (row & 63) : 128 * tile + row;
                const bool valid = nrow < a.N;
                // parts are rows of NB floats: [part][row][NB]
                if (valid) {
                    float4* pb = reinterpret_cast<float4*>(a.part + (static_cast<size_t>(pt) * a.N + nrow) * NB);
#pragma unroll
                    for (int c = 0; c < NB / 4; ++c)
                        if (4 * c < a.B) pb[c] = make_float4(v[4 * c], v[4 * c + 1], v[4 * c + 2], v[4 * c + 3]);
                }
                __threadfence();
                named_barrier_sync(3, 128);
                if (row == 0) {
                    const uint32_t prev = atomicAdd(&a.cnt[tile], 1u);
                    *last_sh = (prev == static_cast<uint32_t>(P - 1)) ? 1u : 0u;
                    if (prev == static_cast<uint32_t>(P - 1)) a.cnt[tile] = 0u;   // ready for the next stage
                }
                named_barrier_sync(3, 128);
                if (*last_sh == 0u) continue;
                __threadfence();
                if (valid) {
                    // every part, this unit's included, from L2, summed in part
                    // order; all parts of four batch rows are loaded at once
#pragma unroll
                    for (int c = 0; c < NB / 4; ++c) {
                        if (4 * c < a.B) {
                            float4 t[kTcMaxParts];
#pragma unroll
                            for (int q = 0; q < kTcMaxParts; ++q)
                                if (q < P)
                                    t[q] = __ldcg(reinterpret_cast<const float4*>(a.part + (static_cast<size_t>(q) * a.N + nrow) * NB) + c);
                            float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
#pragma unroll
                            for (int q = 0; q < kTcMaxParts; ++q)
                                if (q < P) {
                                    s0 += t[q].x;
                                    s1 += t[q].y;
                                    s2 += t[q].z;
                                    s3 += t[q].w;
                                }
                            v[4 * c] = s0;
                            v[4 * c + 1] = s1;
                            v[4 * c + 2] = s2;
                            v[4 * c + 3] = s3;
                        }
                    }
                }
            }
            tile_epilogue<NB>(a, tile, row, v, resv, ep);
            named_barrier_sync(3, 128);   // scratch reuse across units
        }
    }

    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    if (warp == kTcIssuer) tc::tmem_dealloc(tbase, kTcTmemCols);
}

// Token start (one CTA per batch row b): the permuted token input and the sums
// of squares of its 128-element tiles.
__global__ void __launch_bounds__(128) tc_prologue_kernel(const uint16_t* __restrict__ x, int H, int B,
                                                          float* __restrict__ sq_out, uint16_t* __restrict__ xp)
{
    __shared__ float red[4];
    grid_dep_wait();
    grid_dep_launch();
    const int b = blockIdx.x;
    const uint16_t* xb = x + static_cast<size_t>(b) * H;
    for (int t = 0; t < H / 128; ++t) {
        const int n = 128 * t + threadIdx.x;
        const uint16_t val = xb[n];
        xp[static_cast<size_t>(b) * H + (n & ~7) + perm_pos(n & 7)] = val;
        const float f = half_bits_to_float(val);
        const float s = warp_sum(f * f);
        if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = s;
        __syncthreads();
        if (threadIdx.x == 0) sq_out[t * B + b] = ((red[0] + red[1]) + red[2]) + red[3];
        __syncthreads();
    }
}

// ----------------------------------------------------------------- host --

bool encode_2d(CUtensorMap* m, CUtensorMapDataType dt, const void* base, uint64_t inner, uint64_t outer,
               uint64_t row_bytes, uint32_t box_inner, uint32_t box_outer, CUtensorMapSwizzle swz)
{
    return encode_tensor_map_2d(m, dt, base, inner, outer, row_bytes, box_inner, box_outer, swz);
}

struct TcMatMaps {
    CUtensorMap codes, scales;   // boxes of 64 rows
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

// K parts of a stage: enough units to fill the GPU, each at least one chunk.
int stage_parts(int tiles, int nch, int sms)
{
    int P = sms / tiles;
    if (P < 1) P = 1;
    if (P > nch) P = nch;
    if (P > kTcMaxParts) P = kTcMaxParts;
    return P;
}

}  // namespace

static PFN_cuTensorMapEncodeTiled_v12000 encode_fn()
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

bool encode_tensor_map_2d(CUtensorMap* m, CUtensorMapDataType dt, const void* base, uint64_t inner, uint64_t outer,
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

struct TcPlan {
    std::vector<TcMatMaps> mats;   // [4L + 1]
    CUtensorMap xH[2], xF;
    TcBuffers buf;
    int L, H, F, Nqkv, V, B, NB, sms;
    float eps;
    uint32_t* err;
};

size_t tc_part_floats(int L, int H, int F, int Nqkv, int V, int B, int sms)
{
    (void)L;
    auto pn = [&](int N, int K, int tiles) {
        const int P = stage_parts(tiles, K / 256, sms);
        return P > 1 ? static_cast<size_t>(P) * N : 0;
    };
    size_t m = pn(Nqkv, H, (Nqkv + 127) / 128);
    m = std::max(m, pn(H, H, H / 128));
    m = std::max(m, pn(2 * F, H, F / 64));
    m = std::max(m, pn(H, F, H / 128));
    m = std::max(m, pn(V, H, (V + 127) / 128));
    return m * (B <= 16 ? 16 : 32);   // rows of NB floats (batch padded)
}

int tc_plan_create(const wq4_layer_table* t, int H, int F, int Nqkv, int V, int B, const TcBuffers& buf, int sms,
                   uint32_t* err, TcPlan** out)
{
    *out = nullptr;
    if (B > 32 || H % 256 || F % 256 || !encode_fn()) return WQ4_ERR_UNSUPPORTED;
    if ((Nqkv + 127) / 128 > kTcCounterWords || H / 128 > kTcCounterWords || F / 64 > kTcCounterWords)
        return WQ4_ERR_UNSUPPORTED;
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
        const bool ok = encode_2d(&mm.codes, CU_TENSOR_MAP_DATA_TYPE_UINT8, m.W, K / 2, N, K / 2, 128, 64,
                                  CU_TENSOR_MAP_SWIZZLE_128B) &&
                        encode_2d(&mm.scales, CU_TENSOR_MAP_DATA_TYPE_UINT16, m.s, K / 32, N, K / 16, 8, 64,
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
    for (int i = 0; i < 2 && ok; ++i)
        ok = encode_2d(&p->xH[i], CU_TENSOR_MAP_DATA_TYPE_FLOAT16, buf.xpH[i], H, 32, static_cast<uint64_t>(H) * 2, 64,
                       p->NB, CU_TENSOR_MAP_SWIZZLE_128B);
    ok = ok && encode_2d(&p->xF, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, buf.xpF, F, 32, static_cast<uint64_t>(F) * 2, 64,
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

// Records one token on `cs` (inside a stream capture): the prologue, then per
// layer the QKV, O, gate_up and down stages, then the LM head.  Every launch
// may overlap its set-up and weight stream with the tail of the previous one
// (programmatic dependent launch); it reads the previous stage's outputs only
// after that grid has completed.
int tc_launch_prologue(const uint16_t* x, int H, int B, float* sq, uint16_t* xp, cudaStream_t cs)
{
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(B);
    cfg.blockDim = dim3(128);
    cfg.stream = cs;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, tc_prologue_kernel, x, H, B, sq, xp) == cudaSuccess ? WQ4_OK : WQ4_ERR_CUDA;
}

int tc_record_token(const TcPlan* p, cudaStream_t cs, const TcAttnHook* att)
{
    const int B = p->B, H = p->H, F = p->F, L = p->L;
    const TcBuffers& u = p->buf;
    const size_t LH = static_cast<size_t>(B) * H;
    float* sq_u = u.sq;                                           // [H/128][B] each
    float* sq_a = u.sq + static_cast<size_t>(H / 128) * B;
    float* sq_x1 = u.sq + 2 * static_cast<size_t>(H / 128) * B;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    bool ok = true;
    auto stage = [&](int type, const TcMatMaps& m, const CUtensorMap& xmap, TcArgs a) {
        const int tiles = type == kTcGU ? F / 64 : (m.N + 127) / 128;
        const int P = stage_parts(tiles, m.K / 256, p->sms);
        a.type = type;
        a.N = m.N;
        a.K = m.K;
        a.B = B;
        a.P = P;
        a.tiles = tiles;
        a.units = tiles * P;
        a.H = H;
        a.F = F;
        a.eps = p->eps;
        a.part = u.part;
        a.cnt = u.cnt;
        a.err = p->err;
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(a.units < p->sms ? a.units : p->sms);
        cfg.blockDim = dim3(kTcThreads);
        cfg.stream = cs;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        cudaError_t e;
        if (p->NB == 16) {
            cfg.dynamicSmemBytes = TcSmem<16>::kBytes;
            e = cudaLaunchKernelEx(&cfg, tc_stage_kernel<16>, m.codes, m.scales, xmap, a);
        } else {
            cfg.dynamicSmemBytes = TcSmem<32>::kBytes;
            e = cudaLaunchKernelEx(&cfg, tc_stage_kernel<32>, m.codes, m.scales, xmap, a);
        }
        ok = ok && e == cudaSuccess;
    };
    {
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(B);
        cfg.blockDim = dim3(128);
        cfg.stream = cs;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        ok = ok && cudaLaunchKernelEx(&cfg, tc_prologue_kernel, u.x_stage, H, B, sq_u, u.xpH[0]) == cudaSuccess;
    }
    int hb = 0;   // which permuted H buffer holds the current stage's input
    for (int l = 0; l < L; ++l) {
        const TcMatMaps* m = &p->mats[4 * static_cast<size_t>(l)];
        const uint16_t* ul = (l == 0) ? u.x_stage : u.pX2 + static_cast<size_t>(l - 1) * LH;
        TcArgs a{};
        a.sq_in = sq_u;
        a.y = u.pQKV + static_cast<size_t>(l) * B * p->Nqkv;
        a.sq_out = sq_a;
        a.xp = u.xpH[hb ^ 1];
        a.ldxp = H;
        stage(kTcQKV, m[0], p->xH[hb], a);
        hb ^= 1;
        // decode step: the attention output replaces the query block as O's input
        if (att) ok = ok && att->record(att->ctx, l, cs, u.xpH[hb], sq_a) == WQ4_OK;

        a = TcArgs{};
        a.sq_in = sq_a;
        a.sq_u = sq_u;
        a.res = ul;
        a.y = u.pO + static_cast<size_t>(l) * LH;
        a.y2 = u.pX1 + static_cast<size_t>(l) * LH;
        a.y3 = u.pV + static_cast<size_t>(l) * LH;
        a.sq_out = sq_x1;
        a.xp = u.xpH[hb ^ 1];
        a.ldxp = H;
        stage(kTcO, m[1], p->xH[hb], a);
        hb ^= 1;

        a = TcArgs{};
        a.sq_in = sq_x1;
        a.y = u.pGU + static_cast<size_t>(l) * B * 2 * F;
        a.y2 = u.pM + static_cast<size_t>(l) * B * F;
        a.xp = u.xpF;
        a.ldxp = F;
        stage(kTcGU, m[2], p->xH[hb], a);

        a = TcArgs{};
        a.res = u.pX1 + static_cast<size_t>(l) * LH;
        a.y = u.pD + static_cast<size_t>(l) * LH;
        a.y2 = u.pX2 + static_cast<size_t>(l) * LH;
        a.sq_out = sq_u;                      // the next layer's (or the LM head's) input
        a.xp = u.xpH[hb ^ 1];
        a.ldxp = H;
        stage(kTcDOWN, m[3], p->xF, a);
        hb ^= 1;
    }
    TcArgs a{};
    a.sq_in = sq_u;
    a.res = u.pX2 + static_cast<size_t>(L - 1) * LH;
    a.y = u.logits;
    a.y3 = u.pV + static_cast<size_t>(L) * LH;
    stage(kTcLM, p->mats[4 * static_cast<size_t>(L)], p->xH[hb], a);
    return ok ? WQ4_OK : WQ4_ERR_CUDA;
}

}  // namespace wq4
