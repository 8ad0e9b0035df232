// wq4_tc_host.h -- internal interface between the chain planner and the
// tensor-core batched stage kernels (wq4_tc.cu).
#pragma once

#include <cstddef>
#include <cstdint>
#include <cuda_runtime.h>

#include "wq4.h"

namespace wq4 {

enum TcStageType { kTcQKV = 0, kTcO = 1, kTcGU = 2, kTcDOWN = 3, kTcLM = 4 };

// Workspace buffers of the batched path (device pointers).
struct TcBuffers {
    const uint16_t* x_stage;   // [B][H] token input
    uint16_t* pV;              // [L+1][B][H]
    uint16_t* pQKV;            // [L][B][Nqkv]
    uint16_t* pO;              // [L][B][H]
    uint16_t* pX1;             // [L][B][H]
    uint16_t* pGU;             // [L][B][2F]
    uint16_t* pM;              // [L][B][F]
    uint16_t* pD;              // [L][B][H]
    uint16_t* pX2;             // [L][B][H]
    uint16_t* logits;          // [B][V]
    float* sq;                 // 3 x [H/128][B] sums of squares of 128-element tiles (u, a, x1)
    uint32_t* cnt;             // [kTcCounterWords] arrival counters, zero-initialised
    uint16_t* xpH[2];          // [32][H] permuted stage inputs (K = H), alternating
    uint16_t* xpF;             // [32][F] permuted stage input (K = F)
    float* part;               // fp32 partial sums [P][B][N]
};

constexpr int kTcCounterWords = 4096;

struct TcPlan;

// Partial-sum floats the batched path needs (sms: an upper bound of the SM count).
size_t tc_part_floats(int L, int H, int F, int Nqkv, int V, int B, int sms);

int tc_plan_create(const wq4_layer_table* t, int H, int F, int Nqkv, int V, int B, const TcBuffers& buf, int sms,
                   uint32_t* err, TcPlan** out);
void tc_plan_destroy(TcPlan* p);

// Records the decode step's attention of layer `layer` on `cs`, between its
// QKV and O stages: it must leave the O stage's permuted input in xp and the
// sums of squares of its 128-element tiles in sq ([H/128][B]).
struct TcAttnHook {
    int (*record)(void* ctx, int layer, cudaStream_t cs, uint16_t* xp, float* sq);
    void* ctx;
};

// Records one token (prologue and every stage kernel) on `cs`; with `att`,
// the attention of every layer between its QKV and O stages.
int tc_record_token(const TcPlan* p, cudaStream_t cs, const TcAttnHook* att = nullptr);

// Records the token-start kernel on `cs` for an arbitrary [B][H] input: its
// permuted copy into xp and the sums of squares of its 128-element tiles
// into sq (programmatic dependent launch, like the stage kernels).
int tc_launch_prologue(const uint16_t* x, int H, int B, float* sq, uint16_t* xp, cudaStream_t cs);

}  // namespace wq4
