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
    float* rf;                 // [L+1][3][B] RMS factors
    uint16_t* xpH;             // [32][H] permuted stage input (K = H)
    uint16_t* xpF;             // [32][F] permuted stage input (K = F)
    float* part;               // fp32 partial sums [P][B][N]
};

// Arguments of one stage epilogue (one CTA per batch row).
struct TcEpi {
    int type, N, B, P, H, F;
    float eps;
    const float* part;
    const float* r_in;       // row factor of the stage (null: 1)
    const uint16_t* v_in;    // residual input (O: v, down: x1)
    uint16_t* y;             // stage output trace
    uint16_t* y2;            // second output (O: x1, gate_up: m, down: x2)
    uint16_t* v_out;         // down: next layer's normalised input
    float* r_out;            // RMS factor of the next stage's input (null: none)
    uint16_t* xp;            // next stage's permuted input row
};

struct TcPlan;

// Partial-sum floats the batched path needs (sms: an upper bound of the SM count).
size_t tc_part_floats(int L, int H, int F, int Nqkv, int V, int B, int sms);

int tc_plan_create(const wq4_layer_table* t, int H, int F, int Nqkv, int V, int B, const TcBuffers& buf, int sms,
                   uint32_t* err, TcPlan** out);
void tc_plan_destroy(TcPlan* p);

// Records one token (every stage kernel and epilogue) on `cs`.
void tc_record_token(const TcPlan* p, cudaStream_t cs);

}  // namespace wq4
