// Tensor-core MSSA backward (tcgen05 + TMA) launcher interface.
#pragma once

#include <cuda_runtime.h>

#include "internal.h"
#include "kernels.h"

namespace msf {

struct BwdTcInput {
    const AttnArgs* a;    // the forward's context segments (q = the forward's q)
    const BwdGroup* g;    // per group (same order as a->g): rows that receive gradients
    const void* q;        // [B, N, H, D] bf16
    const void* dout;     // [B, N, H, D] bf16
    const float* lse;     // [B, H, N]
    const float* delta;   // [B, H, N]
    void* dq;             // [B, N, H, D] bf16, written
    float* dk_ctx;        // [B, R, H, D] fp32 context-row gradients, written
    float* dv_ctx;
    int R;
};

// dq (bf16) for every query (one launch), and the key/value gradients of
// every group's window-derived context rows (one launch).
msf_status launch_bwd_tc(msf_plan_t plan, const BwdTcInput& in, cudaStream_t st);

}  // namespace msf
