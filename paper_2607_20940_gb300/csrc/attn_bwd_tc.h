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
    float* dk_acc;        // [B, N, H, D] fp32, accumulated into
    float* dv_acc;
};

// dq (bf16) for every query, and the window key/value gradients added into
// dk_acc/dv_acc: one launch for dq, one per query group for dk/dv.
msf_status launch_bwd_tc(msf_plan_t plan, const BwdTcInput& in, cudaStream_t st);

}  // namespace msf
