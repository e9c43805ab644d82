// Tensor-core bf16 GEMM (C = A * B^T, K-contiguous operands) for the MSP
// tier projections.
#pragma once

#include <cuda_runtime.h>

#include "internal.h"

namespace msf {

struct GemmTcArgs {
    const void* A;  // [batch][M rows, stride lda][K] bf16
    const void* B;  // [N rows, stride ldb][K] bf16 (shared by the batch)
    void* C;        // [batch][M rows, stride ldc][N] bf16
    int M, N, K;
    long long lda, ldb, ldc;       // elements
    long long a_bstride, c_bstride;  // elements
    unsigned int* status;
};

bool gemm_tc_supported(const GemmTcArgs& g);
cudaError_t launch_gemm_tc(const GemmTcArgs& g, int batch, cudaStream_t st);

}  // namespace msf
