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
    // Optional split-K: room for max_splits fp32 partial outputs
    // [split][batch][M][N] (contiguous). The launcher reports the split count
    // it used in splits_used; 1 means C was written directly.
    float* C32 = nullptr;
    int max_splits = 1;
    mutable int splits_used = 1;
    // Scale applied to the accumulator before the output is written.
    float alpha = 1.0f;
    // Rows of B actually present (0: N). Rows [b_rows, N) read as zeros, so
    // output columns past b_rows are written as zeros.
    int b_rows = 0;
};

constexpr int kMaxGemmProblems = 4;

bool gemm_tc_supported(const GemmTcArgs& g);
cudaError_t launch_gemm_tc(const GemmTcArgs& g, int batch, cudaStream_t st);
// Several independent problems (no K split) in one launch.
cudaError_t launch_gemm_tc_grouped(const GemmTcArgs* gs, int n, int batch, cudaStream_t st);

}  // namespace msf
