// bf16 GEMM on the sm_103a tensor cores for the MSP tier projections:
// C[m, n] = sum_k A[m, k] * B[n, k], A and B K-contiguous (token rows and
// nn.Linear / Conv2d weight rows), fp32 accumulation in TMEM, one rounding
// to bf16. Used for the patch embedding of each tier (K = C*P^2, N = E) and
// the de-embedding of an emitted state (K = E, N = C*P^2).
//
// One CTA computes a 128 x BN tile of one stream's problem (optionally one
// K split of it):
//   warp 0  TMA producer: 64-wide K chunks of A (128 rows) and B (BN rows),
//           128-byte swizzled, into a STAGES ring
//   warp 1  MMA issuer: 4 x tcgen05.mma (K = 16) per chunk, accumulator in TMEM
//   warp 2  TMEM allocation
//   warps 4-7 epilogue: tcgen05.ld of the accumulator rows, then either a
//           bf16 pack and store, or fp32 partial sums of a K split
// The shared-memory ring and TMEM columns are small enough for 2-4 CTAs per
// SM, so short problems overlap one CTA's loads with another's epilogue.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <string.h>

#include "gemm_tc.h"
#include "kernels.h"
#include "ptx.cuh"

namespace msf {

namespace {

constexpr int kThreads = 256;
constexpr long long kWaitLimit = 2000000000LL;

template <int BN, int STAGES>
struct GCfg {
    static constexpr int kStages = STAGES;
    static constexpr int kABytes = 128 * 128;    // 128 rows x 64 bf16
    static constexpr int kBBytes = BN * 128;     // BN rows x 64 bf16
    static constexpr int kStageBytes = kABytes + kBBytes;
    static constexpr int kSmem = kStages * kStageBytes + 1024;
    static constexpr int kTmemCols = BN < 32 ? 32 : BN;
};

// Up to kMaxProblems independent problems (e.g. the tiers of one window) share
// one launch; blockIdx.x runs over all their 128 x BN tiles.
struct GemmTcProblem {
    int M, N, K;
    int m_tiles;
    int tile_base;        // first tile of this problem in blockIdx.x
    __nv_bfloat16* C;     // splits == 1: bf16 output
    long long ldc;        // elements
    long long c_bstride;  // elements
    float alpha;          // accumulator scale
};
struct GemmTcParams {
    int n_prob;
    GemmTcProblem pr[kMaxGemmProblems];
    int batch, splits;    // grid.z = batch * splits (splits > 1: one problem)
    float* C32;           // splits > 1: fp32 partial sums [split][batch][M][N]
    unsigned int* status;
};
struct GemmTcMaps {
    CUtensorMap a[kMaxGemmProblems];  // {K, rows, B}
    CUtensorMap b[kMaxGemmProblems];  // {K, N}
};

template <int BN, int STAGES>
__global__ void __launch_bounds__(kThreads, 1)
    gemm_tc_kernel(const __grid_constant__ GemmTcMaps maps, const __grid_constant__ GemmTcParams p) {
    using C = GCfg<BN, STAGES>;
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    unsigned char* smem = (unsigned char*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    __shared__ uint64_t full[C::kStages], empty[C::kStages], acc_full;
    __shared__ uint32_t tmem_base_sh;
    __shared__ int abort_flag;
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    int pi = 0;
    while (pi < p.n_prob - 1 && (int)blockIdx.x >= p.pr[pi + 1].tile_base) ++pi;
    const GemmTcProblem& P = p.pr[pi];
    const int local = (int)blockIdx.x - P.tile_base;
    const int m0 = (local % P.m_tiles) * 128, n0 = (local / P.m_tiles) * BN;
    const int b = blockIdx.z % p.batch, split = blockIdx.z / p.batch;
    const int nk_all = (P.K + 63) / 64;
    const int kc0 = (int)((long long)split * nk_all / p.splits);
    const int nk = (int)((long long)(split + 1) * nk_all / p.splits) - kc0;

    if (threadIdx.x == 0) {
        abort_flag = 0;
        for (int s = 0; s < C::kStages; ++s) {
            ptx::mbar_init(&full[s], 1);
            ptx::mbar_init(&empty[s], 1);
        }
        ptx::mbar_init(&acc_full, 1);
        ptx::fence_mbar_init();
    }
    if (warp == 2) {
        ptx::tmem_alloc(&tmem_base_sh, C::kTmemCols);
        ptx::tmem_relinquish();
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tbase = tmem_base_sh;
    volatile int* abort_p = &abort_flag;
    ptx::grid_dep_wait();  // inputs written by the previous kernel are visible
    ptx::grid_dep_launch();

    if (warp == 0 && lane == 0) {
        ptx::prefetch_tmap(&maps.a[pi]);
        ptx::prefetch_tmap(&maps.b[pi]);
        int issued = 0;
        bool ok = true;
        for (int kc = 0; kc < nk; ++kc) {
            const int st = kc % C::kStages;
            const uint32_t ph = (uint32_t)((kc / C::kStages) & 1);
            if (!ptx::mbar_wait_bounded(&empty[st], ph ^ 1u, abort_p, kWaitLimit)) {
                ok = false;
                break;
            }
            unsigned char* sa = smem + st * C::kStageBytes;
            ptx::mbar_arrive_expect_tx(&full[st], C::kStageBytes);
            ptx::tma_load_3d(sa, &maps.a[pi], &full[st], (kc0 + kc) * 64, m0, b);
            ptx::tma_load_2d(sa + C::kABytes, &maps.b[pi], &full[st], (kc0 + kc) * 64, n0);
            ++issued;
        }
        if (!ok) {
            volatile int never = 0;
            for (int kc = (issued > C::kStages ? issued - C::kStages : 0); kc < issued; ++kc)
                ptx::mbar_wait_bounded(&full[kc % C::kStages], (uint32_t)((kc / C::kStages) & 1),
                                       &never, kWaitLimit);
            atomicOr(p.status, kDevTimeout);
        }
    } else if (warp == 1 && lane == 0) {
        constexpr uint32_t idesc = ptx::idesc_bf16(128, BN, false, false);
        const uint32_t base = ptx::smem_u32(smem);
        bool ok = true;
        for (int kc = 0; kc < nk; ++kc) {
            const int st = kc % C::kStages;
            const uint32_t ph = (uint32_t)((kc / C::kStages) & 1);
            if (!ptx::mbar_wait_bounded(&full[st], ph, abort_p, kWaitLimit)) {
                ok = false;
                break;
            }
            ptx::tc_fence_after();
            const uint32_t sa = base + st * C::kStageBytes;
            const uint32_t sb = sa + C::kABytes;
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
                ptx::mma_ss(tbase, ptx::sdesc_sw128(sa + kk * 32, 16, 1024),
                            ptx::sdesc_sw128(sb + kk * 32, 16, 1024), idesc,
                            (kc > 0 || kk > 0) ? 1u : 0u);
            ptx::mma_commit(&empty[st]);
        }
        ptx::mma_commit(&acc_full);
        if (!ok) {
            volatile int never = 0;
            ptx::mbar_wait_bounded(&acc_full, 0, &never, kWaitLimit);
            atomicOr(p.status, kDevTimeout);
        }
    } else if (warp >= 4) {
        const int wq = warp % 4;
        const int r = wq * 32 + lane;
        bool ok = ptx::mbar_wait_bounded(&acc_full, 0, abort_p, kWaitLimit);
        ok = __all_sync(0xffffffffu, ok);
        if (ok) {
            ptx::tc_fence_after();
            const int m = m0 + r;
            const bool store = m < P.M;
            const uint32_t taddr = tbase + ((uint32_t)(wq * 32) << 16);
            if (p.splits == 1) {
                __nv_bfloat16* crow = P.C + (size_t)b * P.c_bstride + (size_t)m * P.ldc + n0;
#pragma unroll 1
                for (int c = 0; c < BN / 32; ++c) {
                    uint32_t v[32];
                    ptx::tmem_ld32(taddr + c * 32, v);
                    ptx::tmem_wait_ld();
                    uint32_t pk[16];
#pragma unroll
                    for (int e = 0; e < 16; ++e)
                        pk[e] = ptx::pack_bf16(P.alpha * __uint_as_float(v[2 * e]),
                                               P.alpha * __uint_as_float(v[2 * e + 1]));
                    const int ncol = n0 + c * 32;
                    if (store && ncol + 32 <= P.N) {
                        uint4* d4 = reinterpret_cast<uint4*>(crow + c * 32);
#pragma unroll
                        for (int e = 0; e < 4; ++e)
                            d4[e] = make_uint4(pk[4 * e], pk[4 * e + 1], pk[4 * e + 2], pk[4 * e + 3]);
                    } else if (store) {
                        const __nv_bfloat16* hb = reinterpret_cast<const __nv_bfloat16*>(pk);
                        for (int e = 0; e < 32 && ncol + e < P.N; ++e) crow[c * 32 + e] = hb[e];
                    }
                }
            } else {
                float* crow = p.C32 + (((size_t)split * p.batch + b) * P.M + m) * P.N + n0;
#pragma unroll 1
                for (int c = 0; c < BN / 32; ++c) {
                    uint32_t v[32];
                    ptx::tmem_ld32(taddr + c * 32, v);
                    ptx::tmem_wait_ld();
                    const int ncol = n0 + c * 32;
#pragma unroll
                    for (int e = 0; e < 32; ++e) v[e] = __float_as_uint(P.alpha * __uint_as_float(v[e]));
                    if (store && ncol + 32 <= P.N) {
                        float4* d4 = reinterpret_cast<float4*>(crow + c * 32);
#pragma unroll
                        for (int e = 0; e < 8; ++e)
                            d4[e] = make_float4(__uint_as_float(v[4 * e]), __uint_as_float(v[4 * e + 1]),
                                                __uint_as_float(v[4 * e + 2]), __uint_as_float(v[4 * e + 3]));
                    } else if (store) {
                        for (int e = 0; e < 32 && ncol + e < P.N; ++e) crow[c * 32 + e] = __uint_as_float(v[e]);
                    }
                }
            }
        } else if (lane == 0) {
            atomicOr(p.status, kDevTimeout);
        }
    }
    ptx::tc_fence_before();
    __syncthreads();
    if (warp == 2) {
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tbase, C::kTmemCols);
    }
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encoder() {
    static EncodeTiledFn fn = nullptr;
    if (!fn) {
        void* ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000,
                                             cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = (EncodeTiledFn)ptr;
    }
    return fn;
}

template <int BN, int STAGES>
cudaError_t launch_bn(const GemmTcArgs* gs, int n, int batch, int splits, cudaStream_t st) {
    EncodeTiledFn enc = encoder();
    if (!enc) return cudaErrorNotSupported;
    GemmTcMaps maps;
    memset(&maps, 0, sizeof(maps));
    GemmTcParams p;
    memset(&p, 0, sizeof(p));
    int tiles = 0;
    for (int i = 0; i < n; ++i) {
        const GemmTcArgs& g = gs[i];
        cuuint64_t adims[3] = {(cuuint64_t)g.K, (cuuint64_t)g.M, (cuuint64_t)batch};
        cuuint64_t astrides[2] = {(cuuint64_t)g.lda * 2, (cuuint64_t)g.a_bstride * 2};
        cuuint32_t abox[3] = {64, 128, 1};
        cuuint32_t es[3] = {1, 1, 1};
        if (enc(&maps.a[i], CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(g.A), adims, astrides,
                abox, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return cudaErrorInvalidValue;
        cuuint64_t bdims[2] = {(cuuint64_t)g.K, (cuuint64_t)(g.b_rows > 0 ? g.b_rows : g.N)};
        cuuint64_t bstrides[1] = {(cuuint64_t)g.ldb * 2};
        cuuint32_t bbox[2] = {64, (cuuint32_t)BN};
        if (enc(&maps.b[i], CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(g.B), bdims, bstrides,
                bbox, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return cudaErrorInvalidValue;
        GemmTcProblem& pr = p.pr[i];
        pr.M = g.M;
        pr.N = g.N;
        pr.K = g.K;
        pr.alpha = g.alpha;
        pr.m_tiles = (g.M + 127) / 128;
        pr.tile_base = tiles;
        pr.C = (__nv_bfloat16*)g.C;
        pr.ldc = g.ldc;
        pr.c_bstride = g.c_bstride;
        tiles += pr.m_tiles * ((g.N + BN - 1) / BN);
    }
    p.n_prob = n;
    p.batch = batch;
    p.splits = splits;
    p.C32 = gs[0].C32;
    p.status = gs[0].status;
    cudaError_t e = set_smem_attr((const void*)gemm_tc_kernel<BN, STAGES>, GCfg<BN, STAGES>::kSmem);
    if (e != cudaSuccess) return e;
    dim3 grid((unsigned)tiles, 1, (unsigned)(batch * splits));
    return launch_pdl(gemm_tc_kernel<BN, STAGES>, grid, dim3(kThreads), GCfg<BN, STAGES>::kSmem, st,
                      maps, p);
}

}  // namespace

bool gemm_tc_supported(const GemmTcArgs& g) {
    // TMA: 16-byte aligned bases and row strides; K chunks of 64.
    if (((uintptr_t)g.A & 15) || ((uintptr_t)g.B & 15) || ((uintptr_t)g.C & 15)) return false;
    if ((g.lda * 2) % 16 || (g.ldb * 2) % 16 || (g.a_bstride * 2) % 16) return false;
    if (g.ldc % 8 || g.c_bstride % 8) return false;
    if (g.K % 64 || g.M < 1 || g.N < 1) return false;
    return true;
}

cudaError_t launch_gemm_tc(const GemmTcArgs& g, int batch, cudaStream_t st) {
    // Few, long tiles (the de-embedding: K = E, N = C*P^2): split K across
    // CTAs into fp32 partial sums when the caller provides room for them.
    if (g.C32 && g.max_splits > 1) {
        const int tiles = ((g.M + 127) / 128) * ((g.N + 127) / 128) * batch;
        const int nk = g.K / 64;
        int splits = 1;
        while (splits * 2 <= g.max_splits && tiles * splits * 2 <= 160 && nk / (splits * 2) >= 2)
            splits *= 2;
        g.splits_used = splits;
        if (splits > 1) {
            if (g.N <= 64) return launch_bn<64, 4>(&g, 1, batch, splits, st);
            return launch_bn<128, 4>(&g, 1, batch, splits, st);
        }
    }
    g.splits_used = 1;
    if (g.N <= 64) return launch_bn<64, 4>(&g, 1, batch, 1, st);
    return launch_bn<128, 2>(&g, 1, batch, 1, st);
}

cudaError_t launch_gemm_tc_grouped(const GemmTcArgs* gs, int n, int batch, cudaStream_t st) {
    if (n < 1 || n > kMaxGemmProblems) return cudaErrorInvalidValue;
    bool narrow = true;
    for (int i = 0; i < n; ++i) {
        gs[i].splits_used = 1;
        narrow = narrow && gs[i].N <= 64;
    }
    if (narrow) return launch_bn<64, 4>(gs, n, batch, 1, st);
    return launch_bn<128, 2>(gs, n, batch, 1, st);
}

}  // namespace msf
