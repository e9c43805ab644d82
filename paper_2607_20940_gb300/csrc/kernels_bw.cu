// Bandwidth-bound kernels of the window pass:
//   - KV pyramid pooling (Eq. 4's Subsample), also used by the history append
//   - MSP raw patchify / unpatchify (Sec. 4.1 token rearrangement)
//   - a CUDA-core GEMM for the tier projections of fp32 plans
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "kernels.h"
#include "pool.cuh"
#include "ptx.cuh"

namespace msf {

// ----------------------------------------------------------------- pooling
// (arithmetic in pool.cuh)

template <typename T>
__global__ void __launch_bounds__(256, 2) pool_kernel(const PoolBatch jobs) {
    ptx::grid_dep_wait();
    ptx::grid_dep_launch();
    pool_task<T>(jobs, blockIdx.y, blockIdx.z, blockIdx.x * blockDim.x + threadIdx.x);
}

cudaError_t launch_pool(const PoolBatch& jobs, int batch, bool bf16, cudaStream_t st) {
    if (jobs.n == 0) return cudaSuccess;
    int max_n = 0;
    for (int k = 0; k < jobs.n; ++k) max_n = jobs.j[k].out_n > max_n ? jobs.j[k].out_n : max_n;
    long long work = (long long)max_n * (jobs.row_vecs / 2);
    dim3 grid((unsigned)((work + 255) / 256), (unsigned)jobs.n, (unsigned)batch);
    if (bf16)
        return launch_pdl(pool_kernel<__nv_bfloat16>, grid, dim3(256), 0, st, jobs);
    else
        return launch_pdl(pool_kernel<float>, grid, dim3(256), 0, st, jobs);
    return cudaGetLastError();
}

// ------------------------------------------------------------ MSP raw tokens
//
// Raw layout: [B, T, C*Hl*Wl]; state l's block is [G/s_l^2 tokens, C*P^2]
// with P = patch*s_l and feature (c, dy, dx). Threads walk the output
// (patchify) or the latent (unpatchify) linearly so that writes coalesce.

template <typename T>
__global__ void __launch_bounds__(256) patchify_raw_kernel(const T* __restrict__ latent,
                                                           T* __restrict__ raw, MspShape sh, int l0) {
    ptx::grid_dep_wait();
    ptx::grid_dep_launch();
    const int l = l0 + (int)blockIdx.y, b = blockIdx.z;
    const int per = sh.C * sh.Hl * sh.Wl;
    const int o = blockIdx.x * blockDim.x + threadIdx.x;
    if (o >= per) return;
    const int P = sh.patch * sh.scales[l];
    const int PP = P * P, F = sh.C * PP, gw = sh.Wl / P;
    const int t = o / F, f = o - t * F;
    const int c = f / PP, r = f - c * PP, dy = r / P, dx = r - (r / P) * P;
    const int i = t / gw, j = t - (t / gw) * gw;
    const size_t base = ((size_t)b * sh.T + l) * per;
    raw[base + o] = latent[base + (size_t)c * sh.Hl * sh.Wl + (size_t)(P * i + dy) * sh.Wl + P * j + dx];
}

template <typename T>
__global__ void __launch_bounds__(256) unpatchify_raw_kernel(const T* __restrict__ raw,
                                                             T* __restrict__ latent, MspShape sh,
                                                             int position, long long raw_bstride,
                                                             int raw_offset) {
    ptx::grid_dep_wait();
    ptx::grid_dep_launch();
    const int b = blockIdx.z;
    const int per = sh.C * sh.Hl * sh.Wl;
    const int o = blockIdx.x * blockDim.x + threadIdx.x;
    if (o >= per) return;
    const int P = sh.patch * sh.scales[position];
    const int PP = P * P, F = sh.C * PP, gw = sh.Wl / P;
    const int c = o / (sh.Hl * sh.Wl), yx = o - c * (sh.Hl * sh.Wl);
    const int y = yx / sh.Wl, x = yx - (yx / sh.Wl) * sh.Wl;
    const int i = y / P, dy = y - i * P, j = x / P, dx = x - j * P;
    const int t = i * gw + j, f = c * PP + dy * P + dx;
    latent[(size_t)b * per + o] = raw[(size_t)b * raw_bstride + raw_offset + (size_t)t * F + f];
}

cudaError_t launch_patchify_raw(const void* latent, void* raw, const MspShape& sh, int batch,
                                bool bf16, cudaStream_t st, int l0, int n_states) {
    const int per = sh.C * sh.Hl * sh.Wl;
    if (n_states < 0) n_states = sh.T - l0;
    dim3 grid((unsigned)((per + 255) / 256), (unsigned)n_states, (unsigned)batch);
    if (bf16)
        return launch_pdl(patchify_raw_kernel<__nv_bfloat16>, grid, dim3(256), 0, st,
                          (const __nv_bfloat16*)latent, (__nv_bfloat16*)raw, sh, l0);
    return launch_pdl(patchify_raw_kernel<float>, grid, dim3(256), 0, st, (const float*)latent,
                      (float*)raw, sh, l0);
}

cudaError_t launch_unpatchify_raw(const void* raw, void* latent, const MspShape& sh, int position,
                                  long long raw_bstride, int raw_offset, int batch, bool bf16,
                                  cudaStream_t st) {
    const int per = sh.C * sh.Hl * sh.Wl;
    dim3 grid((unsigned)((per + 255) / 256), 1, (unsigned)batch);
    if (bf16)
        return launch_pdl(unpatchify_raw_kernel<__nv_bfloat16>, grid, dim3(256), 0, st,
                          (const __nv_bfloat16*)raw, (__nv_bfloat16*)latent, sh, position, raw_bstride,
                          raw_offset);
    return launch_pdl(unpatchify_raw_kernel<float>, grid, dim3(256), 0, st, (const float*)raw,
                      (float*)latent, sh, position, raw_bstride, raw_offset);
}

__global__ void __launch_bounds__(256) unpatchify_splitk_kernel(const float* __restrict__ part,
                                                                int splits,
                                                                __nv_bfloat16* __restrict__ latent,
                                                                MspShape sh, int position,
                                                                int batch) {
    ptx::grid_dep_wait();
    ptx::grid_dep_launch();
    const int b = blockIdx.z;
    const int per = sh.C * sh.Hl * sh.Wl;
    const int o = blockIdx.x * blockDim.x + threadIdx.x;
    if (o >= per) return;
    const int P = sh.patch * sh.scales[position];
    const int PP = P * P, F = sh.C * PP, gw = sh.Wl / P;
    const int c = o / (sh.Hl * sh.Wl), yx = o - c * (sh.Hl * sh.Wl);
    const int y = yx / sh.Wl, x = yx - (yx / sh.Wl) * sh.Wl;
    const int i = y / P, dy = y - i * P, j = x / P, dx = x - j * P;
    const size_t src = (size_t)(i * gw + j) * F + c * PP + dy * P + dx;
    float acc = 0.f;
    for (int sp = 0; sp < splits; ++sp) acc += __ldg(part + ((size_t)sp * batch + b) * per + src);
    latent[(size_t)b * per + o] = __float2bfloat16_rn(acc);
}

cudaError_t launch_unpatchify_splitk(const float* part, int splits, void* latent, const MspShape& sh,
                                     int position, int batch, cudaStream_t st) {
    const int per = sh.C * sh.Hl * sh.Wl;
    dim3 grid((unsigned)((per + 255) / 256), 1, (unsigned)batch);
    return launch_pdl(unpatchify_splitk_kernel, grid, dim3(256), 0, st, part, splits,
                      (__nv_bfloat16*)latent, sh, position, batch);
}

// --------------------------------------------------------- CUDA-core GEMM
//
// C[m, n] = sum_k A[m, k] * B[n, k] (both operands K-contiguous), fp32
// accumulation, one rounding to T. 64x64 tiles, 256 threads, 4x4 outputs per
// thread, K staged through shared memory 16 at a time.

template <typename T>
__device__ __forceinline__ float ld_f(const T* p);
template <>
__device__ __forceinline__ float ld_f(const float* p) { return __ldg(p); }
template <>
__device__ __forceinline__ float ld_f(const __nv_bfloat16* p) { return __bfloat162float(*p); }
template <typename T>
__device__ __forceinline__ T to_t(float x);
template <>
__device__ __forceinline__ float to_t(float x) { return x; }
template <>
__device__ __forceinline__ __nv_bfloat16 to_t(float x) { return __float2bfloat16_rn(x); }

template <typename T>
__global__ void __launch_bounds__(256) gemm_nt_simt_kernel(GemmArgs g) {
    ptx::grid_dep_wait();
    ptx::grid_dep_launch();
    __shared__ float As[16][65];
    __shared__ float Bs[16][65];
    const int b = blockIdx.z;
    const T* A = (const T*)g.A + (size_t)b * g.a_bstride;
    const T* Bm = (const T*)g.B;
    T* C = (T*)g.C + (size_t)b * g.c_bstride;
    const int m0 = blockIdx.y * 64, n0 = blockIdx.x * 64;
    const int tx = threadIdx.x % 16, ty = threadIdx.x / 16;
    float acc[4][4] = {};
    for (int k0 = 0; k0 < g.K; k0 += 16) {
        for (int e = threadIdx.x; e < 64 * 16; e += 256) {
            int r = e / 16, kk = e % 16;
            int m = m0 + r, n = n0 + r, k = k0 + kk;
            As[kk][r] = (m < g.M && k < g.K) ? ld_f<T>(A + (size_t)m * g.lda + k) : 0.f;
            Bs[kk][r] = (n < g.N && k < g.K) ? ld_f<T>(Bm + (size_t)n * g.ldb + k) : 0.f;
        }
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < 16; ++kk) {
            float a[4], bb[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                a[u] = As[kk][ty + 16 * u];
                bb[u] = Bs[kk][tx + 16 * u];
            }
#pragma unroll
            for (int u = 0; u < 4; ++u)
#pragma unroll
                for (int v = 0; v < 4; ++v) acc[u][v] = fmaf(a[u], bb[v], acc[u][v]);
        }
        __syncthreads();
    }
#pragma unroll
    for (int u = 0; u < 4; ++u)
#pragma unroll
        for (int v = 0; v < 4; ++v) {
            int m = m0 + ty + 16 * u, n = n0 + tx + 16 * v;
            if (m < g.M && n < g.N) C[(size_t)m * g.ldc + n] = to_t<T>(acc[u][v]);
        }
}

cudaError_t launch_gemm_nt_simt(const GemmArgs& g, int batch, bool bf16, cudaStream_t st) {
    dim3 grid((unsigned)((g.N + 63) / 64), (unsigned)((g.M + 63) / 64), (unsigned)batch);
    if (bf16)
        return launch_pdl(gemm_nt_simt_kernel<__nv_bfloat16>, grid, dim3(256), 0, st, g);
    else
        return launch_pdl(gemm_nt_simt_kernel<float>, grid, dim3(256), 0, st, g);
    return cudaGetLastError();
}

}  // namespace msf
