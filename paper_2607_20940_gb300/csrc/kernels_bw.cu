// Bandwidth-bound kernels of the window pass:
//   - KV pyramid pooling (Eq. 4's Subsample), also used by the history append
//   - MSP raw patchify / unpatchify (Sec. 4.1 token rearrangement)
//   - a CUDA-core GEMM for the tier projections of fp32 plans
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "kernels.h"
#include "ptx.cuh"

namespace msf {

// ----------------------------------------------------------------- pooling
//
// One thread produces two adjacent 16-byte vectors of one pooled token's
// [H*D] row, for K and V together: it loads sigma^2 source vectors of each
// (independent 128-bit loads of rows that are contiguous in [B, N, H, D]),
// sums them in fp32 in a fixed (dy, dx) order, scales by 1/sigma^2 (exact)
// and rounds once. STRIDED copies the block's top-left vectors.

template <typename T>
struct Vec;
template <>
struct Vec<__nv_bfloat16> {
    static constexpr int n = 8;
    __device__ static void add(float* acc, const uint4& v) {
        const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            float2 f = __bfloat1622float2(h[i]);
            acc[2 * i] += f.x;
            acc[2 * i + 1] += f.y;
        }
    }
    __device__ static uint4 pack(const float* acc, float mul) {
        uint4 r;
        __nv_bfloat162* h = reinterpret_cast<__nv_bfloat162*>(&r);
#pragma unroll
        for (int i = 0; i < 4; ++i) h[i] = __floats2bfloat162_rn(acc[2 * i] * mul, acc[2 * i + 1] * mul);
        return r;
    }
};
template <>
struct Vec<float> {
    static constexpr int n = 4;
    __device__ static void add(float* acc, const uint4& v) {
        acc[0] += __uint_as_float(v.x);
        acc[1] += __uint_as_float(v.y);
        acc[2] += __uint_as_float(v.z);
        acc[3] += __uint_as_float(v.w);
    }
    __device__ static uint4 pack(const float* acc, float mul) {
        return make_uint4(__float_as_uint(acc[0] * mul), __float_as_uint(acc[1] * mul),
                          __float_as_uint(acc[2] * mul), __float_as_uint(acc[3] * mul));
    }
};

// Two adjacent 16-byte vectors of one pooled token, K and V. With the stride
// known at compile time the loads of RG tap rows are issued before their first
// add (all 4*S*S of them for S <= 2; one row of 4*S for S = 4, which keeps the
// thread under ~128 registers so the kernel does not spill). ck/cv (NULL =
// none) receive a copy of every source vector read, at its source token index
// (the staged history head: one read serves the ring copy and the pooled
// level). Sums run in the fixed (dy, dx) order whatever RG is.
template <typename T, int S>
__device__ __forceinline__ void pool_pair(const char* sk, const char* sv, char* dk, char* dv,
                                          char* ck, char* cv, int src_gw, int i, int jj,
                                          size_t row, int mode) {
    const bool strided = mode == MSF_RESAMPLE_STRIDED;
    if (S == 1 || (strided && !ck)) {
        const size_t src = (size_t)((S * i) * src_gw + S * jj) * row;
        const uint4 k0 = __ldg(reinterpret_cast<const uint4*>(sk + src));
        const uint4 k1 = __ldg(reinterpret_cast<const uint4*>(sk + src + 16));
        const uint4 v0 = __ldg(reinterpret_cast<const uint4*>(sv + src));
        const uint4 v1 = __ldg(reinterpret_cast<const uint4*>(sv + src + 16));
        if (ck) {  // S == 1 here
            *reinterpret_cast<uint4*>(ck + src) = k0;
            *reinterpret_cast<uint4*>(ck + src + 16) = k1;
            *reinterpret_cast<uint4*>(cv + src) = v0;
            *reinterpret_cast<uint4*>(cv + src + 16) = v1;
        }
        *reinterpret_cast<uint4*>(dk) = k0;
        *reinterpret_cast<uint4*>(dk + 16) = k1;
        *reinterpret_cast<uint4*>(dv) = v0;
        *reinterpret_cast<uint4*>(dv + 16) = v1;
        return;
    }
    constexpr int RG = S <= 2 ? S : 1;  // tap rows whose loads are in flight together
    float ak[2][Vec<T>::n], av[2][Vec<T>::n];
#pragma unroll
    for (int h = 0; h < 2; ++h)
#pragma unroll
        for (int e = 0; e < Vec<T>::n; ++e) ak[h][e] = av[h][e] = 0.f;
#pragma unroll 1
    for (int y0 = 0; y0 < S; y0 += RG) {
        uint4 xk[RG * S][2], xv[RG * S][2];
#pragma unroll
        for (int t = 0; t < RG * S; ++t) {
            const int dy = y0 + t / S, dx = t % S;
            const size_t src = (size_t)((S * i + dy) * src_gw + S * jj + dx) * row;
            xk[t][0] = __ldg(reinterpret_cast<const uint4*>(sk + src));
            xk[t][1] = __ldg(reinterpret_cast<const uint4*>(sk + src + 16));
            xv[t][0] = __ldg(reinterpret_cast<const uint4*>(sv + src));
            xv[t][1] = __ldg(reinterpret_cast<const uint4*>(sv + src + 16));
        }
        if (ck) {
#pragma unroll
            for (int t = 0; t < RG * S; ++t) {
                const int dy = y0 + t / S, dx = t % S;
                const size_t src = (size_t)((S * i + dy) * src_gw + S * jj + dx) * row;
                *reinterpret_cast<uint4*>(ck + src) = xk[t][0];
                *reinterpret_cast<uint4*>(ck + src + 16) = xk[t][1];
                *reinterpret_cast<uint4*>(cv + src) = xv[t][0];
                *reinterpret_cast<uint4*>(cv + src + 16) = xv[t][1];
            }
        }
        if (strided) {  // the block's top-left vectors
            if (y0 == 0) {
                *reinterpret_cast<uint4*>(dk) = xk[0][0];
                *reinterpret_cast<uint4*>(dk + 16) = xk[0][1];
                *reinterpret_cast<uint4*>(dv) = xv[0][0];
                *reinterpret_cast<uint4*>(dv + 16) = xv[0][1];
            }
            continue;
        }
#pragma unroll
        for (int t = 0; t < RG * S; ++t)
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                Vec<T>::add(ak[h], xk[t][h]);
                Vec<T>::add(av[h], xv[t][h]);
            }
    }
    if (strided) return;
    const float mul = 1.0f / (float)(S * S);
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        *reinterpret_cast<uint4*>(dk + 16 * h) = Vec<T>::pack(ak[h], mul);
        *reinterpret_cast<uint4*>(dv + 16 * h) = Vec<T>::pack(av[h], mul);
    }
}

template <typename T>
__global__ void __launch_bounds__(256, 2) pool_kernel(const PoolBatch jobs) {
    ptx::grid_dep_wait();
    ptx::grid_dep_launch();
    const PoolJob& jb = jobs.j[blockIdx.y];
    const int b = blockIdx.z;
    const int idx = blockIdx.x * blockDim.x + threadIdx.x;
    const int rp = jobs.row_vecs / 2;  // vector pairs per token row
    const int tok = idx / rp;
    if (tok >= jb.out_n) return;
    const int vec = 2 * (idx - tok * rp);
    const int i = tok / jb.out_gw, jj = tok - (tok / jb.out_gw) * jb.out_gw;
    const size_t row = (size_t)jobs.row_vecs * 16;
    const char* sk = jb.src_k + (size_t)b * jb.src_bstride + (size_t)vec * 16;
    const char* sv = jb.src_v + (size_t)b * jb.src_bstride + (size_t)vec * 16;
    char* dk = jb.dst_k + (size_t)b * jb.dst_bstride + (size_t)tok * row + (size_t)vec * 16;
    char* dv = jb.dst_v + (size_t)b * jb.dst_bstride + (size_t)tok * row + (size_t)vec * 16;
    char* ck = nullptr;
    char* cv = nullptr;
    if (jb.copy_k) {
        ck = jb.copy_k + (size_t)b * jb.copy_bstride + (size_t)vec * 16;
        cv = jb.copy_v + (size_t)b * jb.copy_bstride + (size_t)vec * 16;
    }
    switch (jb.sigma) {
    case 1: pool_pair<T, 1>(sk, sv, dk, dv, ck, cv, jb.src_gw, i, jj, row, jobs.mode); break;
    case 2: pool_pair<T, 2>(sk, sv, dk, dv, ck, cv, jb.src_gw, i, jj, row, jobs.mode); break;
    case 4: pool_pair<T, 4>(sk, sv, dk, dv, ck, cv, jb.src_gw, i, jj, row, jobs.mode); break;
    default: {
        // Larger strides (never with a copy): same arithmetic, loads issued per tap.
        const int s = jb.sigma;
        for (int h = 0; h < 2; ++h) {
            if (jobs.mode == MSF_RESAMPLE_STRIDED) {
                const size_t src = (size_t)((s * i) * jb.src_gw + s * jj) * row + 16 * h;
                *reinterpret_cast<uint4*>(dk + 16 * h) = __ldg(reinterpret_cast<const uint4*>(sk + src));
                *reinterpret_cast<uint4*>(dv + 16 * h) = __ldg(reinterpret_cast<const uint4*>(sv + src));
                continue;
            }
            float ak[Vec<T>::n], av[Vec<T>::n];
            for (int e = 0; e < Vec<T>::n; ++e) ak[e] = av[e] = 0.f;
            for (int dy = 0; dy < s; ++dy)
                for (int dx = 0; dx < s; ++dx) {
                    const size_t src = (size_t)((s * i + dy) * jb.src_gw + s * jj + dx) * row + 16 * h;
                    Vec<T>::add(ak, __ldg(reinterpret_cast<const uint4*>(sk + src)));
                    Vec<T>::add(av, __ldg(reinterpret_cast<const uint4*>(sv + src)));
                }
            const float mul = 1.0f / (float)(s * s);
            *reinterpret_cast<uint4*>(dk + 16 * h) = Vec<T>::pack(ak, mul);
            *reinterpret_cast<uint4*>(dv + 16 * h) = Vec<T>::pack(av, mul);
        }
    }
    }
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
                                                           T* __restrict__ raw, MspShape sh) {
    ptx::grid_dep_wait();
    ptx::grid_dep_launch();
    const int l = blockIdx.y, b = blockIdx.z;
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
                                bool bf16, cudaStream_t st) {
    const int per = sh.C * sh.Hl * sh.Wl;
    dim3 grid((unsigned)((per + 255) / 256), (unsigned)sh.T, (unsigned)batch);
    if (bf16)
        return launch_pdl(patchify_raw_kernel<__nv_bfloat16>, grid, dim3(256), 0, st,
                          (const __nv_bfloat16*)latent, (__nv_bfloat16*)raw, sh);
    return launch_pdl(patchify_raw_kernel<float>, grid, dim3(256), 0, st, (const float*)latent,
                      (float*)raw, sh);
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
