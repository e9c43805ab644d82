// MSSA attention on CUDA cores in fp32 (Eq. 4 context, online softmax).
//
// This is the fp32 path of the library (max |err| <= 1e-4 against the fp64
// definition) and a cross-check of the tensor-core kernel. A block owns 32
// queries of one (stream, head, group); four threads share a query, each
// holding every fourth element of q and of the running output, so that a
// warp reads four consecutive shared-memory words per key (no bank
// conflicts). Keys and values of each context segment are staged 32 rows at
// a time in shared memory as fp32.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math.h>

#include "kernels.h"
#include "ptx.cuh"

namespace msf {

template <typename T>
__device__ __forceinline__ float ldf(const T* p);
template <>
__device__ __forceinline__ float ldf(const float* p) { return *p; }
template <>
__device__ __forceinline__ float ldf(const __nv_bfloat16* p) { return __bfloat162float(*p); }
template <typename T>
__device__ __forceinline__ T tot(float x);
template <>
__device__ __forceinline__ float tot(float x) { return x; }
template <>
__device__ __forceinline__ __nv_bfloat16 tot(float x) { return __float2bfloat16_rn(x); }

template <typename T, int D>
__global__ void __launch_bounds__(128) attn_simt_kernel(const AttnArgs a) {
    ptx::grid_dep_wait();
    ptx::grid_dep_launch();
    constexpr int DP = D / 4;
    constexpr int KT = 32;
    __shared__ float Ks[KT][D];
    __shared__ float Vs[KT][D];

    int tile = blockIdx.x, gi = 0;
    while (gi < a.n_groups) {
        int nt = (a.g[gi].q_end - a.g[gi].q_begin + 31) / 32;
        if (tile < nt) break;
        tile -= nt;
        ++gi;
    }
    if (gi >= a.n_groups) return;
    const AttnGroup& G = a.g[gi];
    const int h = blockIdx.y, b = blockIdx.z;
    const int qi = threadIdx.x / 4, c = threadIdx.x % 4;
    const int t = G.q_begin + tile * 32 + qi;
    const bool valid = t < G.q_end;
    const size_t row = (size_t)a.H * D * sizeof(T);

    const T* qp = (const T*)(a.q + (size_t)b * a.q_bstride + (size_t)(valid ? t : G.q_begin) * row) +
                  (size_t)h * D;
    float q[DP], o[DP];
#pragma unroll
    for (int i = 0; i < DP; ++i) {
        q[i] = ldf<T>(qp + 4 * i + c) * a.scale_log2;
        o[i] = 0.f;
    }
    float m = -INFINITY, l = 0.f;

    for (int s = 0; s < G.n_seg; ++s) {
        const Segment& sg = G.seg[s];
        const char* kb = sg.k + (size_t)b * sg.bstride + (size_t)sg.row0 * row + (size_t)h * D * sizeof(T);
        const char* vb = sg.v + (size_t)b * sg.bstride + (size_t)sg.row0 * row + (size_t)h * D * sizeof(T);
        for (int kt = 0; kt < sg.len; kt += KT) {
            const int n = min(KT, sg.len - kt);
            __syncthreads();
            for (int e = threadIdx.x; e < n * D; e += blockDim.x) {
                const int key = e / D, d = e - key * D;
                Ks[key][d] = ldf<T>((const T*)(kb + (size_t)(kt + key) * row) + d);
                Vs[key][d] = ldf<T>((const T*)(vb + (size_t)(kt + key) * row) + d);
            }
            __syncthreads();
            for (int j = 0; j < n; ++j) {
                float sc = 0.f;
#pragma unroll
                for (int i = 0; i < DP; ++i) sc = fmaf(q[i], Ks[j][4 * i + c], sc);
                sc += __shfl_xor_sync(0xffffffffu, sc, 1);
                sc += __shfl_xor_sync(0xffffffffu, sc, 2);
                if (sc > m) {
                    const float corr = exp2f(m - sc);
                    l *= corr;
#pragma unroll
                    for (int i = 0; i < DP; ++i) o[i] *= corr;
                    m = sc;
                }
                const float p = exp2f(sc - m);
                l += p;
#pragma unroll
                for (int i = 0; i < DP; ++i) o[i] = fmaf(p, Vs[j][4 * i + c], o[i]);
            }
        }
    }
    if (!valid) return;
    T* op = (T*)(a.out + (size_t)b * a.q_bstride + (size_t)t * row) + (size_t)h * D;
    const float inv = 1.0f / l;
    // scores are in log2 units: ln sum_j exp(s_j) = (m + log2 l) * ln 2
    if (a.lse && c == 0) a.lse[((size_t)b * a.H + h) * a.N + t] = (m + log2f(l)) * 0.6931471805599453f;
#pragma unroll
    for (int i = 0; i < DP; ++i) op[4 * i + c] = tot<T>(o[i] * inv);
}

cudaError_t launch_attn_simt(const AttnArgs& a, bool bf16, cudaStream_t st) {
    int tiles = 0;
    for (int gi = 0; gi < a.n_groups; ++gi) tiles += (a.g[gi].q_end - a.g[gi].q_begin + 31) / 32;
    if (tiles == 0) return cudaSuccess;
    dim3 grid((unsigned)tiles, (unsigned)a.H, (unsigned)a.B);
    if (a.D == 128) {
        if (bf16)
            return launch_pdl(attn_simt_kernel<__nv_bfloat16, 128>, grid, dim3(128), 0, st, a);
        else
            return launch_pdl(attn_simt_kernel<float, 128>, grid, dim3(128), 0, st, a);
    } else {
        if (bf16)
            return launch_pdl(attn_simt_kernel<__nv_bfloat16, 64>, grid, dim3(128), 0, st, a);
        else
            return launch_pdl(attn_simt_kernel<float, 64>, grid, dim3(128), 0, st, a);
    }
    return cudaGetLastError();
}

}  // namespace msf
