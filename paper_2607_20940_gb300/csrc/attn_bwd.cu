// MSSA backward on CUDA cores (fp32 arithmetic, bf16 or fp32 storage).
//
// The gradient of Eq. 4 for a loss with dL/dO = dO, per query group g with
// context K_g, V_g (sink, history, window; pooled as in the forward):
//   P = exp(c q.k - lse)   (lse = the forward's row log-sum-exp)
//   delta_i = sum_d dO_i * O_i  (= sum_j P_ij dP_ij)
//   dS_ij = P_ij (dO_i . v_j - delta_i)
//   dq_i = c sum_j dS_ij k_j,  dk_j = c sum_i dS_ij q_i,  dv_j = sum_i P_ij dO_i
// dq is computed query by query over the whole context. dk, dv are needed
// only for context rows that come from the window (the sink and the history
// are a detached cache in Algorithm 1); they are computed key by key and sent
// back through the adjoint of Subsample into fp32 accumulators: a row kept as
// is adds to its window token, a pooled row adds 1/s^2 of itself to each of
// its s x s source tokens (AVG) or all of itself to the top-left one
// (STRIDED). Within one group every window token has a single writer; groups
// run one after another, so the sums are deterministic.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math.h>

#include "kernels.h"
#include "ptx.cuh"

namespace msf {
namespace {

template <typename T>
__device__ __forceinline__ float ld1(const T* p);
template <>
__device__ __forceinline__ float ld1(const float* p) { return *p; }
template <>
__device__ __forceinline__ float ld1(const __nv_bfloat16* p) { return __bfloat162float(*p); }
template <typename T>
__device__ __forceinline__ T st1(float x);
template <>
__device__ __forceinline__ float st1(float x) { return x; }
template <>
__device__ __forceinline__ __nv_bfloat16 st1(float x) { return __float2bfloat16_rn(x); }

constexpr float kLog2e = 1.4426950408889634f;

// delta[b, h, t] = sum_d dout * out; one warp per (b, t, h) row.
template <typename T, int D>
__global__ void __launch_bounds__(256) bwd_delta_kernel(const BwdCommon c) {
    ptx::grid_dep_wait();
    ptx::grid_dep_launch();
    const long long w = (long long)blockIdx.x * 8 + threadIdx.x / 32;
    const int lane = threadIdx.x % 32;
    if (w >= (long long)c.B * c.N * c.H) return;
    const int h = (int)(w % c.H);
    const int t = (int)((w / c.H) % c.N);
    const int b = (int)(w / ((long long)c.H * c.N));
    const size_t off = (size_t)b * c.bstride + ((size_t)t * c.H + h) * D * sizeof(T);
    const T* go = (const T*)(c.dout + off);
    const T* o = (const T*)(c.out + off);
    float acc = 0.f;
#pragma unroll
    for (int i = 0; i < D / 32; ++i) acc = fmaf(ld1<T>(go + 32 * i + lane), ld1<T>(o + 32 * i + lane), acc);
#pragma unroll
    for (int s = 16; s > 0; s >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, s);
    if (lane == 0) c.delta[((size_t)b * c.H + h) * c.N + t] = acc;
}

// dq: a block owns 32 queries of one (stream, head, group); four threads share
// a query and hold every fourth element of q, dO and dq.
template <typename T, int D>
__global__ void __launch_bounds__(128) bwd_dq_kernel(const BwdCommon c, const AttnArgs a, T* dq) {
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
    const int qi = threadIdx.x / 4, cc = threadIdx.x % 4;
    const int t = G.q_begin + tile * 32 + qi;
    const bool valid = t < G.q_end;
    const int tt = valid ? t : G.q_begin;
    const size_t row = (size_t)c.H * D * sizeof(T);
    const size_t qoff = (size_t)b * c.bstride + (size_t)tt * row + (size_t)h * D * sizeof(T);
    const T* qp = (const T*)(c.q + qoff);
    const T* gp = (const T*)(c.dout + qoff);
    float q[DP], g[DP], acc[DP];
#pragma unroll
    for (int i = 0; i < DP; ++i) {
        q[i] = ld1<T>(qp + 4 * i + cc) * c.scale_log2;
        g[i] = ld1<T>(gp + 4 * i + cc);
        acc[i] = 0.f;
    }
    const size_t rix = ((size_t)b * c.H + h) * c.N + tt;
    const float lse2 = c.lse[rix] * kLog2e;
    const float dl = c.delta[rix];

    for (int s = 0; s < G.n_seg; ++s) {
        const Segment& sg = G.seg[s];
        const char* kb = sg.k + (size_t)b * sg.bstride + (size_t)sg.row0 * row + (size_t)h * D * sizeof(T);
        const char* vb = sg.v + (size_t)b * sg.bstride + (size_t)sg.row0 * row + (size_t)h * D * sizeof(T);
        for (int kt = 0; kt < sg.len; kt += KT) {
            const int n = min(KT, sg.len - kt);
            __syncthreads();
            for (int e = threadIdx.x; e < n * D; e += blockDim.x) {
                const int key = e / D, d = e - key * D;
                Ks[key][d] = ld1<T>((const T*)(kb + (size_t)(kt + key) * row) + d);
                Vs[key][d] = ld1<T>((const T*)(vb + (size_t)(kt + key) * row) + d);
            }
            __syncthreads();
            for (int j = 0; j < n; ++j) {
                float sc = 0.f, dp = 0.f;
#pragma unroll
                for (int i = 0; i < DP; ++i) {
                    sc = fmaf(q[i], Ks[j][4 * i + cc], sc);
                    dp = fmaf(g[i], Vs[j][4 * i + cc], dp);
                }
                sc += __shfl_xor_sync(0xffffffffu, sc, 1);
                sc += __shfl_xor_sync(0xffffffffu, sc, 2);
                dp += __shfl_xor_sync(0xffffffffu, dp, 1);
                dp += __shfl_xor_sync(0xffffffffu, dp, 2);
                const float ds = exp2f(sc - lse2) * (dp - dl);
#pragma unroll
                for (int i = 0; i < DP; ++i) acc[i] = fmaf(ds, Ks[j][4 * i + cc], acc[i]);
            }
        }
    }
    if (!valid) return;
    T* o = (T*)((char*)dq + (size_t)b * c.bstride + (size_t)t * row) + (size_t)h * D;
#pragma unroll
    for (int i = 0; i < DP; ++i) o[4 * i + cc] = st1<T>(acc[i] * c.scale);
}

// Add one context row's fp32 gradient (this thread's DP elements) to the
// window accumulator through the adjoint of Subsample.
template <int D>
__device__ __forceinline__ void scatter_row(float* accb, const GradSeg& gs, int r, int h, int H,
                                            int cc, const float* val, int mode) {
    constexpr int DP = D / 4;
    auto add = [&](int token, float w) {
        float* dst = accb + ((size_t)token * H + h) * D;
#pragma unroll
        for (int i = 0; i < DP; ++i) dst[4 * i + cc] += w * val[i];
    };
    if (gs.sigma == 1) {
        add(gs.dst0 + r, 1.f);
        return;
    }
    const int s = gs.sigma;
    const int i = r / gs.out_gw, j = r - (r / gs.out_gw) * gs.out_gw;
    const int base = gs.dst0 + (s * i) * gs.src_gw + s * j;
    if (mode == MSF_RESAMPLE_STRIDED) {
        add(base, 1.f);
        return;
    }
    const float w = 1.0f / (float)(s * s);
    for (int dy = 0; dy < s; ++dy)
        for (int dx = 0; dx < s; ++dx) add(base + dy * gs.src_gw + dx, w);
}

// dk, dv of one group's gradient rows: a block owns 32 rows of one segment of
// one (stream, head); four threads share a row. The group's queries stream
// through shared memory 32 at a time.
template <typename T, int D>
__global__ void __launch_bounds__(128) bwd_dkdv_kernel(const BwdCommon c, const BwdGroup G) {
    ptx::grid_dep_wait();
    ptx::grid_dep_launch();
    constexpr int DP = D / 4;
    constexpr int QT = 32;
    __shared__ float Qs[QT][D];
    __shared__ float Gs[QT][D];
    __shared__ float Ls[QT], Ds[QT];
    int tile = blockIdx.x, si = 0;
    while (si < G.n_gseg) {
        int nt = (G.gseg[si].len + 31) / 32;
        if (tile < nt) break;
        tile -= nt;
        ++si;
    }
    if (si >= G.n_gseg) return;
    const GradSeg& gs = G.gseg[si];
    const int h = blockIdx.y, b = blockIdx.z;
    const int ki = threadIdx.x / 4, cc = threadIdx.x % 4;
    const int r = tile * 32 + ki;
    const bool valid = r < gs.len;
    const size_t row = (size_t)c.H * D * sizeof(T);
    const size_t koff = (size_t)b * gs.bstride + (size_t)(gs.row0 + (valid ? r : 0)) * row +
                        (size_t)h * D * sizeof(T);
    const T* kp = (const T*)(gs.k + koff);
    const T* vp = (const T*)(gs.v + koff);
    float k[DP], v[DP], dk[DP], dv[DP];
#pragma unroll
    for (int i = 0; i < DP; ++i) {
        k[i] = ld1<T>(kp + 4 * i + cc);
        v[i] = ld1<T>(vp + 4 * i + cc);
        dk[i] = dv[i] = 0.f;
    }
    for (int q0 = G.q_begin; q0 < G.q_end; q0 += QT) {
        const int n = min(QT, G.q_end - q0);
        __syncthreads();
        for (int e = threadIdx.x; e < n * D; e += blockDim.x) {
            const int qq = e / D, d = e - qq * D;
            const size_t off = (size_t)b * c.bstride + (size_t)(q0 + qq) * row + (size_t)h * D * sizeof(T);
            Qs[qq][d] = ld1<T>((const T*)(c.q + off) + d);
            Gs[qq][d] = ld1<T>((const T*)(c.dout + off) + d);
        }
        if (threadIdx.x < n) {
            const size_t rix = ((size_t)b * c.H + h) * c.N + q0 + threadIdx.x;
            Ls[threadIdx.x] = c.lse[rix] * kLog2e;
            Ds[threadIdx.x] = c.delta[rix];
        }
        __syncthreads();
        for (int i = 0; i < n; ++i) {
            float sc = 0.f, dp = 0.f;
#pragma unroll
            for (int e = 0; e < DP; ++e) {
                sc = fmaf(k[e], Qs[i][4 * e + cc], sc);
                dp = fmaf(v[e], Gs[i][4 * e + cc], dp);
            }
            sc += __shfl_xor_sync(0xffffffffu, sc, 1);
            sc += __shfl_xor_sync(0xffffffffu, sc, 2);
            dp += __shfl_xor_sync(0xffffffffu, dp, 1);
            dp += __shfl_xor_sync(0xffffffffu, dp, 2);
            const float p = exp2f(sc * c.scale_log2 - Ls[i]);
            const float ds = p * (dp - Ds[i]);
#pragma unroll
            for (int e = 0; e < DP; ++e) {
                dv[e] = fmaf(p, Gs[i][4 * e + cc], dv[e]);
                dk[e] = fmaf(ds, Qs[i][4 * e + cc], dk[e]);
            }
        }
    }
    if (!valid) return;
#pragma unroll
    for (int e = 0; e < DP; ++e) dk[e] *= c.scale;
    const size_t accb = (size_t)b * c.N * c.H * D;
    scatter_row<D>(c.dk_acc + accb, gs, r, h, c.H, cc, dk, c.mode);
    scatter_row<D>(c.dv_acc + accb, gs, r, h, c.H, cc, dv, c.mode);
}

template <typename T>
__global__ void __launch_bounds__(256) bwd_cast_kernel(const float* __restrict__ a,
                                                        const float* __restrict__ bsrc,
                                                        T* __restrict__ oa, T* __restrict__ ob,
                                                        long long n4) {
    ptx::grid_dep_wait();
    ptx::grid_dep_launch();
    const long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= n4) return;
    const float4 x = reinterpret_cast<const float4*>(a)[i];
    const float4 y = reinterpret_cast<const float4*>(bsrc)[i];
    oa[4 * i] = st1<T>(x.x);
    oa[4 * i + 1] = st1<T>(x.y);
    oa[4 * i + 2] = st1<T>(x.z);
    oa[4 * i + 3] = st1<T>(x.w);
    ob[4 * i] = st1<T>(y.x);
    ob[4 * i + 1] = st1<T>(y.y);
    ob[4 * i + 2] = st1<T>(y.z);
    ob[4 * i + 3] = st1<T>(y.w);
}

}  // namespace

cudaError_t launch_bwd_delta(const BwdCommon& c, bool bf16, cudaStream_t st) {
    const long long rows = (long long)c.B * c.N * c.H;
    dim3 grid((unsigned)((rows + 7) / 8));
    if (c.D == 128)
        return bf16 ? launch_pdl(bwd_delta_kernel<__nv_bfloat16, 128>, grid, dim3(256), 0, st, c)
                    : launch_pdl(bwd_delta_kernel<float, 128>, grid, dim3(256), 0, st, c);
    return bf16 ? launch_pdl(bwd_delta_kernel<__nv_bfloat16, 64>, grid, dim3(256), 0, st, c)
                : launch_pdl(bwd_delta_kernel<float, 64>, grid, dim3(256), 0, st, c);
}

cudaError_t launch_bwd_dq_simt(const BwdCommon& c, const AttnArgs& a, void* dq, bool bf16,
                               cudaStream_t st) {
    int tiles = 0;
    for (int gi = 0; gi < a.n_groups; ++gi) tiles += (a.g[gi].q_end - a.g[gi].q_begin + 31) / 32;
    if (tiles == 0) return cudaSuccess;
    dim3 grid((unsigned)tiles, (unsigned)c.H, (unsigned)c.B);
    if (c.D == 128)
        return bf16 ? launch_pdl(bwd_dq_kernel<__nv_bfloat16, 128>, grid, dim3(128), 0, st, c, a,
                                 (__nv_bfloat16*)dq)
                    : launch_pdl(bwd_dq_kernel<float, 128>, grid, dim3(128), 0, st, c, a, (float*)dq);
    return bf16 ? launch_pdl(bwd_dq_kernel<__nv_bfloat16, 64>, grid, dim3(128), 0, st, c, a,
                             (__nv_bfloat16*)dq)
                : launch_pdl(bwd_dq_kernel<float, 64>, grid, dim3(128), 0, st, c, a, (float*)dq);
}

cudaError_t launch_bwd_dkdv_simt(const BwdCommon& c, const BwdGroup& g, bool bf16,
                                 cudaStream_t st) {
    int tiles = 0;
    for (int s = 0; s < g.n_gseg; ++s) tiles += (g.gseg[s].len + 31) / 32;
    if (tiles == 0 || g.q_end <= g.q_begin) return cudaSuccess;
    dim3 grid((unsigned)tiles, (unsigned)c.H, (unsigned)c.B);
    if (c.D == 128)
        return bf16 ? launch_pdl(bwd_dkdv_kernel<__nv_bfloat16, 128>, grid, dim3(128), 0, st, c, g)
                    : launch_pdl(bwd_dkdv_kernel<float, 128>, grid, dim3(128), 0, st, c, g);
    return bf16 ? launch_pdl(bwd_dkdv_kernel<__nv_bfloat16, 64>, grid, dim3(128), 0, st, c, g)
                : launch_pdl(bwd_dkdv_kernel<float, 64>, grid, dim3(128), 0, st, c, g);
}

cudaError_t launch_bwd_cast(const BwdCommon& c, void* dk, void* dv, bool bf16, cudaStream_t st) {
    const long long n4 = (long long)c.B * c.N * c.H * c.D / 4;
    dim3 grid((unsigned)((n4 + 255) / 256));
    if (bf16)
        return launch_pdl(bwd_cast_kernel<__nv_bfloat16>, grid, dim3(256), 0, st, (const float*)c.dk_acc,
                          (const float*)c.dv_acc, (__nv_bfloat16*)dk, (__nv_bfloat16*)dv, n4);
    return launch_pdl(bwd_cast_kernel<float>, grid, dim3(256), 0, st, (const float*)c.dk_acc,
                      (const float*)c.dv_acc, (float*)dk, (float*)dv, n4);
}

}  // namespace msf
