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
// are a detached cache in Algorithm 1); they are computed key by key into a
// buffer of context-row gradients, and a gather kernel applies the adjoint
// of Subsample: a window token sums the rows that hold it as is and 1/s^2 of
// each pooled row that covers it (AVG; STRIDED: the pooled row whose
// top-left it is), over every group, in a fixed order, and rounds once.
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

// 8 consecutive elements (16-byte aligned) widened to fp32, in one or two
// 16-byte loads.
__device__ __forceinline__ void ld8(const __nv_bfloat16* p, float* x) {
    const uint4 v = __ldg(reinterpret_cast<const uint4*>(p));
    const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const float2 f = __bfloat1622float2(h[i]);
        x[2 * i] = f.x;
        x[2 * i + 1] = f.y;
    }
}
__device__ __forceinline__ void ld8(const float* p, float* x) {
    const float4 a = __ldg(reinterpret_cast<const float4*>(p));
    const float4 b = __ldg(reinterpret_cast<const float4*>(p + 4));
    x[0] = a.x, x[1] = a.y, x[2] = a.z, x[3] = a.w;
    x[4] = b.x, x[5] = b.y, x[6] = b.z, x[7] = b.w;
}

// E (2 or 4) consecutive fp32 values in one aligned vector load; E values
// stored as the dtype in one vector store.
template <int E>
__device__ __forceinline__ void ldE(const float* p, float* x) {
    if (E == 4) {
        const float4 v = __ldg(reinterpret_cast<const float4*>(p));
        x[0] = v.x, x[1] = v.y, x[2] = v.z, x[3] = v.w;
    } else {
        const float2 v = __ldg(reinterpret_cast<const float2*>(p));
        x[0] = v.x, x[1] = v.y;
    }
}
template <int E>
__device__ __forceinline__ void stE(float* p, const float* x) {
    if (E == 4)
        *reinterpret_cast<float4*>(p) = make_float4(x[0], x[1], x[2], x[3]);
    else
        *reinterpret_cast<float2*>(p) = make_float2(x[0], x[1]);
}
template <int E>
__device__ __forceinline__ void stE(__nv_bfloat16* p, const float* x) {
    if (E == 4) {
        __nv_bfloat162 a = __floats2bfloat162_rn(x[0], x[1]), b = __floats2bfloat162_rn(x[2], x[3]);
        *reinterpret_cast<uint2*>(p) =
            make_uint2(*reinterpret_cast<uint32_t*>(&a), *reinterpret_cast<uint32_t*>(&b));
    } else {
        *reinterpret_cast<__nv_bfloat162*>(p) = __floats2bfloat162_rn(x[0], x[1]);
    }
}

constexpr float kLog2e = 1.4426950408889634f;

// delta[b, h, t] = sum_d dout * out: a row of D elements is shared by D/8
// consecutive threads, each loading 8 elements of both tensors (one 16-byte
// vector each for bf16). One row per thread group: giving a warp several
// rows' loads at once (fewer, fuller warps) measured twice as slow.
template <typename T, int D>
__global__ void __launch_bounds__(256) bwd_delta_kernel(const BwdCommon c) {
    ptx::grid_dep_wait();
    ptx::grid_dep_launch();
    constexpr int kTpr = D / 8;
    const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    const long long w = idx / kTpr;
    const int part = (int)(idx % kTpr);
    const bool live = w < (long long)c.B * c.N * c.H;
    float acc = 0.f;
    int b = 0, t = 0, h = 0;
    if (live) {
        h = (int)(w % c.H);
        t = (int)((w / c.H) % c.N);
        b = (int)(w / ((long long)c.H * c.N));
        const size_t off = (size_t)b * c.bstride + (((size_t)t * c.H + h) * D + 8 * part) * sizeof(T);
        float go[8], o[8];
        ld8((const T*)(c.dout + off), go);
        ld8((const T*)(c.out + off), o);
#pragma unroll
        for (int i = 0; i < 8; ++i) acc = fmaf(go[i], o[i], acc);
    }
#pragma unroll
    for (int s = kTpr / 2; s > 0; s >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, s);
    if (live && part == 0) c.delta[((size_t)b * c.H + h) * c.N + t] = acc;
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

// dk, dv of one group's gradient rows: a block owns 32 rows of one segment of
// one (stream, head); four threads share a row. The group's queries stream
// through shared memory 32 at a time. Rows go to the context-gradient buffer.
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
    const size_t o = (((size_t)b * c.R + gs.crow0 + r) * c.H + h) * D;
#pragma unroll
    for (int e = 0; e < DP; ++e) {
        c.dk_ctx[o + 4 * e + cc] = dk[e] * c.scale;
        c.dv_ctx[o + 4 * e + cc] = dv[e];
    }
}

// dk_win, dv_win: one block per (stream, token); the token's rows of every
// head are contiguous (H * D values), so each thread owns 8 consecutive
// values of it and every entry's rows are whole coalesced spans, and the
// entries of the token's state are decoded per block, not per head. Entries
// are summed in their fixed order, two at a time with both entries' loads
// issued before the adds, and the sum is rounded once.
template <typename T, int D>
__global__ void __launch_bounds__(256) bwd_gather_kernel(const BwdCommon c, const GatherArgs g,
                                                         T* __restrict__ dk, T* __restrict__ dv) {
    ptx::grid_dep_wait();
    ptx::grid_dep_launch();
    const int t = (int)(blockIdx.x % (unsigned)c.N);
    const int b = (int)(blockIdx.x / (unsigned)c.N);
    int l = 0;
    while (l + 1 < g.T && t >= g.st_off[l + 1]) ++l;
    const int ne = g.n_ent[l];
    // context-gradient row and weight of entry k (row -1: a STRIDED entry
    // whose pooled row does not start at this token)
    auto decode = [&](int k, int& row, float& wgt) {
        row = -1;
        wgt = 0.f;
        if (k >= ne) return;
        const GatherEntry& en = g.e[l][k];
        if (en.sigma == 1) {
            row = en.crow0 + (t - en.dst0);
            wgt = 1.f;
            return;
        }
        const int s = en.sigma, loc = t - en.dst0;
        const int i = loc / en.src_gw, j = loc - i * en.src_gw;
        if (g.mode == MSF_RESAMPLE_STRIDED && (i % s || j % s)) return;
        row = en.crow0 + (i / s) * en.out_gw + j / s;
        wgt = g.mode == MSF_RESAMPLE_STRIDED ? 1.f : 1.0f / (float)(s * s);
    };
    const int HD = c.H * D;
    const size_t base = (size_t)b * c.R * HD;
    for (int x = 8 * (int)threadIdx.x; x < HD; x += 8 * (int)blockDim.x) {
        float ak[8], av[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) ak[e] = av[e] = 0.f;
        for (int k = 0; k < ne; k += 2) {
            int r0, r1;
            float w0, w1;
            decode(k, r0, w0);
            decode(k + 1, r1, w1);
            float k0[8], v0[8], k1[8], v1[8];
            if (r0 >= 0) {
                ld8(c.dk_ctx + base + (size_t)r0 * HD + x, k0);
                ld8(c.dv_ctx + base + (size_t)r0 * HD + x, v0);
            }
            if (r1 >= 0) {
                ld8(c.dk_ctx + base + (size_t)r1 * HD + x, k1);
                ld8(c.dv_ctx + base + (size_t)r1 * HD + x, v1);
            }
            if (r0 >= 0) {
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    ak[e] = fmaf(w0, k0[e], ak[e]);
                    av[e] = fmaf(w0, v0[e], av[e]);
                }
            }
            if (r1 >= 0) {
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    ak[e] = fmaf(w1, k1[e], ak[e]);
                    av[e] = fmaf(w1, v1[e], av[e]);
                }
            }
        }
        const size_t o = ((size_t)b * c.N + t) * HD + x;
        stE<4>(dk + o, ak);
        stE<4>(dk + o + 4, ak + 4);
        stE<4>(dv + o, av);
        stE<4>(dv + o + 4, av + 4);
    }
}

}  // namespace

cudaError_t launch_bwd_delta(const BwdCommon& c, bool bf16, cudaStream_t st) {
    const long long threads = (long long)c.B * c.N * c.H * (c.D / 8);
    dim3 grid((unsigned)((threads + 255) / 256));
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

cudaError_t launch_bwd_gather(const BwdCommon& c, const GatherArgs& g, void* dk, void* dv,
                              bool bf16, cudaStream_t st) {
    const long long tokens = (long long)c.B * c.N;
    if (tokens == 0) return cudaSuccess;
    // one thread per 8 values of a token's H * D, in whole warps, at most 256
    int threads = (c.H * c.D / 8 + 31) / 32 * 32;
    if (threads > 256) threads = 256;
    dim3 grid((unsigned)tokens);
    if (c.D == 128)
        return bf16 ? launch_pdl(bwd_gather_kernel<__nv_bfloat16, 128>, grid, dim3(threads), 0, st, c, g,
                                 (__nv_bfloat16*)dk, (__nv_bfloat16*)dv)
                    : launch_pdl(bwd_gather_kernel<float, 128>, grid, dim3(threads), 0, st, c, g, (float*)dk,
                                 (float*)dv);
    return bf16 ? launch_pdl(bwd_gather_kernel<__nv_bfloat16, 64>, grid, dim3(threads), 0, st, c, g,
                             (__nv_bfloat16*)dk, (__nv_bfloat16*)dv)
                : launch_pdl(bwd_gather_kernel<float, 64>, grid, dim3(threads), 0, st, c, g, (float*)dk,
                             (float*)dv);
}

}  // namespace msf
