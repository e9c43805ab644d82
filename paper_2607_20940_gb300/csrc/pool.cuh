// K/V pyramid pooling (Eq. 4's Subsample) as device functions, shared by the
// pool kernel and the fused MSP embedding + pyramid launch.
#pragma once

#include <cuda_bf16.h>
#include <stdint.h>

#include "kernels.h"

namespace msf {

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

// One thread's share of a pool batch: the vector pair `idx` (token idx /
// (row_vecs/2), vector pair idx % (row_vecs/2)) of job `job`, stream b.
template <typename T>
__device__ __forceinline__ void pool_task(const PoolBatch& jobs, int job, int b, int idx) {
    const PoolJob& jb = jobs.j[job];
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

}  // namespace msf
