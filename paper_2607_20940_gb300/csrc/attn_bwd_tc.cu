// MSSA backward on the sm_103a tensor cores (bf16 operands, fp32 accumulation).
//
// Same mathematics as the CUDA-core backward (attn_bwd.cu): with the
// forward's row log-sum-exp, P = exp(c S - lse) is rebuilt tile by tile and
//   dS = P * (dP - delta),  dP = dO V^T,  delta = rowsum(dO * O)
//   dQ = c dS K,  dK = c dS^T Q,  dV = P^T dO.
// Two kernels, neither needs atomics:
//
// bwd_dq_tc_kernel: one CTA per 128-row query tile of one (stream, head,
//   group). It walks the group's whole context (sink, history or pyramid
//   part, window suffix) in 128-row K/V tiles:
//     S = Q K^T (SS), dP = dO V^T (SS)              -> TMEM
//     softmax warps: P, dS (bf16, over S's columns)  -> TMEM
//     dQ += dS K (TS, K read MN-major)              -> TMEM
//   then scales dQ by c and stores it.
// bwd_dkdv_tc_kernel: one CTA per 128-row tile of context rows that come
//   from the window (one group per launch). It walks the group's queries in
//   128-row tiles:
//     S^T = K Q^T (SS), dP^T = V dO^T (SS)            -> TMEM (lanes = keys)
//     softmax warps: P^T, dS^T (bf16, over S^T/dP^T)  -> TMEM
//     dV += P^T dO (TS), dK += dS^T Q (TS)           -> TMEM
//   then sends c dK and dV through the adjoint of Subsample into the fp32
//   window accumulators; each window token has one writer per launch.
//
// Roles (256 threads): warp 0 TMA producer, warp 1 MMA issuer (warp-wide
// loop, one elected lane issues), warp 2 TMEM allocation, warps 4-7 one
// thread per TMEM lane (query row or key row). TMEM columns: S [0,128),
// dP [128,256), then dQ (or dV, dK) from 256. The tensor pipe executes MMAs
// in issue order, so an MMA that overwrites S or dP never overtakes the MMA
// that reads the bf16 P or dS stored there. Every wait is bounded.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math.h>
#include <string.h>

#include "attn_bwd_tc.h"
#include "attn_tc.h"
#include "ptx.cuh"

namespace msf {
namespace {

constexpr int kBM = 128;       // rows of every Q / dO / K / V tile
constexpr int kThreads = 256;  // 8 warps
constexpr long long kWaitLimit = 2000000000LL;  // ~1 s of SM clock
constexpr float kLog2e = 1.4426950408889634f;

struct BSeg {
    int map, row0, len, tile0;
};
struct BGroupQ {
    int q_begin, q_end;
    int n_qt;       // 128-row query tiles
    int item_base;  // first item of this group
    int n_seg, n_tiles;
    BSeg seg[kMaxSeg];
};
struct BGrad {
    int map, row0, len, kt0;  // row0 relative to the map; kt0 = first key tile of the run
    int sigma, dst0, src_gw, out_gw;
};
struct BwdTcParams {
    int H, B, N;
    float scale, scale_log2;
    const float* lse;
    const float* delta;
    __nv_bfloat16* dq;
    float* dk_acc;
    float* dv_acc;
    int mode;
    unsigned int* status;
    long long wait_limit;
    // bwd_dq_tc_kernel
    int n_groups;
    BGroupQ g[MSF_MAX_GROUPS];
    // bwd_dkdv_tc_kernel (one group)
    int q_begin, q_end, n_qt, n_grad;
    BGrad gr[kMaxGradSeg];
};
struct BwdMaps {
    CUtensorMap q, dout;
    CUtensorMap k[kNumMaps];
    CUtensorMap v[kNumMaps];
};

template <int D>
struct BCfg {
    static constexpr int kTile = kBM * D * 2;
    // Q, dO and two K/V stages (dQ kernel) or K, V and two Q/dO stages (dK/dV
    // kernel); at least 120 KB so that one CTA (and one 512-column TMEM
    // allocation) sits on an SM.
    static constexpr int kSmem = 6 * kTile + 1024 > 120 * 1024 ? 6 * kTile + 1024 : 120 * 1024;
};

__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// K-step offset (16-byte units) inside a K-major SW128 tile of 128 rows.
__device__ __forceinline__ uint64_t kmajor_step(int kk) {
    constexpr int kChunk = kBM * 128;
    return (uint64_t)(((kk / 4) * kChunk + (kk % 4) * 32) >> 4);
}

// 128 rows x D of a [B, rows, H, D] tensor: D/64 swizzled boxes.
template <int D>
__device__ __forceinline__ void load_tile(unsigned char* dst, const CUtensorMap* m, uint64_t* bar,
                                          int h, int row, int b) {
#pragma unroll
    for (int c = 0; c < D / 64; ++c) ptx::tma_load_4d(dst + c * (kBM * 128), m, bar, c * 64, h, row, b);
}

// ============================================================== dQ kernel

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    bwd_dq_tc_kernel(const __grid_constant__ BwdMaps maps, const __grid_constant__ BwdTcParams p) {
    using C = BCfg<D>;
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    unsigned char* smem = (unsigned char*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    unsigned char* sQ = smem;
    unsigned char* sG = smem + C::kTile;       // dO
    unsigned char* sK = smem + 2 * C::kTile;   // [2]
    unsigned char* sV = smem + 4 * C::kTile;   // [2]

    __shared__ uint64_t qg_full, kv_full[2], kv_empty[2], st_full, ds_full, dq_full, drain_bar;
    __shared__ uint32_t tmem_base_sh;
    __shared__ int abort_flag;

    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    int gi = 0;
    while (gi + 1 < p.n_groups && (int)blockIdx.x >= p.g[gi + 1].item_base) ++gi;
    const BGroupQ& G = p.g[gi];
    const int local = (int)blockIdx.x - G.item_base;
    const int qt = local % G.n_qt;
    const int h = (local / G.n_qt) % p.H;
    const int b = local / (G.n_qt * p.H);
    const int q_row0 = G.q_begin + qt * kBM;
    const int n = G.n_tiles;

    if (threadIdx.x == 0) {
        abort_flag = 0;
        ptx::mbar_init(&qg_full, 1);
        for (int s = 0; s < 2; ++s) {
            ptx::mbar_init(&kv_full[s], 1);
            ptx::mbar_init(&kv_empty[s], 1);
        }
        ptx::mbar_init(&st_full, 1);
        ptx::mbar_init(&ds_full, 4);
        ptx::mbar_init(&dq_full, 1);
        ptx::mbar_init(&drain_bar, 1);
        ptx::fence_mbar_init();
    }
    if (warp == 2) {
        ptx::tmem_alloc(&tmem_base_sh, 512);
        ptx::tmem_relinquish();
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tbase = tmem_base_sh;
    volatile int* abort_p = &abort_flag;
    volatile int never = 0;
    ptx::grid_dep_wait();
    ptx::grid_dep_launch();

    auto tile_of = [&](int u, int& seg, int& row, int& valid) {
        int s = 0;
        while (s < G.n_seg - 1 && u >= G.seg[s + 1].tile0) ++s;
        const int kt = u - G.seg[s].tile0;
        seg = s;
        row = G.seg[s].row0 + kt * kBM;
        valid = min(kBM, G.seg[s].len - kt * kBM);
    };

    if (warp == 0) {
        // ============================ TMA producer ============================
        if (lane == 0) {
            bool ok = true;
            ptx::mbar_arrive_expect_tx(&qg_full, 2 * C::kTile);
            load_tile<D>(sQ, &maps.q, &qg_full, h, q_row0, b);
            load_tile<D>(sG, &maps.dout, &qg_full, h, q_row0, b);
            int j = 0;
            for (; j < n; ++j) {
                int seg, row, valid;
                tile_of(j, seg, row, valid);
                const int st = j & 1;
                if (!ptx::mbar_wait_bounded(&kv_empty[st], (uint32_t)(((j >> 1) & 1) ^ 1), abort_p,
                                            p.wait_limit)) {
                    ok = false;
                    break;
                }
                ptx::mbar_arrive_expect_tx(&kv_full[st], 2 * C::kTile);
                load_tile<D>(sK + st * C::kTile, &maps.k[G.seg[seg].map], &kv_full[st], h, row, b);
                load_tile<D>(sV + st * C::kTile, &maps.v[G.seg[seg].map], &kv_full[st], h, row, b);
            }
            if (!ok) {
                ptx::mbar_wait_bounded(&qg_full, 0, &never, kWaitLimit);
                for (int jj = (j > 2 ? j - 2 : 0); jj < j; ++jj)
                    ptx::mbar_wait_bounded(&kv_full[jj & 1], (uint32_t)((jj >> 1) & 1), &never, kWaitLimit);
                atomicOr(p.status, kDevTimeout);
            }
        }
    } else if (warp == 1) {
        // ============================= MMA issuer =============================
        constexpr uint32_t idS = ptx::idesc_bf16(kBM, kBM, false, false);
        constexpr uint32_t idQ = ptx::idesc_bf16(kBM, D, false, true);
        constexpr uint64_t kTileDesc = (uint64_t)(C::kTile >> 4);
        const uint64_t q_desc = ptx::sdesc_sw128(ptx::smem_u32(sQ), 16, 1024);
        const uint64_t g_desc = ptx::sdesc_sw128(ptx::smem_u32(sG), 16, 1024);
        const uint64_t k_desc = ptx::sdesc_sw128(ptx::smem_u32(sK), 16, 1024);
        const uint64_t v_desc = ptx::sdesc_sw128(ptx::smem_u32(sV), 16, 1024);
        const uint64_t kmn_desc = ptx::sdesc_sw128(ptx::smem_u32(sK), kBM * 128, 1024);
        auto wait_all = [&](uint64_t* bar, uint32_t parity) {
            const bool r = ptx::mbar_wait_bounded(bar, parity, abort_p, p.wait_limit);
            return __all_sync(0xffffffffu, r);
        };
        bool ok = wait_all(&qg_full, 0);
        for (int j = 0; j < n && ok; ++j) {
            const int st = j & 1;
            ok = wait_all(&kv_full[st], (uint32_t)((j >> 1) & 1));
            if (!ok) break;
            ptx::tc_fence_after();
            if (ptx::elect_one_sync()) {
                const uint64_t kd = k_desc + (uint64_t)st * kTileDesc;
                const uint64_t vd = v_desc + (uint64_t)st * kTileDesc;
#pragma unroll
                for (int kk = 0; kk < D / 16; ++kk)
                    ptx::mma_ss(tbase, q_desc + kmajor_step(kk), kd + kmajor_step(kk), idS, kk > 0 ? 1u : 0u);
#pragma unroll
                for (int kk = 0; kk < D / 16; ++kk)
                    ptx::mma_ss(tbase + 128, g_desc + kmajor_step(kk), vd + kmajor_step(kk), idS,
                                kk > 0 ? 1u : 0u);
                ptx::mma_commit(&st_full);
            }
            __syncwarp();
            ok = wait_all(&ds_full, (uint32_t)(j & 1));
            if (!ok) break;
            ptx::tc_fence_after();
            if (ptx::elect_one_sync()) {
                const uint64_t kd = kmn_desc + (uint64_t)st * kTileDesc;
#pragma unroll
                for (int kk = 0; kk < kBM / 16; ++kk)
                    ptx::mma_ts(tbase + 256, tbase + kk * 8, kd + (uint64_t)(kk * (2048 >> 4)), idQ,
                                (j > 0 || kk > 0) ? 1u : 0u);
                ptx::mma_commit(&kv_empty[st]);
                if (j + 1 == n) ptx::mma_commit(&dq_full);
            }
            __syncwarp();
        }
        if (!ok) {
            if (ptx::elect_one_sync()) ptx::mma_commit(&drain_bar);
            __syncwarp();
            ptx::mbar_wait_bounded(&drain_bar, 0, &never, kWaitLimit);
            if (lane == 0) atomicOr(p.status, kDevTimeout);
        }
    } else if (warp >= 4) {
        // ===================== softmax: one thread per query row =====================
        const int wq = warp % 4;
        const int r = wq * 32 + lane;
        const uint32_t lane_off = (uint32_t)(wq * 32) << 16;
        const uint32_t tS = tbase + lane_off, tP = tbase + 128 + lane_off, tQ = tbase + 256 + lane_off;
        const int q = q_row0 + r;
        const bool qv = q < G.q_end;
        const size_t rix = ((size_t)b * p.H + h) * p.N + (qv ? q : 0);
        const float nl = qv ? -p.lse[rix] * kLog2e : -INFINITY;  // -lse in log2 units
        const float dl = qv ? p.delta[rix] : 0.f;
        const float sl2 = p.scale_log2;
        bool ok = true;
        for (int j = 0; j < n && ok; ++j) {
            int seg, row, valid;
            tile_of(j, seg, row, valid);
            ok = __all_sync(0xffffffffu, ptx::mbar_wait_bounded(&st_full, (uint32_t)(j & 1), abort_p,
                                                                p.wait_limit));
            if (!ok) break;
            ptx::tc_fence_after();
#pragma unroll
            for (int c4 = 0; c4 < 4; ++c4) {
                uint32_t s[32], dp[32];
                ptx::tmem_ld32(tS + 32 * c4, s);
                ptx::tmem_ld32(tP + 32 * c4, dp);
                ptx::tmem_wait_ld();
                uint32_t pk[16];
#pragma unroll
                for (int e = 0; e < 16; ++e) {
                    const int c0 = 32 * c4 + 2 * e;
                    float p0 = ex2(fmaf(__uint_as_float(s[2 * e]), sl2, nl));
                    float p1 = ex2(fmaf(__uint_as_float(s[2 * e + 1]), sl2, nl));
                    if (c0 >= valid) p0 = 0.f;
                    if (c0 + 1 >= valid) p1 = 0.f;
                    pk[e] = ptx::pack_bf16(p0 * (__uint_as_float(dp[2 * e]) - dl),
                                           p1 * (__uint_as_float(dp[2 * e + 1]) - dl));
                }
                ptx::tmem_st16(tS + 16 * c4, pk);
            }
            ptx::tmem_wait_st();
            ptx::tc_fence_before();
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&ds_full);
        }
        if (ok) ok = __all_sync(0xffffffffu, ptx::mbar_wait_bounded(&dq_full, 0, abort_p, p.wait_limit));
        if (ok) {
            ptx::tc_fence_after();
            __nv_bfloat16* dst = p.dq + (((size_t)b * p.N + (qv ? q : 0)) * p.H + h) * D;
#pragma unroll
            for (int c = 0; c < D / 32; ++c) {
                uint32_t o[32];
                ptx::tmem_ld32(tQ + 32 * c, o);
                ptx::tmem_wait_ld();
                uint32_t pk[16];
#pragma unroll
                for (int e = 0; e < 16; ++e)
                    pk[e] = ptx::pack_bf16(__uint_as_float(o[2 * e]) * p.scale,
                                           __uint_as_float(o[2 * e + 1]) * p.scale);
                if (qv) {
                    uint4* d4 = reinterpret_cast<uint4*>(dst + 32 * c);
#pragma unroll
                    for (int e = 0; e < 4; ++e)
                        d4[e] = make_uint4(pk[4 * e], pk[4 * e + 1], pk[4 * e + 2], pk[4 * e + 3]);
                }
            }
        }
        if (!ok && lane == 0) atomicOr(p.status, kDevTimeout);
    }

    ptx::tc_fence_before();
    __syncthreads();
    if (warp == 2) {
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tbase, 512);
    }
}

// ============================================================ dK/dV kernel

// Add one key row's gradient (D fp32 values) to the window accumulator
// through the adjoint of Subsample.
template <int D>
__device__ __forceinline__ void scatter_row_tc(float* accb, const BGrad& gr, int rr, int h, int H,
                                               const float* val, int mode) {
    auto add = [&](int token, float w) {
        float4* dst = reinterpret_cast<float4*>(accb + ((size_t)token * H + h) * D);
#pragma unroll
        for (int i = 0; i < D / 4; ++i) {
            float4 x = dst[i];
            x.x = fmaf(w, val[4 * i], x.x);
            x.y = fmaf(w, val[4 * i + 1], x.y);
            x.z = fmaf(w, val[4 * i + 2], x.z);
            x.w = fmaf(w, val[4 * i + 3], x.w);
            dst[i] = x;
        }
    };
    if (gr.sigma == 1) {
        add(gr.dst0 + rr, 1.f);
        return;
    }
    const int s = gr.sigma;
    const int i = rr / gr.out_gw, j = rr - (rr / gr.out_gw) * gr.out_gw;
    const int base = gr.dst0 + (s * i) * gr.src_gw + s * j;
    if (mode == MSF_RESAMPLE_STRIDED) {
        add(base, 1.f);
        return;
    }
    const float w = 1.0f / (float)(s * s);
    for (int dy = 0; dy < s; ++dy)
        for (int dx = 0; dx < s; ++dx) add(base + dy * gr.src_gw + dx, w);
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    bwd_dkdv_tc_kernel(const __grid_constant__ BwdMaps maps, const __grid_constant__ BwdTcParams p) {
    using C = BCfg<D>;
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    unsigned char* smem = (unsigned char*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    unsigned char* sK = smem;
    unsigned char* sV = smem + C::kTile;
    unsigned char* sQ = smem + 2 * C::kTile;   // [2]
    unsigned char* sG = smem + 4 * C::kTile;   // [2] dO

    __shared__ uint64_t kv_full, qg_full[2], qg_empty[2], st_full, pds_full, kv_done, drain_bar;
    __shared__ uint32_t tmem_base_sh;
    __shared__ int abort_flag;
    __shared__ float sL[2][kBM], sD[2][kBM];

    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const int n_kt_items = p.gr[p.n_grad - 1].kt0 + (p.gr[p.n_grad - 1].len + kBM - 1) / kBM;
    const int kt_all = (int)blockIdx.x % n_kt_items;
    const int h = ((int)blockIdx.x / n_kt_items) % p.H;
    const int b = (int)blockIdx.x / (n_kt_items * p.H);
    int gsi = 0;
    while (gsi + 1 < p.n_grad && kt_all >= p.gr[gsi + 1].kt0) ++gsi;
    const BGrad& gr = p.gr[gsi];
    const int kt = kt_all - gr.kt0;
    const int key_row = gr.row0 + kt * kBM;
    const int valid_keys = min(kBM, gr.len - kt * kBM);
    const int nq = p.n_qt;

    if (threadIdx.x == 0) {
        abort_flag = 0;
        ptx::mbar_init(&kv_full, 1);
        for (int s = 0; s < 2; ++s) {
            ptx::mbar_init(&qg_full[s], 1);
            ptx::mbar_init(&qg_empty[s], 1);
        }
        ptx::mbar_init(&st_full, 1);
        ptx::mbar_init(&pds_full, 4);
        ptx::mbar_init(&kv_done, 1);
        ptx::mbar_init(&drain_bar, 1);
        ptx::fence_mbar_init();
    }
    if (warp == 2) {
        ptx::tmem_alloc(&tmem_base_sh, 512);
        ptx::tmem_relinquish();
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tbase = tmem_base_sh;
    volatile int* abort_p = &abort_flag;
    volatile int never = 0;
    ptx::grid_dep_wait();
    ptx::grid_dep_launch();

    if (warp == 0) {
        // ============================ TMA producer ============================
        if (lane == 0) {
            bool ok = true;
            ptx::mbar_arrive_expect_tx(&kv_full, 2 * C::kTile);
            load_tile<D>(sK, &maps.k[gr.map], &kv_full, h, key_row, b);
            load_tile<D>(sV, &maps.v[gr.map], &kv_full, h, key_row, b);
            int i = 0;
            for (; i < nq; ++i) {
                const int st = i & 1;
                if (!ptx::mbar_wait_bounded(&qg_empty[st], (uint32_t)(((i >> 1) & 1) ^ 1), abort_p,
                                            p.wait_limit)) {
                    ok = false;
                    break;
                }
                ptx::mbar_arrive_expect_tx(&qg_full[st], 2 * C::kTile);
                load_tile<D>(sQ + st * C::kTile, &maps.q, &qg_full[st], h, p.q_begin + i * kBM, b);
                load_tile<D>(sG + st * C::kTile, &maps.dout, &qg_full[st], h, p.q_begin + i * kBM, b);
            }
            if (!ok) {
                ptx::mbar_wait_bounded(&kv_full, 0, &never, kWaitLimit);
                for (int ii = (i > 2 ? i - 2 : 0); ii < i; ++ii)
                    ptx::mbar_wait_bounded(&qg_full[ii & 1], (uint32_t)((ii >> 1) & 1), &never, kWaitLimit);
                atomicOr(p.status, kDevTimeout);
            }
        }
    } else if (warp == 1) {
        // ============================= MMA issuer =============================
        constexpr uint32_t idS = ptx::idesc_bf16(kBM, kBM, false, false);
        constexpr uint32_t idO = ptx::idesc_bf16(kBM, D, false, true);
        constexpr uint64_t kTileDesc = (uint64_t)(C::kTile >> 4);
        const uint64_t k_desc = ptx::sdesc_sw128(ptx::smem_u32(sK), 16, 1024);
        const uint64_t v_desc = ptx::sdesc_sw128(ptx::smem_u32(sV), 16, 1024);
        const uint64_t q_desc = ptx::sdesc_sw128(ptx::smem_u32(sQ), 16, 1024);
        const uint64_t g_desc = ptx::sdesc_sw128(ptx::smem_u32(sG), 16, 1024);
        const uint64_t qmn_desc = ptx::sdesc_sw128(ptx::smem_u32(sQ), kBM * 128, 1024);
        const uint64_t gmn_desc = ptx::sdesc_sw128(ptx::smem_u32(sG), kBM * 128, 1024);
        auto wait_all = [&](uint64_t* bar, uint32_t parity) {
            const bool r = ptx::mbar_wait_bounded(bar, parity, abort_p, p.wait_limit);
            return __all_sync(0xffffffffu, r);
        };
        bool ok = wait_all(&kv_full, 0);
        for (int i = 0; i < nq && ok; ++i) {
            const int st = i & 1;
            ok = wait_all(&qg_full[st], (uint32_t)((i >> 1) & 1));
            if (!ok) break;
            ptx::tc_fence_after();
            if (ptx::elect_one_sync()) {
                const uint64_t qd = q_desc + (uint64_t)st * kTileDesc;
                const uint64_t gd = g_desc + (uint64_t)st * kTileDesc;
#pragma unroll
                for (int kk = 0; kk < D / 16; ++kk)
                    ptx::mma_ss(tbase, k_desc + kmajor_step(kk), qd + kmajor_step(kk), idS, kk > 0 ? 1u : 0u);
#pragma unroll
                for (int kk = 0; kk < D / 16; ++kk)
                    ptx::mma_ss(tbase + 128, v_desc + kmajor_step(kk), gd + kmajor_step(kk), idS,
                                kk > 0 ? 1u : 0u);
                ptx::mma_commit(&st_full);
            }
            __syncwarp();
            ok = wait_all(&pds_full, (uint32_t)(i & 1));
            if (!ok) break;
            ptx::tc_fence_after();
            if (ptx::elect_one_sync()) {
                const uint64_t gd = gmn_desc + (uint64_t)st * kTileDesc;
                const uint64_t qd = qmn_desc + (uint64_t)st * kTileDesc;
#pragma unroll
                for (int kk = 0; kk < kBM / 16; ++kk)
                    ptx::mma_ts(tbase + 256, tbase + kk * 8, gd + (uint64_t)(kk * (2048 >> 4)), idO,
                                (i > 0 || kk > 0) ? 1u : 0u);
#pragma unroll
                for (int kk = 0; kk < kBM / 16; ++kk)
                    ptx::mma_ts(tbase + 256 + D, tbase + 128 + kk * 8, qd + (uint64_t)(kk * (2048 >> 4)),
                                idO, (i > 0 || kk > 0) ? 1u : 0u);
                ptx::mma_commit(&qg_empty[st]);
                if (i + 1 == nq) ptx::mma_commit(&kv_done);
            }
            __syncwarp();
        }
        if (!ok) {
            if (ptx::elect_one_sync()) ptx::mma_commit(&drain_bar);
            __syncwarp();
            ptx::mbar_wait_bounded(&drain_bar, 0, &never, kWaitLimit);
            if (lane == 0) atomicOr(p.status, kDevTimeout);
        }
    } else if (warp >= 4) {
        // ====================== softmax: one thread per key row ======================
        const int wq = warp % 4;
        const int r = wq * 32 + lane;
        const uint32_t lane_off = (uint32_t)(wq * 32) << 16;
        const uint32_t tS = tbase + lane_off, tP = tbase + 128 + lane_off;
        const float sl2 = p.scale_log2;
        bool ok = true;
        for (int i = 0; i < nq && ok; ++i) {
            // this tile's per-query statistics, shared by the 128 key rows
            {
                const int q = p.q_begin + i * kBM + r;
                const bool qv = q < p.q_end;
                const size_t rix = ((size_t)b * p.H + h) * p.N + (qv ? q : 0);
                sL[i & 1][r] = qv ? -p.lse[rix] * kLog2e : -INFINITY;
                sD[i & 1][r] = qv ? p.delta[rix] : 0.f;
            }
            ptx::named_bar_sync(1, 128);
            const float* L = sL[i & 1];
            const float* Dl = sD[i & 1];
            ok = __all_sync(0xffffffffu, ptx::mbar_wait_bounded(&st_full, (uint32_t)(i & 1), abort_p,
                                                                p.wait_limit));
            if (!ok) break;
            ptx::tc_fence_after();
#pragma unroll
            for (int c4 = 0; c4 < 4; ++c4) {
                uint32_t s[32], dp[32];
                ptx::tmem_ld32(tS + 32 * c4, s);
                ptx::tmem_ld32(tP + 32 * c4, dp);
                ptx::tmem_wait_ld();
                uint32_t pp[16], pd[16];
#pragma unroll
                for (int e = 0; e < 16; ++e) {
                    const int c0 = 32 * c4 + 2 * e;
                    const float p0 = ex2(fmaf(__uint_as_float(s[2 * e]), sl2, L[c0]));
                    const float p1 = ex2(fmaf(__uint_as_float(s[2 * e + 1]), sl2, L[c0 + 1]));
                    pp[e] = ptx::pack_bf16(p0, p1);
                    pd[e] = ptx::pack_bf16(p0 * (__uint_as_float(dp[2 * e]) - Dl[c0]),
                                           p1 * (__uint_as_float(dp[2 * e + 1]) - Dl[c0 + 1]));
                }
                ptx::tmem_st16(tS + 16 * c4, pp);
                ptx::tmem_st16(tP + 16 * c4, pd);
            }
            ptx::tmem_wait_st();
            ptx::tc_fence_before();
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&pds_full);
        }
        if (ok) ok = __all_sync(0xffffffffu, ptx::mbar_wait_bounded(&kv_done, 0, abort_p, p.wait_limit));
        if (ok) {
            ptx::tc_fence_after();
            const bool kv = r < valid_keys;
            const size_t accb = (size_t)b * p.N * p.H * D;
            const int rr = kt * kBM + r;  // row inside the gradient run
            for (int which = 0; which < 2; ++which) {
                float val[D];
#pragma unroll
                for (int c = 0; c < D / 32; ++c) {
                    uint32_t o[32];
                    ptx::tmem_ld32(tbase + 256 + (which == 0 ? D : 0) + 32 * c + lane_off, o);
                    ptx::tmem_wait_ld();
#pragma unroll
                    for (int e = 0; e < 32; ++e)
                        val[32 * c + e] = __uint_as_float(o[e]) * (which == 0 ? p.scale : 1.f);
                }
                if (kv)
                    scatter_row_tc<D>((which == 0 ? p.dk_acc : p.dv_acc) + accb, gr, rr, h, p.H, val, p.mode);
            }
        }
        if (!ok && lane == 0) atomicOr(p.status, kDevTimeout);
    }

    ptx::tc_fence_before();
    __syncthreads();
    if (warp == 2) {
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tbase, 512);
    }
}

bool encode_all(BwdMaps& m, const Plan& P, const BwdTcInput& in) {
    const long long row = (long long)P.H * P.D * 2;
    if (!encode_rows(&m.q, in.q, P.D, P.H, P.N, P.B, (long long)P.N * row)) return false;
    if (!encode_rows(&m.dout, in.dout, P.D, P.H, P.N, P.B, (long long)P.N * row)) return false;
    bool done[kNumMaps] = {false};
    for (int gi = 0; gi < in.a->n_groups; ++gi) {
        const AttnGroup& ag = in.a->g[gi];
        for (int s = 0; s < ag.n_seg; ++s) {
            const Segment& sg = ag.seg[s];
            int slot = sg.map_id, rows = sg.rows_total;
            const char* kb = sg.k;
            const char* vb = sg.v;
            if (slot == kMapPyr) {
                slot = kMapPyr0 + gi;
                kb += (size_t)sg.row0 * row;
                vb += (size_t)sg.row0 * row;
                rows = sg.len;
            } else if (slot == kMapHist) {
                rows = sg.len;
            }
            if (done[slot]) continue;
            if (!encode_rows(&m.k[slot], kb, P.D, P.H, rows, P.B, sg.bstride) ||
                !encode_rows(&m.v[slot], vb, P.D, P.H, rows, P.B, sg.bstride))
                return false;
            done[slot] = true;
        }
    }
    return true;
}

}  // namespace

msf_status launch_bwd_tc(msf_plan_t plan, const BwdTcInput& in, cudaStream_t st) {
    const Plan& P = *plan;
    const AttnArgs& a = *in.a;
    BwdMaps maps;
    memset(&maps, 0, sizeof(maps));
    if (!encode_all(maps, P, in)) {
        set_cuda_error((int)cudaErrorInvalidValue);
        return MSF_ERR_CUDA;
    }
    BwdTcParams tp;
    memset(&tp, 0, sizeof(tp));
    tp.H = P.H;
    tp.B = P.B;
    tp.N = P.N;
    tp.scale = P.scale;
    tp.scale_log2 = P.scale * kLog2e;
    tp.lse = in.lse;
    tp.delta = in.delta;
    tp.dq = (__nv_bfloat16*)in.dq;
    tp.dk_acc = in.dk_acc;
    tp.dv_acc = in.dv_acc;
    tp.mode = P.d.resample;
    tp.status = a.status;
    tp.wait_limit = kWaitLimit;
    // dQ: every query tile of every group, longest contexts first.
    int order[MSF_MAX_GROUPS];
    int len[MSF_MAX_GROUPS];
    for (int i = 0; i < a.n_groups; ++i) {
        order[i] = i;
        len[i] = 0;
        for (int s = 0; s < a.g[i].n_seg; ++s) len[i] += a.g[i].seg[s].len;
    }
    for (int i = 0; i < a.n_groups; ++i)
        for (int k = i + 1; k < a.n_groups; ++k)
            if (len[order[k]] > len[order[i]]) {
                const int t = order[i];
                order[i] = order[k];
                order[k] = t;
            }
    int items = 0;
    for (int oi = 0; oi < a.n_groups; ++oi) {
        const int gi = order[oi];
        const AttnGroup& ag = a.g[gi];
        BGroupQ& g = tp.g[oi];
        g.q_begin = ag.q_begin;
        g.q_end = ag.q_end;
        g.n_qt = (ag.q_end - ag.q_begin + kBM - 1) / kBM;
        g.item_base = items;
        g.n_seg = ag.n_seg;
        g.n_tiles = 0;
        for (int s = 0; s < ag.n_seg; ++s) {
            const Segment& sg = ag.seg[s];
            BSeg& bs = g.seg[s];
            bs.map = sg.map_id == kMapPyr ? kMapPyr0 + gi : sg.map_id;
            bs.row0 = sg.map_id == kMapPyr ? 0 : sg.row0;
            bs.len = sg.len;
            bs.tile0 = g.n_tiles;
            g.n_tiles += (sg.len + kBM - 1) / kBM;
        }
        items += g.n_qt * P.H * P.B;
    }
    tp.n_groups = a.n_groups;
    const bool d128 = P.D == 128;
    const int smem = d128 ? BCfg<128>::kSmem : BCfg<64>::kSmem;
    static bool attr_set = false;
    if (!attr_set) {
        cudaError_t e = cudaFuncSetAttribute(bwd_dq_tc_kernel<128>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, BCfg<128>::kSmem);
        if (e == cudaSuccess)
            e = cudaFuncSetAttribute(bwd_dq_tc_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     BCfg<64>::kSmem);
        if (e == cudaSuccess)
            e = cudaFuncSetAttribute(bwd_dkdv_tc_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     BCfg<128>::kSmem);
        if (e == cudaSuccess)
            e = cudaFuncSetAttribute(bwd_dkdv_tc_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     BCfg<64>::kSmem);
        if (e != cudaSuccess) {
            set_cuda_error((int)e);
            return MSF_ERR_CUDA;
        }
        attr_set = true;
    }
    cudaError_t e = cudaSuccess;
    if (items > 0)
        e = d128 ? launch_pdl(bwd_dq_tc_kernel<128>, dim3((unsigned)items), dim3(kThreads), smem, st, maps, tp)
                 : launch_pdl(bwd_dq_tc_kernel<64>, dim3((unsigned)items), dim3(kThreads), smem, st, maps, tp);
    if (e != cudaSuccess) {
        set_cuda_error((int)e);
        return MSF_ERR_CUDA;
    }
    // dK/dV: one launch per group, so that every accumulator row has one
    // writer per launch and the sums over groups come in a fixed order.
    for (int gi = 0; gi < a.n_groups; ++gi) {
        const BwdGroup& bg = in.g[gi];
        if (bg.n_gseg == 0 || bg.q_end <= bg.q_begin) continue;
        tp.q_begin = bg.q_begin;
        tp.q_end = bg.q_end;
        tp.n_qt = (bg.q_end - bg.q_begin + kBM - 1) / kBM;
        tp.n_grad = bg.n_gseg;
        int kt0 = 0;
        for (int s = 0; s < bg.n_gseg; ++s) {
            const GradSeg& gs = bg.gseg[s];
            BGrad& g = tp.gr[s];
            g.map = gs.map_id == kMapPyr ? kMapPyr0 + gi : gs.map_id;
            // pyramid rows are addressed from the group's pyramid part, the
            // ring from its first slot, the window from token 0
            g.row0 = gs.map_id == kMapPyr ? gs.row0 - P.groups[gi].pyr_offset : gs.row0;
            g.len = gs.len;
            g.kt0 = kt0;
            g.sigma = gs.sigma;
            g.dst0 = gs.dst0;
            g.src_gw = gs.src_gw;
            g.out_gw = gs.out_gw;
            kt0 += (gs.len + kBM - 1) / kBM;
        }
        const unsigned grid = (unsigned)(kt0 * P.H * P.B);
        e = d128 ? launch_pdl(bwd_dkdv_tc_kernel<128>, dim3(grid), dim3(kThreads), smem, st, maps, tp)
                 : launch_pdl(bwd_dkdv_tc_kernel<64>, dim3(grid), dim3(kThreads), smem, st, maps, tp);
        if (e != cudaSuccess) {
            set_cuda_error((int)e);
            return MSF_ERR_CUDA;
        }
    }
    return MSF_OK;
}

}  // namespace msf
