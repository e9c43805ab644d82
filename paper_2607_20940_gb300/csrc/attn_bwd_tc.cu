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
//     S = Q K^T (SS, two buffers), dP = dO V^T (SS)  -> TMEM
//     softmax warps: P, dS (bf16, over S's columns)   -> TMEM
//     dQ += dS K (TS, K read MN-major)               -> TMEM
//   then scales dQ by c and stores it.
// bwd_dkdv_tc_kernel: one CTA per 128-row tile of context rows that come
//   from the window, every group in one launch. It walks its group's
//   queries in 128-row tiles:
//     S^T = K Q^T (SS), dP^T = V dO^T (SS)            -> TMEM (lanes = keys)
//     softmax warps: P^T, dS^T (bf16, over S^T/dP^T)  -> TMEM
//     dV += P^T dO (TS), dK += dS^T Q (TS)           -> TMEM
//   then writes c dK and dV (fp32) to its rows of the context-gradient
//   buffers, staged through shared memory so that every warp stores whole
//   rows. A gather kernel applies the adjoint of Subsample afterwards.
//
// Roles (384 threads): warp 0 TMA producer, warp 1 MMA issuer (warp-wide
// loop, one elected lane issues), warp 2 TMEM allocation, warps 4-11 the
// softmax: a thread per TMEM lane (query row or key row) and column half,
// warps 4-7 columns 0-63, warps 8-11 columns 64-127. Each half writes its
// bf16 P / dS into its own columns (the MMA that reads them takes its A
// operand per 16-column step), so the halves never wait for each other.
// TMEM columns of the dK/dV
// kernel: S^T [0,128), dP^T [128,256), dV, dK from 256 (the dQ kernel's
// layout is given with it). The tensor pipe executes MMAs
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
constexpr int kThreads = 384;  // 12 warps
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
    int crow0;                // first row of the run in the context-gradient buffers
};
struct BGroupK {
    int q_begin, q_end, n_qt;
    int item_base;  // first item of this group
    int n_kt;       // key tiles of this group (all runs)
    int n_grad;
    BGrad gr[kMaxGradSeg];
};
struct BwdTcParams {
    int H, B, N;
    float scale, scale_log2;
    const float* lse;
    const float* delta;
    __nv_bfloat16* dq;
    float* dk_ctx;
    float* dv_ctx;
    int R;  // rows per stream of the context-gradient buffers
    unsigned int* status;
    long long wait_limit;
    // bwd_dq_tc_kernel
    int n_groups;
    BGroupQ g[MSF_MAX_GROUPS];
    // dK/dV work
    int n_kgroups;
    BGroupK kg[MSF_MAX_GROUPS];
    // Block ranges of the one launch, most expensive items first: kind 0 =
    // dq items of group g[group], kind 1 = dK/dV items of kg[group].
    int n_ranges;
    struct Range {
        int kind, group, base, count;
    } range[2 * MSF_MAX_GROUPS];
};
struct BwdMaps {
    CUtensorMap q, dout;
    CUtensorMap k[kNumMaps];
    CUtensorMap v[kNumMaps];
};

// Dynamic shared memory of the launch: seven 128 x D bf16 tiles (dq items:
// Q, dO, a 3-deep K ring and a 2-deep V ring; dK/dV items: K, V, a 2-deep
// Q/dO ring and the per-query statistics), at least 120 KB so that one CTA
// (and one 512-column TMEM allocation) sits on an SM.
template <int D>
struct BCfg {
    static constexpr int kTile = kBM * D * 2;
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
//
// TMEM: S for even tiles [0,128), S for odd tiles [128,256), dP [256,384),
// dQ from 384. Smem: Q, dO, a 3-deep K ring, a 2-deep V ring. The softmax
// warps first copy dP_j into registers and release it, so dP_{j+1} (and
// S_{j+1}, issued a tile ahead into the other S buffer) run on the tensor
// pipe while they compute dS_j; dQ_j and S_{j+2} then run while the softmax
// works on tile j+1.

template <int D>
struct QCfg {
    static constexpr int kTile = kBM * D * 2;
    static constexpr int kSmem = 7 * kTile + 1024 > 120 * 1024 ? 7 * kTile + 1024 : 120 * 1024;
};
static_assert(7 * QCfg<128>::kTile + 1024 + 2048 <= 227 * 1024, "shared memory of the launch");

template <int D>
__device__ __forceinline__ void dq_item(const BwdMaps& maps, const BwdTcParams& p, int gi, int local) {
    using C = QCfg<D>;
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    unsigned char* smem = (unsigned char*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    unsigned char* sQ = smem;
    unsigned char* sG = smem + C::kTile;       // dO
    unsigned char* sK = smem + 2 * C::kTile;   // [3]
    unsigned char* sV = smem + 5 * C::kTile;   // [2]

    __shared__ uint64_t qg_full, k_full[3], k_empty[3], v_full[2], v_empty[2];
    __shared__ uint64_t sdp_full, dp_free, ds_full, dq_full, drain_bar;
    __shared__ uint32_t tmem_base_sh;
    __shared__ int abort_flag;

    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const BGroupQ& G = p.g[gi];
    const int qt = local % G.n_qt;
    const int h = (local / G.n_qt) % p.H;
    const int b = local / (G.n_qt * p.H);
    const int q_row0 = G.q_begin + qt * kBM;
    const int n = G.n_tiles;

    if (threadIdx.x == 0) {
        abort_flag = 0;
        ptx::mbar_init(&qg_full, 1);
        for (int s = 0; s < 3; ++s) {
            ptx::mbar_init(&k_full[s], 1);
            ptx::mbar_init(&k_empty[s], 1);
        }
        for (int s = 0; s < 2; ++s) {
            ptx::mbar_init(&v_full[s], 1);
            ptx::mbar_init(&v_empty[s], 1);
        }
        ptx::mbar_init(&sdp_full, 1);
        ptx::mbar_init(&dp_free, 8);
        ptx::mbar_init(&ds_full, 8);
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
            int j = 0, nk = 0, nv = 0;
            for (; j < n; ++j) {
                int seg, row, valid;
                tile_of(j, seg, row, valid);
                const int ks = j % 3, vs = j & 1;
                if (!ptx::mbar_wait_bounded(&k_empty[ks], (uint32_t)(((j / 3) & 1) ^ 1), abort_p,
                                            p.wait_limit)) {
                    ok = false;
                    break;
                }
                ptx::mbar_arrive_expect_tx(&k_full[ks], C::kTile);
                load_tile<D>(sK + ks * C::kTile, &maps.k[G.seg[seg].map], &k_full[ks], h, row, b);
                ++nk;
                if (!ptx::mbar_wait_bounded(&v_empty[vs], (uint32_t)(((j >> 1) & 1) ^ 1), abort_p,
                                            p.wait_limit)) {
                    ok = false;
                    break;
                }
                ptx::mbar_arrive_expect_tx(&v_full[vs], C::kTile);
                load_tile<D>(sV + vs * C::kTile, &maps.v[G.seg[seg].map], &v_full[vs], h, row, b);
                ++nv;
            }
            if (!ok) {
                // every copy issued lands before the CTA exits
                ptx::mbar_wait_bounded(&qg_full, 0, &never, kWaitLimit);
                for (int jj = (nk > 3 ? nk - 3 : 0); jj < nk; ++jj)
                    ptx::mbar_wait_bounded(&k_full[jj % 3], (uint32_t)((jj / 3) & 1), &never, kWaitLimit);
                for (int jj = (nv > 2 ? nv - 2 : 0); jj < nv; ++jj)
                    ptx::mbar_wait_bounded(&v_full[jj & 1], (uint32_t)((jj >> 1) & 1), &never, kWaitLimit);
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
        auto issue_s = [&](int j) {  // S_j = Q K_j^T into the S buffer of j's parity
            const uint64_t kd = k_desc + (uint64_t)(j % 3) * kTileDesc;
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk)
                ptx::mma_ss(tbase + (j & 1) * 128, q_desc + kmajor_step(kk), kd + kmajor_step(kk), idS,
                            kk > 0 ? 1u : 0u);
        };
        auto issue_dp = [&](int j) {  // dP_j = dO V_j^T
            const uint64_t vd = v_desc + (uint64_t)(j & 1) * kTileDesc;
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk)
                ptx::mma_ss(tbase + 256, g_desc + kmajor_step(kk), vd + kmajor_step(kk), idS,
                            kk > 0 ? 1u : 0u);
            ptx::mma_commit(&v_empty[j & 1]);
            ptx::mma_commit(&sdp_full);
        };
        bool ok = wait_all(&qg_full, 0) && wait_all(&k_full[0], 0) && wait_all(&v_full[0], 0);
        if (ok) {
            ptx::tc_fence_after();
            if (ptx::elect_one_sync()) {
                issue_s(0);
                issue_dp(0);
            }
            __syncwarp();
            if (n > 1) {
                ok = wait_all(&k_full[1], 0);
                if (ok) {
                    ptx::tc_fence_after();
                    if (ptx::elect_one_sync()) issue_s(1);
                    __syncwarp();
                }
            }
        }
        // Two probe points per tile. A tcgen05.mma holds its issuing thread
        // about as long as the tensor pipe takes to run it, and only ~250
        // cycles of work stay in flight after the last issue, so every
        // barrier check here is pipe time: the probes of each point go out
        // together, and the bounded waits run only if one is not ready.
        for (int j = 0; j < n && ok; ++j) {
            const bool next = j + 1 < n, next2 = j + 2 < n;
            {
                const bool rd = ptx::mbar_try_wait(&dp_free, (uint32_t)(j & 1));
                const bool rv = !next || ptx::mbar_try_wait(&v_full[(j + 1) & 1], (uint32_t)(((j + 1) >> 1) & 1));
                if (!__all_sync(0xffffffffu, rd && rv))
                    ok = wait_all(&dp_free, (uint32_t)(j & 1)) &&
                         (!next || wait_all(&v_full[(j + 1) & 1], (uint32_t)(((j + 1) >> 1) & 1)));
            }
            if (!ok) break;
            if (next) {
                ptx::tc_fence_after();
                if (ptx::elect_one_sync()) issue_dp(j + 1);
                __syncwarp();
            }
            // dS_j, and K_{j+2} for the S two tiles ahead; if K has not
            // landed yet, dQ_j goes first and S_{j+2} after its own wait.
            bool k_ready;
            {
                const bool rs = ptx::mbar_try_wait(&ds_full, (uint32_t)(j & 1));
                k_ready = !next2 || ptx::mbar_try_wait(&k_full[(j + 2) % 3], (uint32_t)(((j + 2) / 3) & 1));
                k_ready = __all_sync(0xffffffffu, k_ready);
                if (!__all_sync(0xffffffffu, rs)) ok = wait_all(&ds_full, (uint32_t)(j & 1));
            }
            if (!ok) break;
            ptx::tc_fence_after();
            if (ptx::elect_one_sync()) {
                const uint64_t kd = kmn_desc + (uint64_t)(j % 3) * kTileDesc;
#pragma unroll
                for (int kk = 0; kk < kBM / 16; ++kk)
                    ptx::mma_ts(tbase + 384, tbase + (j & 1) * 128 + 64 * (kk / 4) + (kk % 4) * 8,
                                kd + (uint64_t)(kk * (2048 >> 4)), idQ, (j > 0 || kk > 0) ? 1u : 0u);
                ptx::mma_commit(&k_empty[j % 3]);
                if (j + 1 == n) ptx::mma_commit(&dq_full);
                if (next2 && k_ready) issue_s(j + 2);
            }
            __syncwarp();
            if (next2 && !k_ready) {
                ok = wait_all(&k_full[(j + 2) % 3], (uint32_t)(((j + 2) / 3) & 1));
                if (!ok) break;
                ptx::tc_fence_after();
                if (ptx::elect_one_sync()) issue_s(j + 2);
                __syncwarp();
            }
        }
        if (!ok) {
            if (ptx::elect_one_sync()) ptx::mma_commit(&drain_bar);
            __syncwarp();
            ptx::mbar_wait_bounded(&drain_bar, 0, &never, kWaitLimit);
            if (lane == 0) atomicOr(p.status, kDevTimeout);
        }
    } else if (warp >= 4) {
        // ============ softmax: one thread per query row and column half ============
        const int half = (warp - 4) / 4;
        const int wq = warp % 4;
        const int r = wq * 32 + lane;
        const uint32_t lane_off = (uint32_t)(wq * 32) << 16;
        const uint32_t tP = tbase + 256 + 64 * half + lane_off;
        const int q = q_row0 + r;
        const bool qv = q < G.q_end;
        const size_t rix = ((size_t)b * p.H + h) * p.N + (qv ? q : 0);
        const float nl = qv ? -p.lse[rix] * kLog2e : -INFINITY;  // -lse in log2 units
        const float dl = qv ? p.delta[rix] : 0.f;
        const uint64_t sl2x2 = ptx::f2_pack(p.scale_log2, p.scale_log2), nlx2 = ptx::f2_pack(nl, nl);
        const uint64_t ndlx2 = ptx::f2_pack(-dl, -dl);
        bool ok = true;
        for (int j = 0; j < n && ok; ++j) {
            int seg, row, valid;
            tile_of(j, seg, row, valid);
            ok = __all_sync(0xffffffffu, ptx::mbar_wait_bounded(&sdp_full, (uint32_t)(j & 1), abort_p,
                                                                p.wait_limit));
            if (!ok) break;
            ptx::tc_fence_after();
            // this half's dP_j into registers, then release its columns
            uint32_t dp[2][32];
            ptx::tmem_ld32(tP, dp[0]);
            ptx::tmem_ld32(tP + 32, dp[1]);
            ptx::tmem_wait_ld();
            ptx::tc_fence_before();
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&dp_free);
            const uint32_t tS = tbase + (j & 1) * 128 + 64 * half + lane_off;
#pragma unroll
            for (int c2 = 0; c2 < 2; ++c2) {
                uint32_t s[32];
                ptx::tmem_ld32(tS + 32 * c2, s);
                ptx::tmem_wait_ld();
                const int lim = valid - (64 * half + 32 * c2);
                if (lim < 32) {
                    // keys past the segment's end: score -inf, probability 0
#pragma unroll
                    for (int e = 0; e < 32; ++e)
                        if (e >= lim) s[e] = 0xff800000u;
                }
                uint32_t pk[16];
#pragma unroll
                for (int e = 0; e < 16; ++e) {
                    const uint64_t arg = ptx::f2_fma(
                        ptx::f2_pack(__uint_as_float(s[2 * e]), __uint_as_float(s[2 * e + 1])), sl2x2, nlx2);
                    float a0, a1;
                    ptx::f2_unpack(arg, a0, a1);
                    const uint64_t pp = ptx::f2_pack(ex2(a0), ex2(a1));
                    const uint64_t dd = ptx::f2_add(
                        ptx::f2_pack(__uint_as_float(dp[c2][2 * e]), __uint_as_float(dp[c2][2 * e + 1])), ndlx2);
                    const uint64_t ds = ptx::f2_mul(pp, dd);
                    float d0, d1;
                    ptx::f2_unpack(ds, d0, d1);
                    pk[e] = ptx::pack_bf16(d0, d1);
                }
                ptx::tmem_st16(tS + 16 * c2, pk);
            }
            ptx::tmem_wait_st();
            ptx::tc_fence_before();
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&ds_full);
        }
        if (ok) ok = __all_sync(0xffffffffu, ptx::mbar_wait_bounded(&dq_full, 0, abort_p, p.wait_limit));
        if (ok) {
            // each half stores D/2 columns of its row
            ptx::tc_fence_after();
            constexpr int DH = D / 2;
            const uint32_t tQ = tbase + 384 + DH * half + lane_off;
            __nv_bfloat16* dst = p.dq + (((size_t)b * p.N + (qv ? q : 0)) * p.H + h) * D + DH * half;
#pragma unroll
            for (int c = 0; c < DH / 32; ++c) {
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

template <int D>
__device__ __forceinline__ void dkdv_item(const BwdMaps& maps, const BwdTcParams& p, int kgi,
                                          int local) {
    using C = BCfg<D>;
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    unsigned char* smem = (unsigned char*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    unsigned char* sK = smem;
    unsigned char* sV = smem + C::kTile;
    unsigned char* sQ = smem + 2 * C::kTile;   // [2]
    unsigned char* sG = smem + 4 * C::kTile;   // [2] dO

    __shared__ uint64_t kv_full, qg_full[2], qg_empty[2], st_full[2], pds_full[2], kv_done, drain_bar;
    __shared__ uint32_t tmem_base_sh;
    __shared__ int abort_flag;
    // per-query statistics of the current and the previous query tile, in
    // the seventh tile of the dynamic shared memory
    float(*sL)[kBM] = reinterpret_cast<float(*)[kBM]>(smem + 6 * C::kTile);
    float(*sD)[kBM] = reinterpret_cast<float(*)[kBM]>(smem + 6 * C::kTile + 2 * kBM * 4);

    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const BGroupK& KG = p.kg[kgi];
    const int kt_all = local % KG.n_kt;
    const int h = (local / KG.n_kt) % p.H;
    const int b = local / (KG.n_kt * p.H);
    int gsi = 0;
    while (gsi + 1 < KG.n_grad && kt_all >= KG.gr[gsi + 1].kt0) ++gsi;
    const BGrad& gr = KG.gr[gsi];
    const int kt = kt_all - gr.kt0;
    const int key_row = gr.row0 + kt * kBM;
    const int valid_keys = min(kBM, gr.len - kt * kBM);
    const int nq = KG.n_qt;

    if (threadIdx.x == 0) {
        abort_flag = 0;
        ptx::mbar_init(&kv_full, 1);
        for (int s = 0; s < 2; ++s) {
            ptx::mbar_init(&qg_full[s], 1);
            ptx::mbar_init(&qg_empty[s], 1);
        }
        for (int s = 0; s < 2; ++s) {
            ptx::mbar_init(&st_full[s], 1);
            ptx::mbar_init(&pds_full[s], 4);  // one arrival per warp of the column half
        }
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
                load_tile<D>(sQ + st * C::kTile, &maps.q, &qg_full[st], h, KG.q_begin + i * kBM, b);
                load_tile<D>(sG + st * C::kTile, &maps.dout, &qg_full[st], h, KG.q_begin + i * kBM, b);
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
        // Query tile i is done in two halves of 64 queries: half A's
        // dV/dK MMAs and the next tile's S^T/dP^T of half A run while the
        // softmax works on half B, and the other way round.
        constexpr uint32_t idS64 = ptx::idesc_bf16(kBM, 64, false, false);
        auto issue_st = [&](int i, int hf) {  // S^T, dP^T of half hf of query tile i
            const int st = i & 1;
            const uint64_t qd = q_desc + (uint64_t)st * kTileDesc + (uint64_t)((64 * 128 * hf) >> 4);
            const uint64_t gd = g_desc + (uint64_t)st * kTileDesc + (uint64_t)((64 * 128 * hf) >> 4);
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk)
                ptx::mma_ss(tbase + 64 * hf, k_desc + kmajor_step(kk), qd + kmajor_step(kk), idS64,
                            kk > 0 ? 1u : 0u);
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk)
                ptx::mma_ss(tbase + 128 + 64 * hf, v_desc + kmajor_step(kk), gd + kmajor_step(kk), idS64,
                            kk > 0 ? 1u : 0u);
            ptx::mma_commit(&st_full[hf]);
        };
        auto issue_kv = [&](int i, int hf) {  // dV += P^T dO, dK += dS^T Q over half hf
            const int st = i & 1;
            const uint64_t gd = gmn_desc + (uint64_t)st * kTileDesc;
            const uint64_t qd = qmn_desc + (uint64_t)st * kTileDesc;
#pragma unroll
            for (int kk = 0; kk < 4; ++kk) {
                const uint64_t roff = (uint64_t)((4 * hf + kk) * (2048 >> 4));
                ptx::mma_ts(tbase + 256, tbase + 64 * hf + kk * 8, gd + roff, idO,
                            (i > 0 || hf > 0 || kk > 0) ? 1u : 0u);
                ptx::mma_ts(tbase + 256 + D, tbase + 128 + 64 * hf + kk * 8, qd + roff, idO,
                            (i > 0 || hf > 0 || kk > 0) ? 1u : 0u);
            }
        };
        bool ok = wait_all(&kv_full, 0) && wait_all(&qg_full[0], 0);
        if (ok) {
            ptx::tc_fence_after();
            if (ptx::elect_one_sync()) {
                issue_st(0, 0);
                issue_st(0, 1);
            }
            __syncwarp();
        }
        for (int i = 0; i < nq && ok; ++i) {
            const int st = i & 1;
            const bool more = i + 1 < nq;
            // P/dS of half 0 and the next query tile's Q/dO, probed together
            // (each barrier check of this thread is pipe time); if Q/dO has
            // not landed, half 0's dV/dK go first.
            bool q_ready;
            {
                const bool rp = ptx::mbar_try_wait(&pds_full[0], (uint32_t)(i & 1));
                q_ready = !more || ptx::mbar_try_wait(&qg_full[st ^ 1], (uint32_t)(((i + 1) >> 1) & 1));
                q_ready = __all_sync(0xffffffffu, q_ready);
                if (!__all_sync(0xffffffffu, rp)) ok = wait_all(&pds_full[0], (uint32_t)(i & 1));
            }
            if (!ok) break;
            ptx::tc_fence_after();
            if (ptx::elect_one_sync()) {
                issue_kv(i, 0);
                if (more && q_ready) issue_st(i + 1, 0);
            }
            __syncwarp();
            if (more && !q_ready) {
                ok = wait_all(&qg_full[st ^ 1], (uint32_t)(((i + 1) >> 1) & 1));
                if (!ok) break;
                ptx::tc_fence_after();
                if (ptx::elect_one_sync()) issue_st(i + 1, 0);
                __syncwarp();
            }
            ok = wait_all(&pds_full[1], (uint32_t)(i & 1));
            if (!ok) break;
            ptx::tc_fence_after();
            if (ptx::elect_one_sync()) {
                issue_kv(i, 1);
                ptx::mma_commit(&qg_empty[st]);
                if (more)
                    issue_st(i + 1, 1);
                else
                    ptx::mma_commit(&kv_done);
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
        // ============= softmax: one thread per key row and column half =============
        const int half = (warp - 4) / 4;
        const int wq = warp % 4;
        const int r = wq * 32 + lane;
        const int tix = (warp - 4) * 32 + lane;  // 0..255
        const uint32_t lane_off = (uint32_t)(wq * 32) << 16;
        const uint32_t tS = tbase + 64 * half + lane_off, tP = tbase + 128 + 64 * half + lane_off;
        const uint64_t sl2x2 = ptx::f2_pack(p.scale_log2, p.scale_log2);
        bool ok = true;
        for (int i = 0; i < nq && ok; ++i) {
            // this half's 64 per-query statistics, shared by its 128 key rows:
            // threads 0-63 of the half load -lse (log2 units), 64-127 -delta
            {
                const int hix = tix & 127;
                const int qq = 64 * half + (hix & 63);
                const int q = KG.q_begin + i * kBM + qq;
                const bool qv = q < KG.q_end;
                const size_t rix = ((size_t)b * p.H + h) * p.N + (qv ? q : 0);
                if (hix < 64)
                    sL[i & 1][qq] = qv ? -p.lse[rix] * kLog2e : -INFINITY;
                else
                    sD[i & 1][qq] = qv ? -p.delta[rix] : 0.f;
            }
            ptx::named_bar_sync(1 + half, 128);
            const float* L = sL[i & 1] + 64 * half;
            const float* ND = sD[i & 1] + 64 * half;
            ok = __all_sync(0xffffffffu, ptx::mbar_wait_bounded(&st_full[half], (uint32_t)(i & 1), abort_p,
                                                                p.wait_limit));
            if (!ok) break;
            ptx::tc_fence_after();
#pragma unroll
            for (int c2 = 0; c2 < 2; ++c2) {
                uint32_t s[32], dp[32];
                ptx::tmem_ld32(tS + 32 * c2, s);
                ptx::tmem_ld32(tP + 32 * c2, dp);
                ptx::tmem_wait_ld();
                uint32_t pp[16], pd[16];
#pragma unroll
                for (int e = 0; e < 16; ++e) {
                    const int c0 = 32 * c2 + 2 * e;
                    const uint64_t arg = ptx::f2_fma(
                        ptx::f2_pack(__uint_as_float(s[2 * e]), __uint_as_float(s[2 * e + 1])), sl2x2,
                        ptx::f2_pack(L[c0], L[c0 + 1]));
                    float a0, a1;
                    ptx::f2_unpack(arg, a0, a1);
                    const float p0 = ex2(a0), p1 = ex2(a1);
                    pp[e] = ptx::pack_bf16(p0, p1);
                    const uint64_t dd = ptx::f2_add(
                        ptx::f2_pack(__uint_as_float(dp[2 * e]), __uint_as_float(dp[2 * e + 1])),
                        ptx::f2_pack(ND[c0], ND[c0 + 1]));
                    float d0, d1;
                    ptx::f2_unpack(ptx::f2_mul(ptx::f2_pack(p0, p1), dd), d0, d1);
                    pd[e] = ptx::pack_bf16(d0, d1);
                }
                ptx::tmem_st16(tS + 16 * c2, pp);
                ptx::tmem_st16(tP + 16 * c2, pd);
            }
            ptx::tmem_wait_st();
            ptx::tc_fence_before();
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&pds_full[half]);
        }
        if (ok) ok = __all_sync(0xffffffffu, ptx::mbar_wait_bounded(&kv_done, 0, abort_p, p.wait_limit));
        if (ok) {
            // Every MMA has completed: the Q/dO ring is free and stages one
            // fp32 [128][D + 4] tile (dK, then dV); each half fills D/2
            // columns of its rows, then every warp stores whole rows.
            ptx::tc_fence_after();
            float* stage = reinterpret_cast<float*>(sQ);
            constexpr int kStride = D + 4;
            constexpr int E = D / 32;
            constexpr int DH = D / 2;
            for (int which = 0; which < 2; ++which) {
                const float mul = which == 0 ? p.scale : 1.f;
#pragma unroll
                for (int c = 0; c < DH / 32; ++c) {
                    uint32_t o[32];
                    ptx::tmem_ld32(tbase + 256 + (which == 0 ? D : 0) + DH * half + 32 * c + lane_off, o);
                    ptx::tmem_wait_ld();
                    float4* dst = reinterpret_cast<float4*>(stage + r * kStride + DH * half + 32 * c);
#pragma unroll
                    for (int e = 0; e < 8; ++e)
                        dst[e] = make_float4(__uint_as_float(o[4 * e]) * mul, __uint_as_float(o[4 * e + 1]) * mul,
                                             __uint_as_float(o[4 * e + 2]) * mul,
                                             __uint_as_float(o[4 * e + 3]) * mul);
                }
                ptx::named_bar_sync(3, 256);
                float* base = (which == 0 ? p.dk_ctx : p.dv_ctx);
                for (int rr = warp - 4; rr < valid_keys; rr += 8) {
                    const size_t o = (((size_t)b * p.R + gr.crow0 + kt * kBM + rr) * p.H + h) * D + E * lane;
                    const float* src = stage + rr * kStride + E * lane;
                    if (E == 4)
                        *reinterpret_cast<float4*>(base + o) = *reinterpret_cast<const float4*>(src);
                    else
                        *reinterpret_cast<float2*>(base + o) = *reinterpret_cast<const float2*>(src);
                }
                ptx::named_bar_sync(3, 256);
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

// One launch for both kinds of work, so that short dK/dV items fill the
// SMs that long dq items leave idle at the end.
template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    bwd_tc_kernel(const __grid_constant__ BwdMaps maps, const __grid_constant__ BwdTcParams p) {
    int r = 0;
    while (r + 1 < p.n_ranges && (int)blockIdx.x >= p.range[r + 1].base) ++r;
    const int local = (int)blockIdx.x - p.range[r].base;
    if (p.range[r].kind == 0)
        dq_item<D>(maps, p, p.range[r].group, local);
    else
        dkdv_item<D>(maps, p, p.range[r].group, local);
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
    tp.dk_ctx = in.dk_ctx;
    tp.dv_ctx = in.dv_ctx;
    tp.R = in.R;
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
    tp.n_groups = a.n_groups;
    // dK/dV: every group's window-derived rows in one launch, groups with
    // the most query tiles first.
    int korder[MSF_MAX_GROUPS];
    int nk = 0;
    for (int gi = 0; gi < a.n_groups; ++gi)
        if (in.g[gi].n_gseg > 0 && in.g[gi].q_end > in.g[gi].q_begin) korder[nk++] = gi;
    for (int i = 0; i < nk; ++i)
        for (int k = i + 1; k < nk; ++k)
            if (in.g[korder[k]].q_end - in.g[korder[k]].q_begin >
                in.g[korder[i]].q_end - in.g[korder[i]].q_begin) {
                const int t = korder[i];
                korder[i] = korder[k];
                korder[k] = t;
            }
    int kitems = 0;
    for (int oi = 0; oi < nk; ++oi) {
        const int gi = korder[oi];
        const BwdGroup& bg = in.g[gi];
        BGroupK& kg = tp.kg[oi];
        kg.q_begin = bg.q_begin;
        kg.q_end = bg.q_end;
        kg.n_qt = (bg.q_end - bg.q_begin + kBM - 1) / kBM;
        kg.item_base = kitems;
        kg.n_grad = bg.n_gseg;
        int kt0 = 0;
        for (int s = 0; s < bg.n_gseg; ++s) {
            const GradSeg& gs = bg.gseg[s];
            BGrad& g = kg.gr[s];
            g.map = gs.map_id == kMapPyr ? kMapPyr0 + gi : gs.map_id;
            // pyramid rows are addressed from the group's pyramid part, the
            // ring from its first slot, the window from token 0
            g.row0 = gs.map_id == kMapPyr ? gs.row0 - P.groups[gi].pyr_offset : gs.row0;
            g.len = gs.len;
            g.kt0 = kt0;
            g.crow0 = gs.crow0;
            kt0 += (gs.len + kBM - 1) / kBM;
        }
        kg.n_kt = kt0;
        kitems += kt0 * P.H * P.B;
    }
    tp.n_kgroups = nk;
    // Ranges in decreasing cost per item (MMA blocks of 128x128xD: 3 per
    // K/V tile of a dq item, 4 per query tile of a dK/dV item).
    struct R {
        int kind, group, count;
        long long cost;
    } rs[2 * MSF_MAX_GROUPS];
    int nr = 0;
    for (int oi = 0; oi < a.n_groups; ++oi)
        if (tp.g[oi].n_qt > 0)
            rs[nr++] = {0, oi, tp.g[oi].n_qt * P.H * P.B, 3LL * tp.g[oi].n_tiles};
    for (int oi = 0; oi < nk; ++oi)
        if (tp.kg[oi].n_kt > 0)
            rs[nr++] = {1, oi, tp.kg[oi].n_kt * P.H * P.B, 4LL * tp.kg[oi].n_qt};
    for (int i = 0; i < nr; ++i)
        for (int k = i + 1; k < nr; ++k)
            if (rs[k].cost > rs[i].cost) {
                const R t = rs[i];
                rs[i] = rs[k];
                rs[k] = t;
            }
    int total = 0;
    for (int i = 0; i < nr; ++i) {
        tp.range[i].kind = rs[i].kind;
        tp.range[i].group = rs[i].group;
        tp.range[i].base = total;
        tp.range[i].count = rs[i].count;
        total += rs[i].count;
    }
    tp.n_ranges = nr;
    (void)items;
    (void)kitems;
    if (total == 0) return MSF_OK;
    const bool d128 = P.D == 128;
    const int smem = d128 ? QCfg<128>::kSmem : QCfg<64>::kSmem;
    cudaError_t e = d128 ? set_smem_attr((const void*)bwd_tc_kernel<128>, QCfg<128>::kSmem)
                         : set_smem_attr((const void*)bwd_tc_kernel<64>, QCfg<64>::kSmem);
    if (e != cudaSuccess) {
        set_cuda_error((int)e);
        return MSF_ERR_CUDA;
    }
    e = d128 ? launch_pdl(bwd_tc_kernel<128>, dim3((unsigned)total), dim3(kThreads), smem, st, maps, tp)
             : launch_pdl(bwd_tc_kernel<64>, dim3((unsigned)total), dim3(kThreads), smem, st, maps, tp);
    if (e != cudaSuccess) {
        set_cuda_error((int)e);
        return MSF_ERR_CUDA;
    }
    return MSF_OK;
}

}  // namespace msf
