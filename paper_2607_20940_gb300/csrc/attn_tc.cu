// MSSA attention on the sm_103a tensor cores (Eq. 4 context, bf16 operands,
// fp32 online softmax and accumulation).
//
// One CTA owns a 256-row query block (two 128-row tiles Q0, Q1) of one
// (stream, head, query group) and walks that group's context segments
// (sink, history or pyramid part, window suffix) in 128-row K/V tiles:
//   warp 0      TMA producer: Q0/Q1 once, then K_j and V_j into a 2-stage ring
//   warp 1      MMA issuer (one thread): S_t = Q_t K_j^T into TMEM (SS form),
//               O_t += P_t V_j with P_t read from TMEM (TS form, V MN-major)
//   warp 2      TMEM allocation (all 512 columns)
//   warps 4-7   softmax of tile 0, warps 8-11 softmax of tile 1: one thread
//               per query row; tcgen05.ld of S, row max, exp2, row sum, P as
//               bf16 written over S's first 64 columns, lazy rescale of O
//               (only when the running max grows by more than 2^8)
// TMEM columns: S0 [0,128) S1 [128,256) O0 [256,384) O1 [384,512).
// The MMA thread issues S_t(j+1) right after PV_t(j), so the commit that
// signals S_t(j+1) also covers PV_t(j): a softmax warp that sees S ready may
// rescale O_t in place. Every segment has its own tensor map whose extent is
// the segment's end, so rows past it load as zeros; their scores are masked.
// Waits are bounded; a wait that gives up raises the CTA's abort flag, sets
// the device status word, and every role winds down without hanging.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdlib.h>
#include <string.h>

#include "attn_tc.h"
#include "ptx.cuh"

namespace msf {

namespace {

constexpr int kBlockM = 128;   // query rows per tile
constexpr int kBlockN = 128;   // context rows per K/V tile
constexpr int kStages = 2;     // K/V ring depth
constexpr int kThreads = 384;  // 12 warps
constexpr long long kWaitLimit = 2000000000LL;  // ~1 s of SM clock

struct TcSeg {
    int map;
    int row0;
    int len;
    int ntiles;
};
struct TcGroup {
    int q_begin, q_end;
    int n_qb;      // 256-row query blocks
    int n_items;   // B * H * n_qb
    int n_seg;
    int n_tiles;   // sum of segment tiles
    TcSeg seg[kMaxSeg];
};
struct TcParams {
    int H, B;
    float scale_log2;
    int n_groups;
    TcGroup g[MSF_MAX_GROUPS];  // longest context first
    __nv_bfloat16* out;
    long long out_bstride;  // elements
    unsigned int* status;
    long long wait_limit;
};
struct TcMaps {
    CUtensorMap q;
    CUtensorMap k[kNumMaps];
    CUtensorMap v[kNumMaps];
};

template <int D>
struct Cfg {
    static constexpr int kChunks = D / 64;                    // 128-byte swizzle chunks per row
    static constexpr int kTileBytes = kBlockM * D * 2;        // one Q / K / V tile
    static constexpr int kSmem = (2 + 2 * kStages) * kTileBytes + 1024;
};

__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    mssa_tc_kernel(const __grid_constant__ TcMaps maps, const __grid_constant__ TcParams p) {
    using C = Cfg<D>;
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    unsigned char* smem = (unsigned char*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    unsigned char* sQ = smem;                                  // [2][tile]
    unsigned char* sK = smem + 2 * C::kTileBytes;              // [kStages][tile]
    unsigned char* sV = sK + kStages * C::kTileBytes;          // [kStages][tile]

    __shared__ uint64_t q_full, o_full;
    __shared__ uint64_t k_full[kStages], k_empty[kStages], v_full[kStages], v_empty[kStages];
    __shared__ uint64_t s_full[2], p_full[2];
    __shared__ uint32_t tmem_base_sh;
    __shared__ int abort_flag;

    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;

    // ---- work item: group (longest first), then q block fastest, head, stream
    int item = blockIdx.x, gi = 0;
    while (gi < p.n_groups - 1 && item >= p.g[gi].n_items) {
        item -= p.g[gi].n_items;
        ++gi;
    }
    const TcGroup& G = p.g[gi];
    const int qb = item % G.n_qb;
    const int h = (item / G.n_qb) % p.H;
    const int b = item / (G.n_qb * p.H);
    const int q_row0 = G.q_begin + qb * 2 * kBlockM;
    const int n_tiles = G.n_tiles;

    if (threadIdx.x == 0) {
        abort_flag = 0;
        ptx::mbar_init(&q_full, 1);
        ptx::mbar_init(&o_full, 1);
        for (int s = 0; s < kStages; ++s) {
            ptx::mbar_init(&k_full[s], 1);
            ptx::mbar_init(&k_empty[s], 1);
            ptx::mbar_init(&v_full[s], 1);
            ptx::mbar_init(&v_empty[s], 1);
        }
        for (int t = 0; t < 2; ++t) {
            ptx::mbar_init(&s_full[t], 1);
            ptx::mbar_init(&p_full[t], 128);
        }
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

    if (warp == 0) {
        // =========================== TMA producer ===========================
        if (lane == 0) {
            ptx::prefetch_tmap(&maps.q);
            bool ok = true;
            ptx::mbar_arrive_expect_tx(&q_full, 2 * C::kTileBytes);
            for (int t = 0; t < 2; ++t)
                for (int c = 0; c < C::kChunks; ++c)
                    ptx::tma_load_4d(sQ + t * C::kTileBytes + c * (kBlockM * 128), &maps.q, &q_full,
                                     c * 64, h, q_row0 + t * kBlockM, b);
            int issued = 0;
            for (int si = 0; si < G.n_seg && ok; ++si) {
                const TcSeg& sg = G.seg[si];
                const CUtensorMap* mk = &maps.k[sg.map];
                const CUtensorMap* mv = &maps.v[sg.map];
                for (int kt = 0; kt < sg.ntiles; ++kt) {
                    const int j = issued;
                    const int st = j % kStages;
                    const uint32_t ph = (uint32_t)((j / kStages) & 1);
                    const int row = sg.row0 + kt * kBlockN;
                    if (!ptx::mbar_wait_bounded(&k_empty[st], ph ^ 1u, abort_p, p.wait_limit)) {
                        ok = false;
                        break;
                    }
                    ptx::mbar_arrive_expect_tx(&k_full[st], C::kTileBytes);
                    for (int c = 0; c < C::kChunks; ++c)
                        ptx::tma_load_4d(sK + st * C::kTileBytes + c * (kBlockN * 128), mk,
                                         &k_full[st], c * 64, h, row, b);
                    if (!ptx::mbar_wait_bounded(&v_empty[st], ph ^ 1u, abort_p, p.wait_limit)) {
                        // K of this step is in flight: let it land before leaving
                        volatile int never = 0;
                        ptx::mbar_wait_bounded(&k_full[st], ph, &never, kWaitLimit);
                        ok = false;
                        break;
                    }
                    ptx::mbar_arrive_expect_tx(&v_full[st], C::kTileBytes);
                    for (int c = 0; c < C::kChunks; ++c)
                        ptx::tma_load_4d(sV + st * C::kTileBytes + c * (kBlockN * 128), mv,
                                         &v_full[st], c * 64, h, row, b);
                    ++issued;
                }
            }
            if (!ok) {
                // Drain: every copy issued must land before the CTA exits.
                volatile int never = 0;
                ptx::mbar_wait_bounded(&q_full, 0, &never, kWaitLimit);
                for (int j = (issued > kStages ? issued - kStages : 0); j < issued; ++j) {
                    const int st = j % kStages;
                    const uint32_t ph = (uint32_t)((j / kStages) & 1);
                    ptx::mbar_wait_bounded(&k_full[st], ph, &never, kWaitLimit);
                    ptx::mbar_wait_bounded(&v_full[st], ph, &never, kWaitLimit);
                }
                atomicOr(p.status, kDevTimeout);
            }
        }
    } else if (warp == 1) {
        // ============================ MMA issuer ============================
        if (lane == 0) {
            constexpr uint32_t idS = ptx::idesc_bf16(kBlockM, kBlockN, false, false);
            constexpr uint32_t idO = ptx::idesc_bf16(kBlockM, D, false, true);
            const uint32_t q_addr = ptx::smem_u32(sQ);
            const uint32_t k_addr = ptx::smem_u32(sK);
            const uint32_t v_addr = ptx::smem_u32(sV);
            auto issue_s = [&](int t, int st) {
                const uint32_t qa = q_addr + t * C::kTileBytes;
                const uint32_t ka = k_addr + st * C::kTileBytes;
#pragma unroll
                for (int kk = 0; kk < D / 16; ++kk) {
                    const uint32_t off = (kk / 4) * (kBlockM * 128) + (kk % 4) * 32;
                    ptx::mma_ss(tbase + t * 128, ptx::sdesc_sw128(qa + off, 16, 1024),
                                ptx::sdesc_sw128(ka + off, 16, 1024), idS, kk > 0 ? 1u : 0u);
                }
                ptx::mma_commit(&s_full[t]);
            };
            auto issue_pv = [&](int t, int st, bool acc) {
                const uint32_t va = v_addr + st * C::kTileBytes;
#pragma unroll
                for (int kk = 0; kk < kBlockN / 16; ++kk) {
                    ptx::mma_ts(tbase + 256 + t * 128, tbase + t * 128 + kk * 8,
                                ptx::sdesc_sw128(va + kk * 2048, kBlockN * 128, 1024), idO,
                                (acc || kk > 0) ? 1u : 0u);
                }
            };
            bool ok = ptx::mbar_wait_bounded(&q_full, 0, abort_p, p.wait_limit);
            ok = ok && ptx::mbar_wait_bounded(&k_full[0], 0, abort_p, p.wait_limit);
            if (ok) {
                ptx::tc_fence_after();
                issue_s(0, 0);
                issue_s(1, 0);
                ptx::mma_commit(&k_empty[0]);
            }
            for (int j = 0; j < n_tiles && ok; ++j) {
                const int st = j % kStages;
                const uint32_t ph = (uint32_t)((j / kStages) & 1);
                const int st1 = (j + 1) % kStages;
                const uint32_t ph1 = (uint32_t)(((j + 1) / kStages) & 1);
                const bool more = j + 1 < n_tiles;
                ok = ptx::mbar_wait_bounded(&v_full[st], ph, abort_p, p.wait_limit) &&
                     ptx::mbar_wait_bounded(&p_full[0], (uint32_t)(j & 1), abort_p, p.wait_limit);
                if (!ok) break;
                ptx::tc_fence_after();
                issue_pv(0, st, j > 0);
                if (more) {
                    ok = ptx::mbar_wait_bounded(&k_full[st1], ph1, abort_p, p.wait_limit);
                    if (!ok) break;
                    ptx::tc_fence_after();
                    issue_s(0, st1);
                }
                ok = ptx::mbar_wait_bounded(&p_full[1], (uint32_t)(j & 1), abort_p, p.wait_limit);
                if (!ok) break;
                ptx::tc_fence_after();
                issue_pv(1, st, j > 0);
                ptx::mma_commit(&v_empty[st]);
                if (more) {
                    issue_s(1, st1);
                    ptx::mma_commit(&k_empty[st1]);
                }
            }
            // o_full covers every MMA issued, on the normal and the abort path,
            // so TMEM is never released under a running MMA.
            ptx::mma_commit(&o_full);
            if (!ok) {
                volatile int never = 0;
                ptx::mbar_wait_bounded(&o_full, 0, &never, kWaitLimit);
                atomicOr(p.status, kDevTimeout);
            }
        }
    } else if (warp >= 4) {
        // ============================== softmax =============================
        const int t = (warp - 4) / 4;
        const int wq = warp % 4;
        const int r = wq * 32 + lane;
        const uint32_t lane_off = (uint32_t)(wq * 32) << 16;
        const uint32_t tS = tbase + t * 128 + lane_off;
        const uint32_t tO = tbase + 256 + t * 128 + lane_off;
        const float sl2 = p.scale_log2;
        float m_used = -INFINITY, l = 0.f;
        bool ok = true;
        int j = 0;
        for (int si = 0; si < G.n_seg && ok; ++si) {
            const TcSeg& sg = G.seg[si];
            for (int kt = 0; kt < sg.ntiles; ++kt, ++j) {
                const int valid = min(kBlockN, sg.len - kt * kBlockN);
                ok = ptx::mbar_wait_bounded(&s_full[t], (uint32_t)(j & 1), abort_p, p.wait_limit);
                ok = __all_sync(0xffffffffu, ok);
                if (!ok) break;
                ptx::tc_fence_after();
                uint32_t s[4][32];
#pragma unroll
                for (int q4 = 0; q4 < 4; ++q4) ptx::tmem_ld32(tS + 32 * q4, s[q4]);
                ptx::tmem_wait_ld();
                float mx = -INFINITY;
                if (valid == kBlockN) {
#pragma unroll
                    for (int c = 0; c < 128; ++c) mx = fmaxf(mx, __uint_as_float(s[c >> 5][c & 31]));
                } else {
#pragma unroll
                    for (int c = 0; c < 128; ++c)
                        if (c < valid) mx = fmaxf(mx, __uint_as_float(s[c >> 5][c & 31]));
                }
                const float m_new = fmaxf(m_used, mx * sl2);
                if (j == 0) {
                    m_used = m_new;
                } else if (__any_sync(0xffffffffu, m_new > m_used + 8.0f)) {
                    // O_t holds every PV up to step j-1 (the S_t(j) commit covers it).
                    const float f = ex2(m_used - m_new);
                    l *= f;
                    m_used = m_new;
#pragma unroll 1
                    for (int c = 0; c < D / 16; ++c) {
                        uint32_t o[16];
                        ptx::tmem_ld16(tO + c * 16, o);
                        ptx::tmem_wait_ld();
#pragma unroll
                        for (int e = 0; e < 16; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * f);
                        ptx::tmem_st16(tO + c * 16, o);
                    }
                    ptx::tmem_wait_st();
                }
                const float nm = -m_used;
                float sum = 0.f;
                if (valid == kBlockN) {
#pragma unroll
                    for (int c = 0; c < 64; ++c) {
                        const float p0 = ex2(fmaf(__uint_as_float(s[(2 * c) >> 5][(2 * c) & 31]), sl2, nm));
                        const float p1 = ex2(fmaf(__uint_as_float(s[(2 * c + 1) >> 5][(2 * c + 1) & 31]), sl2, nm));
                        sum += p0 + p1;
                        s[c >> 5][c & 31] = ptx::pack_bf16(p0, p1);
                    }
                } else {
#pragma unroll
                    for (int c = 0; c < 64; ++c) {
                        const float p0 =
                            (2 * c < valid) ? ex2(fmaf(__uint_as_float(s[(2 * c) >> 5][(2 * c) & 31]), sl2, nm)) : 0.f;
                        const float p1 = (2 * c + 1 < valid)
                                             ? ex2(fmaf(__uint_as_float(s[(2 * c + 1) >> 5][(2 * c + 1) & 31]), sl2, nm))
                                             : 0.f;
                        sum += p0 + p1;
                        s[c >> 5][c & 31] = ptx::pack_bf16(p0, p1);
                    }
                }
                l += sum;
                ptx::tmem_st32(tS + 0, s[0]);
                ptx::tmem_st32(tS + 32, s[1]);
                ptx::tmem_wait_st();
                ptx::tc_fence_before();
                ptx::mbar_arrive(&p_full[t]);
            }
        }
        if (ok) {
            ok = ptx::mbar_wait_bounded(&o_full, 0, abort_p, p.wait_limit);
            ok = __all_sync(0xffffffffu, ok);
        }
        if (ok) {
            ptx::tc_fence_after();
            const int qrow = q_row0 + t * kBlockM + r;
            const bool store = qrow < G.q_end;
            const float inv = 1.0f / l;
            __nv_bfloat16* dst = p.out + (size_t)b * p.out_bstride +
                                 ((size_t)qrow * p.H + h) * D;
#pragma unroll
            for (int c = 0; c < D / 32; ++c) {
                uint32_t o[32];
                ptx::tmem_ld32(tO + c * 32, o);
                ptx::tmem_wait_ld();
                uint32_t pk[16];
#pragma unroll
                for (int e = 0; e < 16; ++e)
                    pk[e] = ptx::pack_bf16(__uint_as_float(o[2 * e]) * inv,
                                           __uint_as_float(o[2 * e + 1]) * inv);
                if (store) {
                    uint4* d4 = reinterpret_cast<uint4*>(dst + c * 32);
#pragma unroll
                    for (int e = 0; e < 4; ++e)
                        d4[e] = make_uint4(pk[4 * e], pk[4 * e + 1], pk[4 * e + 2], pk[4 * e + 3]);
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
        ptx::tmem_dealloc(tbase, 512);
    }
}

// ---------------------------------------------------------------- host side

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn get_encode() {
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

// A [B, rows, H, D] bf16 tensor seen as 4-D {D, H, rows, B}; boxes of
// 64 x 1 x 128 x 1 with 128-byte swizzle (one K-major MMA chunk).
bool encode_rows(CUtensorMap* m, const void* base, int D, int H, int rows, int B,
                 long long bstride_bytes) {
    EncodeTiledFn enc = get_encode();
    if (!enc) return false;
    cuuint64_t dims[4] = {(cuuint64_t)D, (cuuint64_t)H, (cuuint64_t)(rows > 0 ? rows : 1),
                          (cuuint64_t)B};
    cuuint64_t strides[3] = {(cuuint64_t)D * 2, (cuuint64_t)H * D * 2, (cuuint64_t)bstride_bytes};
    cuuint32_t box[4] = {64, 1, (cuuint32_t)kBlockN, 1};
    cuuint32_t es[4] = {1, 1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box,
               es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
           CUDA_SUCCESS;
}

struct TcCache {
    TcMaps maps;
    // what the maps were built from
    const void* key_ptr[2 * kNumMaps + 1];
    int key_rows[2 * kNumMaps + 1];
    bool valid[2 * kNumMaps + 1];
    bool attr_set[2];
};

}  // namespace

void tc_cache_free(msf_plan_t plan) {
    if (plan && plan->tc_cache) {
        free(plan->tc_cache);
        plan->tc_cache = nullptr;
    }
}

void tc_cache_invalidate(msf_plan_t plan) {
    if (plan && plan->tc_cache) {
        TcCache* c = (TcCache*)plan->tc_cache;
        for (int i = 0; i < 2 * kNumMaps + 1; ++i) c->valid[i] = false;
    }
}

msf_status launch_attn_tc(msf_plan_t plan, const AttnArgs& a, cudaStream_t st) {
    Plan& P = *plan;
    if (!P.tc_cache) {
        P.tc_cache = calloc(1, sizeof(TcCache));
        if (!P.tc_cache) return MSF_ERR_INVALID_ARG;
    }
    TcCache& cache = *(TcCache*)P.tc_cache;
    const long long row = (long long)P.H * P.D * 2;

    auto ensure = [&](int slot, CUtensorMap* m, const void* base, int rows, long long bs) -> bool {
        if (cache.valid[slot] && cache.key_ptr[slot] == base && cache.key_rows[slot] == rows)
            return true;
        if (!encode_rows(m, base, P.D, P.H, rows, P.B, bs)) return false;
        cache.valid[slot] = true;
        cache.key_ptr[slot] = base;
        cache.key_rows[slot] = rows;
        return true;
    };

    TcParams tp;
    memset(&tp, 0, sizeof(tp));
    tp.H = P.H;
    tp.B = P.B;
    tp.scale_log2 = a.scale_log2;
    tp.out = (__nv_bfloat16*)a.out;
    tp.out_bstride = (long long)P.N * P.H * P.D;
    tp.status = a.status;
    tp.wait_limit = kWaitLimit;

    if (!ensure(2 * kNumMaps, &cache.maps.q, a.q, P.N, a.q_bstride)) {
        set_cuda_error((int)cudaErrorInvalidValue);
        return MSF_ERR_CUDA;
    }
    // Order groups by context length, longest first (their CTAs start first).
    int order[MSF_MAX_GROUPS];
    for (int i = 0; i < a.n_groups; ++i) order[i] = i;
    for (int i = 0; i < a.n_groups; ++i)
        for (int k = i + 1; k < a.n_groups; ++k) {
            int ni = 0, nk = 0;
            for (int s = 0; s < a.g[order[i]].n_seg; ++s) ni += a.g[order[i]].seg[s].len;
            for (int s = 0; s < a.g[order[k]].n_seg; ++s) nk += a.g[order[k]].seg[s].len;
            if (nk > ni) {
                int tmp = order[i];
                order[i] = order[k];
                order[k] = tmp;
            }
        }
    long long total_items = 0;
    for (int oi = 0; oi < a.n_groups; ++oi) {
        const int gi = order[oi];
        const AttnGroup& ag = a.g[gi];
        TcGroup& tg = tp.g[oi];
        tg.q_begin = ag.q_begin;
        tg.q_end = ag.q_end;
        tg.n_qb = (ag.q_end - ag.q_begin + 2 * kBlockM - 1) / (2 * kBlockM);
        tg.n_items = tg.n_qb * P.H * P.B;
        tg.n_seg = ag.n_seg;
        tg.n_tiles = 0;
        for (int s = 0; s < ag.n_seg; ++s) {
            const Segment& sg = ag.seg[s];
            TcSeg& ts = tg.seg[s];
            int slot = sg.map_id;
            int rows_total = sg.rows_total;
            const char* kb = sg.k;
            const char* vb = sg.v;
            int row0 = sg.row0;
            if (slot == kMapPyr) {
                // per-group map starting at the group's pyramid part, extent = live rows
                slot = kMapPyr0 + gi;
                kb = sg.k + (size_t)sg.row0 * row;
                vb = sg.v + (size_t)sg.row0 * row;
                rows_total = sg.len;
                row0 = 0;
            } else if (slot == kMapHist) {
                rows_total = sg.len;  // live history frames only
            }
            if (!ensure(slot, &cache.maps.k[slot], kb, rows_total, sg.bstride) ||
                !ensure(kNumMaps + slot, &cache.maps.v[slot], vb, rows_total, sg.bstride)) {
                set_cuda_error((int)cudaErrorInvalidValue);
                return MSF_ERR_CUDA;
            }
            ts.map = slot;
            ts.row0 = row0;
            ts.len = sg.len;
            ts.ntiles = (sg.len + kBlockN - 1) / kBlockN;
            tg.n_tiles += ts.ntiles;
        }
        total_items += tg.n_items;
    }
    tp.n_groups = a.n_groups;
    if (total_items == 0) return MSF_OK;
    if (total_items > 0x7fffffffLL) return MSF_ERR_UNSUPPORTED;

    cudaError_t e;
    if (P.D == 128) {
        if (!cache.attr_set[1]) {
            e = cudaFuncSetAttribute(mssa_tc_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     Cfg<128>::kSmem);
            if (e != cudaSuccess) {
                set_cuda_error((int)e);
                return MSF_ERR_CUDA;
            }
            cache.attr_set[1] = true;
        }
        mssa_tc_kernel<128><<<(unsigned)total_items, kThreads, Cfg<128>::kSmem, st>>>(cache.maps, tp);
    } else {
        if (!cache.attr_set[0]) {
            e = cudaFuncSetAttribute(mssa_tc_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     Cfg<64>::kSmem);
            if (e != cudaSuccess) {
                set_cuda_error((int)e);
                return MSF_ERR_CUDA;
            }
            cache.attr_set[0] = true;
        }
        mssa_tc_kernel<64><<<(unsigned)total_items, kThreads, Cfg<64>::kSmem, st>>>(cache.maps, tp);
    }
    e = cudaGetLastError();
    if (e != cudaSuccess) {
        set_cuda_error((int)e);
        return MSF_ERR_CUDA;
    }
    return MSF_OK;
}

}  // namespace msf
