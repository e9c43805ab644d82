// Fused Multi-Scale Patchification kernels on the sm_103a tensor cores
// (Sec. 3.2: a latent state of scale s_l is cut into patches of edge
// P = patch * s_l; Eq. 3 token counts; feature order (c, dy, dx)).
//
// msp_embed_kernel    patchify + tier embedding in one pass. The A operand
//                     (raw patch vectors, K = C*P^2) is gathered from the
//                     latent straight into 128-byte-swizzled shared memory by
//                     four warps, B (the tier's [E, K] weight) arrives by TMA,
//                     and the accumulator is written once as bf16 tokens.
//
// msp_deembed_kernel  de-embedding + unpatchify of one window position,
//                     split-K over a thread-block cluster and reduced over
//                     distributed shared memory (see its section below).
//
// Roles (256 threads): warp 0 TMA producer, warp 1 MMA issuer (one elected
// lane of the converged warp), warp 2 TMEM allocation, warps 4-7 gather and
// epilogue. Every wait is bounded and winds down through the status word.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <string.h>

#include "gemm_tc.h"
#include "kernels.h"
#include "msp_tc.h"
#include "pool.cuh"
#include "ptx.cuh"

namespace msf {

namespace {

constexpr int kThreads = 256;
constexpr long long kWaitLimit = 2000000000LL;
constexpr int kChunkA = 128 * 128;  // 128 rows x 64 bf16 (one K chunk), swizzled
constexpr int kEmbedBN = 256;
constexpr int kEmbedStages = 2;

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

bool encode_2d(CUtensorMap* m, const void* base, int inner, int outer, long long stride_bytes,
               int box_inner, int box_outer) {
    EncodeTiledFn enc = encoder();
    if (!enc) return false;
    cuuint64_t dims[2] = {(cuuint64_t)inner, (cuuint64_t)outer};
    cuuint64_t strides[1] = {(cuuint64_t)stride_bytes};
    cuuint32_t box[2] = {(cuuint32_t)box_inner, (cuuint32_t)box_outer};
    cuuint32_t es[2] = {1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Byte offset of bf16 element (row, k) inside one 128-row x 64-column K chunk
// in the 128-byte swizzle layout the tensor core and TMA use: rows are 128
// bytes, eight rows form a 1024-byte atom, and the 16-byte unit index is
// XOR-ed with the row's position in its atom.
__device__ __forceinline__ uint32_t swz_offset(int row, int k) {
    const int byte = k * 2;
    return (uint32_t)((row >> 3) * 1024 + (row & 7) * 128 + (((byte >> 4) ^ (row & 7)) << 4) + (byte & 15));
}

// ----------------------------------------------------------------- embedding

// Features [64 kc, 64 kc + 64) of one token row in (c, dy, dx) order: 64 / P
// runs of P pixels, each run one row segment of one channel. The loads and the
// stores are apart, so a row's next chunk can be in flight while the current
// one waits for its stage.
template <int P, typename V>
__device__ __forceinline__ void load_chunk(V (&v)[64 / P], const __nv_bfloat16* base, size_t plane, int Wl,
                                           int kc, bool valid) {
#pragma unroll
    for (int g = 0; g < 64 / P; ++g) {
        const int f0 = kc * 64 + g * P;
        const int c = f0 / (P * P), dy = (f0 % (P * P)) / P;
        if (valid)
            v[g] = __ldg(reinterpret_cast<const V*>(base + c * plane + (size_t)dy * Wl));
        else
            memset(&v[g], 0, sizeof(V));
    }
}
template <int P, typename V>
__device__ __forceinline__ void store_chunk(unsigned char* dst, const V (&v)[64 / P], int r) {
#pragma unroll
    for (int g = 0; g < 64 / P; ++g) *reinterpret_cast<V*>(dst + swz_offset(r, g * P)) = v[g];
}

// Every K chunk of one token row into the A ring, each chunk's loads issued
// before the wait for the previous chunk's stage, so that the L2 round trips
// of consecutive chunks overlap. Returns false if a wait gave up.
template <int P, typename V>
__device__ __forceinline__ bool gather_row(unsigned char* sA, uint64_t* a_full, uint64_t* a_empty,
                                           const __nv_bfloat16* base, size_t plane, int Wl, int r, int nk,
                                           bool valid, volatile int* abort_p) {
    V cur[64 / P], nxt[64 / P];
    load_chunk<P, V>(cur, base, plane, Wl, 0, valid);
    for (int kc = 0; kc < nk; ++kc) {
        if (kc + 1 < nk) load_chunk<P, V>(nxt, base, plane, Wl, kc + 1, valid);
        const int st = kc % kEmbedStages;
        const uint32_t ph = (uint32_t)((kc / kEmbedStages) & 1);
        const bool ok = __all_sync(0xffffffffu, ptx::mbar_wait_bounded(&a_empty[st], ph ^ 1u, abort_p, kWaitLimit));
        if (!ok) return false;
        store_chunk<P, V>(sA + st * kChunkA, cur, r);
        ptx::fence_proxy_async_smem();  // the tensor core reads through the async proxy
        ptx::mbar_arrive(&a_full[st]);
#pragma unroll
        for (int g = 0; g < 64 / P; ++g) cur[g] = nxt[g];
    }
    return true;
}

struct EmbedRun {
    int tile_base;  // first CTA of this run in blockIdx.x
    int m_tiles;
    int M;          // tokens of the run (per stream)
    int l0;         // first state of the run
    int n_l;        // tokens per state
    int gw;         // tokens per grid row (Wl / P)
    int P;          // patch edge in latent pixels
    int K;          // C * P * P
    int tok_off;    // first token row of the run in the output
    int lora;       // 1: one more K chunk (LoRA codes x up projection)
    float scale;    // accumulator scale
};
struct EmbedParams {
    int n_runs;
    EmbedRun run[kMaxGemmProblems];
    int T, C, Hl, Wl, E;
    int n_tiles_n;  // 256-column tiles per 128-row tile: ceil(E / 256)
    int n_embed_tiles;  // CTAs [0, n_embed_tiles) of a stream embed; the rest pool
    int pool_ctas;      // CTAs per stream that run the pyramid jobs (0: none)
    int pool_tasks;     // vector-pair tasks per pyramid job
    const __nv_bfloat16* latent;  // [B, T, C, Hl, Wl]
    __nv_bfloat16* tokens;        // [B, N, E]
    long long tok_bstride;        // elements
    unsigned int* status;
};
struct EmbedMaps {
    CUtensorMap w[kMaxGemmProblems];      // [E, K] weight of each run: dims {K, E}
    CUtensorMap out[kMaxGemmProblems];    // the run's tokens: dims {E, M, B}, rows past M clipped
    CUtensorMap codes[kMaxGemmProblems];  // LoRA codes of the run's tokens: dims {64, M, B}
    CUtensorMap up[kMaxGemmProblems];     // LoRA up projection [E, r]: dims {r, E}
};

// 128 tokens x 256 embedding columns per CTA (one N=256 MMA per K step, half
// the gathers of 128-column tiles); two CTAs per SM (97 KB of shared memory
// each), so the 480p window's 210 tiles run in one wave on 152 SMs.
__global__ void __launch_bounds__(kThreads, 2)
    msp_embed_kernel(const __grid_constant__ EmbedMaps maps, const __grid_constant__ EmbedParams p,
                     const __grid_constant__ PoolBatch pool) {
    if ((int)blockIdx.x >= p.n_embed_tiles) {
        // ---- K/V pyramid jobs in the CTAs after the embedding tiles (the
        // longest tiles, those of the runs with the most K chunks, come
        // first): the same per-thread pooling as pool_kernel, one task per
        // thread. The two parts read and write disjoint buffers; the block
        // scheduler starts these CTAs in the slots the embedding leaves free
        // and, as its short tiles finish, in theirs.
        ptx::grid_dep_wait();
        ptx::grid_dep_launch();
        const int stride = p.pool_ctas * kThreads;
        const int total = pool.n * p.pool_tasks;
        for (int t = ((int)blockIdx.x - p.n_embed_tiles) * kThreads + (int)threadIdx.x; t < total; t += stride)
            pool_task<__nv_bfloat16>(pool, t / p.pool_tasks, blockIdx.z, t % p.pool_tasks);
        return;
    }
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    unsigned char* smem = (unsigned char*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    unsigned char* sA = smem;                                   // [stage][chunk]
    unsigned char* sB = smem + kEmbedStages * kChunkA;          // [stage][BN rows x 128 B]
    constexpr int kBBytes = kEmbedBN * 128;
    __shared__ uint64_t a_full[kEmbedStages], a_empty[kEmbedStages];
    __shared__ uint64_t b_full[kEmbedStages], b_empty[kEmbedStages], acc_full;
    __shared__ uint32_t tmem_base_sh;
    __shared__ int abort_flag;

    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const int tile = (int)blockIdx.x;
    int ri = 0;
    while (ri < p.n_runs - 1 && tile >= p.run[ri + 1].tile_base) ++ri;
    const EmbedRun& R = p.run[ri];
    const int local = tile - R.tile_base;
    const int mt = local % R.m_tiles, nt = local / R.m_tiles;
    const int b = blockIdx.z;
    const int nk_patch = R.K / 64;      // chunks gathered from the latent
    const int nk = nk_patch + R.lora;   // plus the LoRA chunk

    if (threadIdx.x == 0) {
        abort_flag = 0;
        for (int s = 0; s < kEmbedStages; ++s) {
            ptx::mbar_init(&a_full[s], 128);  // one arrival per gathering thread
            ptx::mbar_init(&a_empty[s], 1);
            ptx::mbar_init(&b_full[s], 1);
            ptx::mbar_init(&b_empty[s], 1);
        }
        ptx::mbar_init(&acc_full, 1);
        ptx::fence_mbar_init();
    }
    if (warp == 2) {
        ptx::tmem_alloc(&tmem_base_sh, kEmbedBN);
        ptx::tmem_relinquish();
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tbase = tmem_base_sh;
    volatile int* abort_p = &abort_flag;
    volatile int never = 0;
    ptx::grid_dep_wait();  // the latent and weights written before are visible
    ptx::grid_dep_launch();

    if (warp == 0) {
        if (lane == 0) {
            ptx::prefetch_tmap(&maps.w[ri]);
            int issued = 0;
            bool ok = true;
            for (int kc = 0; kc < nk; ++kc) {
                const int st = kc % kEmbedStages;
                const uint32_t ph = (uint32_t)((kc / kEmbedStages) & 1);
                if (!ptx::mbar_wait_bounded(&b_empty[st], ph ^ 1u, abort_p, kWaitLimit)) {
                    ok = false;
                    break;
                }
                ptx::mbar_arrive_expect_tx(&b_full[st], kBBytes);
                if (kc < nk_patch)
                    ptx::tma_load_2d(sB + st * kBBytes, &maps.w[ri], &b_full[st], kc * 64, nt * kEmbedBN);
                else
                    ptx::tma_load_2d(sB + st * kBBytes, &maps.up[ri], &b_full[st], 0, nt * kEmbedBN);
                ++issued;
            }
            if (!ok) {
                for (int kc = (issued > kEmbedStages ? issued - kEmbedStages : 0); kc < issued; ++kc)
                    ptx::mbar_wait_bounded(&b_full[kc % kEmbedStages],
                                           (uint32_t)((kc / kEmbedStages) & 1), &never, kWaitLimit);
                atomicOr(p.status, kDevTimeout);
            }
        }
    } else if (warp == 1) {
        constexpr uint32_t idesc = ptx::idesc_bf16(128, kEmbedBN, false, false);
        const uint64_t a_desc = ptx::sdesc_sw128(ptx::smem_u32(sA), 16, 1024);
        const uint64_t b_desc = ptx::sdesc_sw128(ptx::smem_u32(sB), 16, 1024);
        bool ok = true;
        for (int kc = 0; kc < nk && ok; ++kc) {
            const int st = kc % kEmbedStages;
            const uint32_t ph = (uint32_t)((kc / kEmbedStages) & 1);
            const bool ra = ptx::mbar_wait_bounded(&a_full[st], ph, abort_p, kWaitLimit);
            const bool rb = ra && ptx::mbar_wait_bounded(&b_full[st], ph, abort_p, kWaitLimit);
            ok = __all_sync(0xffffffffu, rb);
            if (!ok) break;
            ptx::tc_fence_after();
            if (ptx::elect_one_sync()) {
                const uint64_t ad = a_desc + (uint64_t)(st * (kChunkA >> 4));
                const uint64_t bd = b_desc + (uint64_t)(st * (kBBytes >> 4));
#pragma unroll
                for (int kk = 0; kk < 4; ++kk)
                    ptx::mma_ss(tbase, ad + (uint64_t)(kk * 2), bd + (uint64_t)(kk * 2), idesc,
                                (kc > 0 || kk > 0) ? 1u : 0u);
                ptx::mma_commit(&a_empty[st]);
                ptx::mma_commit(&b_empty[st]);
            }
            __syncwarp();
        }
        if (ptx::elect_one_sync()) ptx::mma_commit(&acc_full);  // also after an abort: drains the MMAs
        __syncwarp();
        if (!ok && lane == 0) atomicOr(p.status, kDevTimeout);
    } else if (warp >= 4) {
        // ---- gather: one token row per thread
        const int r = (warp - 4) * 32 + lane;
        const int m = mt * 128 + r;
        const bool valid = m < R.M;
        const int P = R.P;
        const __nv_bfloat16* base = p.latent;
        if (valid) {
            const int l = R.l0 + m / R.n_l;
            const int loc = m % R.n_l;
            const int i = loc / R.gw, jj = loc % R.gw;
            base = p.latent + ((size_t)b * p.T + l) * p.C * p.Hl * p.Wl + (size_t)(P * i) * p.Wl + P * jj;
        }
        const size_t plane = (size_t)p.Hl * p.Wl;
        bool ok = true;
        if (P == 2) {
            ok = gather_row<2, uint32_t>(sA, a_full, a_empty, base, plane, p.Wl, r, nk_patch, valid, abort_p);
        } else if (P == 4) {
            ok = gather_row<4, uint2>(sA, a_full, a_empty, base, plane, p.Wl, r, nk_patch, valid, abort_p);
        } else if (P == 8) {
            ok = gather_row<8, uint4>(sA, a_full, a_empty, base, plane, p.Wl, r, nk_patch, valid, abort_p);
        } else for (int kc = 0; kc < nk_patch; ++kc) {
            const int st = kc % kEmbedStages;
            const uint32_t ph = (uint32_t)((kc / kEmbedStages) & 1);
            ok = ptx::mbar_wait_bounded(&a_empty[st], ph ^ 1u, abort_p, kWaitLimit);
            ok = __all_sync(0xffffffffu, ok);
            if (!ok) break;
            unsigned char* dst = sA + st * kChunkA;
            {
                for (int g = 0; g < 64 / P; ++g) {
                    const int f0 = kc * 64 + g * P;
                    const int c = f0 / (P * P), dy = (f0 % (P * P)) / P;
                    const __nv_bfloat16* src = base + c * plane + (size_t)dy * p.Wl;
                    for (int x = 0; x < P; ++x)
                        *reinterpret_cast<__nv_bfloat16*>(dst + swz_offset(r, g * P + x)) =
                            valid ? src[x] : __float2bfloat16(0.f);
                }
            }
            ptx::fence_proxy_async_smem();  // the tensor core reads through the async proxy
            ptx::mbar_arrive(&a_full[st]);
        }
        if (ok && R.lora) {
            // ---- LoRA chunk: the 128 rows' codes arrive by TMA into the A
            // stage; one thread adds the bytes to the stage's barrier, the
            // others arrive as for a gathered chunk.
            const int st = nk_patch % kEmbedStages;
            const uint32_t ph = (uint32_t)((nk_patch / kEmbedStages) & 1);
            ok = __all_sync(0xffffffffu, ptx::mbar_wait_bounded(&a_empty[st], ph ^ 1u, abort_p, kWaitLimit));
            if (ok) {
                if (r == 0) {
                    ptx::mbar_arrive_expect_tx(&a_full[st], kChunkA);
                    ptx::tma_load_3d(sA + st * kChunkA, &maps.codes[ri], &a_full[st], 0, mt * 128, b);
                } else {
                    ptx::mbar_arrive(&a_full[st]);
                }
            }
        }
        // ---- epilogue: bf16 tile staged in the (now idle) A and B stages in
        // the 128-byte swizzle layout, then TMA stores of 128 rows x 64 columns.
        ok = ok && ptx::mbar_wait_bounded(&acc_full, 0, abort_p, kWaitLimit);
        ok = __all_sync(0xffffffffu, ok);
        if (ok) {
            ptx::tc_fence_after();
            const uint32_t taddr = tbase + ((uint32_t)((warp - 4) * 32) << 16);
#pragma unroll 1
            for (int c = 0; c < kEmbedBN / 32; ++c) {
                uint32_t v[32];
                ptx::tmem_ld32(taddr + c * 32, v);
                ptx::tmem_wait_ld();
                unsigned char* stage = sA + (c / 2) * kChunkA;
                const float sc = R.scale;
#pragma unroll
                for (int e = 0; e < 4; ++e)
                    *reinterpret_cast<uint4*>(stage + swz_offset(r, (c % 2) * 32 + 8 * e)) = make_uint4(
                        ptx::pack_bf16(sc * __uint_as_float(v[8 * e]), sc * __uint_as_float(v[8 * e + 1])),
                        ptx::pack_bf16(sc * __uint_as_float(v[8 * e + 2]), sc * __uint_as_float(v[8 * e + 3])),
                        ptx::pack_bf16(sc * __uint_as_float(v[8 * e + 4]), sc * __uint_as_float(v[8 * e + 5])),
                        ptx::pack_bf16(sc * __uint_as_float(v[8 * e + 6]), sc * __uint_as_float(v[8 * e + 7])));
            }
            ptx::fence_proxy_async_smem();
        }
        // The four epilogue warps meet before one thread stores the tile.
        ok = ptx::named_bar_and(1, 128, ok);
        if (ok && warp == 4 && lane == 0) {
            for (int h = 0; h < kEmbedBN / 64 && nt * kEmbedBN + h * 64 < p.E; ++h)
                ptx::tma_store_3d(&maps.out[ri], sA + h * kChunkA, nt * kEmbedBN + h * 64, mt * 128, b);
            ptx::bulk_commit();
            ptx::bulk_wait_read_all();
        }
        if (!ok && lane == 0) atomicOr(p.status, kDevTimeout);
    }
    ptx::tc_fence_before();
    __syncthreads();
    if (warp == 2) {
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tbase, kEmbedBN);
    }
}


// ------------------------------------------------------------ de-embedding
//
// msp_deembed_kernel: de-embedding + unpatchify of one window position. The
// K = E contraction is split over the S CTAs of a thread-block cluster
// (S <= 8 divides 128). Each CTA leaves its fp32 partial 128 x 64 tile in its
// own shared memory; after a cluster barrier CTA r sums rows [r*128/S,
// (r+1)*128/S) of all S partials in split order over distributed shared
// memory, rounds once to bf16 and scatters them into the latent layout
// [B, C, Hl, Wl]. No partial sums go through global memory and no second
// kernel is needed.

constexpr int kDeBN = 64;
constexpr int kDeStages = 4;
constexpr int kDeMaxSplits = 8;  // cluster size along the split (portable limit)
constexpr int kDePartStride = kDeBN + 4;  // floats per staged row (padding spreads the banks)

struct DeembedParams {
    int M;              // tokens of the position (per stream)
    int K;              // embedding width E
    int nk_all;         // K chunks: E / 64 token chunks, then the tier's extras
    int lora;           // 1: chunk E/64 is (LoRA codes, up projection)
    int nk_res;         // then this many (raw patch vector, latent residual) chunks
    int m_tiles;
    int splits;         // cluster size along y
    int P, gw, C, Hl, Wl;
    int tok_row0;       // first token row of the position
    __nv_bfloat16* latent;  // [B, C, Hl, Wl]
    unsigned int* status;
    // Row output instead of the latent scatter (NULL: scatter): row m of
    // stream b, columns [0, F), at rows_out + b * rows_bstride + m * rows_ld,
    // each value scaled by rows_scale before the one rounding.
    __nv_bfloat16* rows_out;
    long long rows_bstride;
    int rows_ld;
    float rows_scale;
};
struct DeembedMaps {
    CUtensorMap a;      // tokens {E, rows, B}
    CUtensorMap b;      // W_out {E, F}
    CUtensorMap codes;  // LoRA codes of the tokens {64, rows, B}
    CUtensorMap up;     // LoRA up projection [F, r]: {r, F}
    CUtensorMap xraw;   // the state's raw patch vectors {F, M, B}
    CUtensorMap res;    // latent residual [F, F]: {F, F}
};

__global__ void __launch_bounds__(kThreads, 1)
    msp_deembed_kernel(const __grid_constant__ DeembedMaps maps, const __grid_constant__ DeembedParams p) {
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    unsigned char* smem = (unsigned char*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    constexpr int kBBytes = kDeBN * 128;
    constexpr int kStageBytes = kChunkA + kBBytes;
    float* part = reinterpret_cast<float*>(smem);  // reuses the ring once every MMA is done
    __shared__ uint64_t full[kDeStages], empty[kDeStages], acc_full;
    __shared__ uint32_t tmem_base_sh;
    __shared__ int abort_flag;

    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const int tile = blockIdx.x;
    const int mt = tile % p.m_tiles, nt = tile / p.m_tiles;
    const int split = (int)ptx::cluster_rank();
    const int b = blockIdx.z;
    const int nk_all = p.nk_all;
    const int nk_tok = p.K / 64;
    const int kc0 = (int)((long long)split * nk_all / p.splits);
    const int nk = (int)((long long)(split + 1) * nk_all / p.splits) - kc0;

    if (threadIdx.x == 0) {
        abort_flag = 0;
        for (int s = 0; s < kDeStages; ++s) {
            ptx::mbar_init(&full[s], 1);
            ptx::mbar_init(&empty[s], 1);
        }
        ptx::mbar_init(&acc_full, 1);
        ptx::fence_mbar_init();
    }
    if (warp == 2) {
        ptx::tmem_alloc(&tmem_base_sh, kDeBN);
        ptx::tmem_relinquish();
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tbase = tmem_base_sh;
    volatile int* abort_p = &abort_flag;
    volatile int never = 0;
    ptx::grid_dep_wait();  // the tokens written by the attention kernel are visible
    ptx::grid_dep_launch();

    bool ok = true;
    if (warp == 0) {
        if (lane == 0) {
            ptx::prefetch_tmap(&maps.a);
            ptx::prefetch_tmap(&maps.b);
            int issued = 0;
            for (int kc = 0; kc < nk; ++kc) {
                const int st = kc % kDeStages;
                const uint32_t ph = (uint32_t)((kc / kDeStages) & 1);
                if (!ptx::mbar_wait_bounded(&empty[st], ph ^ 1u, abort_p, kWaitLimit)) {
                    ok = false;
                    break;
                }
                unsigned char* sa = smem + st * kStageBytes;
                ptx::mbar_arrive_expect_tx(&full[st], kStageBytes);
                const int g = kc0 + kc;
                if (g < nk_tok) {
                    ptx::tma_load_3d(sa, &maps.a, &full[st], g * 64, p.tok_row0 + mt * 128, b);
                    ptx::tma_load_2d(sa + kChunkA, &maps.b, &full[st], g * 64, nt * kDeBN);
                } else if (g == nk_tok && p.lora) {
                    ptx::tma_load_3d(sa, &maps.codes, &full[st], 0, p.tok_row0 + mt * 128, b);
                    ptx::tma_load_2d(sa + kChunkA, &maps.up, &full[st], 0, nt * kDeBN);
                } else {
                    const int j = g - nk_tok - p.lora;
                    ptx::tma_load_3d(sa, &maps.xraw, &full[st], j * 64, mt * 128, b);
                    ptx::tma_load_2d(sa + kChunkA, &maps.res, &full[st], j * 64, nt * kDeBN);
                }
                ++issued;
            }
            if (!ok) {
                for (int kc = (issued > kDeStages ? issued - kDeStages : 0); kc < issued; ++kc)
                    ptx::mbar_wait_bounded(&full[kc % kDeStages], (uint32_t)((kc / kDeStages) & 1), &never,
                                           kWaitLimit);
                atomicOr(p.status, kDevTimeout);
            }
        }
    } else if (warp == 1) {
        constexpr uint32_t idesc = ptx::idesc_bf16(128, kDeBN, false, false);
        const uint64_t desc0 = ptx::sdesc_sw128(ptx::smem_u32(smem), 16, 1024);
        for (int kc = 0; kc < nk && ok; ++kc) {
            const int st = kc % kDeStages;
            const uint32_t ph = (uint32_t)((kc / kDeStages) & 1);
            ok = __all_sync(0xffffffffu, ptx::mbar_wait_bounded(&full[st], ph, abort_p, kWaitLimit));
            if (!ok) break;
            ptx::tc_fence_after();
            if (ptx::elect_one_sync()) {
                const uint64_t ad = desc0 + (uint64_t)(st * (kStageBytes >> 4));
                const uint64_t bd = ad + (uint64_t)(kChunkA >> 4);
#pragma unroll
                for (int kk = 0; kk < 4; ++kk)
                    ptx::mma_ss(tbase, ad + (uint64_t)(kk * 2), bd + (uint64_t)(kk * 2), idesc,
                                (kc > 0 || kk > 0) ? 1u : 0u);
                ptx::mma_commit(&empty[st]);
            }
            __syncwarp();
        }
        if (ptx::elect_one_sync()) ptx::mma_commit(&acc_full);  // also after an abort: drains the MMAs
        __syncwarp();
        if (!ok && lane == 0) atomicOr(p.status, kDevTimeout);
    } else if (warp >= 4) {
        // ---- this split's partial tile into shared memory (row-major, padded rows)
        const int r = (warp - 4) * 32 + lane;
        ok = __all_sync(0xffffffffu, ptx::mbar_wait_bounded(&acc_full, 0, abort_p, kWaitLimit));
        if (ok) {
            ptx::tc_fence_after();
            const uint32_t taddr = tbase + ((uint32_t)((warp - 4) * 32) << 16);
            uint32_t vb[kDeBN / 32][32];
#pragma unroll
            for (int c = 0; c < kDeBN / 32; ++c) ptx::tmem_ld32(taddr + c * 32, vb[c]);
            ptx::tmem_wait_ld();
#pragma unroll
            for (int c = 0; c < kDeBN / 32; ++c) {
                const uint32_t* v = vb[c];
                float4* d4 = reinterpret_cast<float4*>(part + r * kDePartStride + c * 32);
#pragma unroll
                for (int e = 0; e < 8; ++e)
                    d4[e] = make_float4(__uint_as_float(v[4 * e]), __uint_as_float(v[4 * e + 1]),
                                        __uint_as_float(v[4 * e + 2]), __uint_as_float(v[4 * e + 3]));
            }
        } else if (lane == 0) {
            atomicOr(p.status, kDevTimeout);
        }
    }
    // Every thread of every CTA of the cluster: partials are staged.
    __syncwarp();
    ptx::tc_fence_before();
    ptx::cluster_sync();
    {
        // ---- rows [rank*R, rank*R + R) of the tile: sum the S partials in
        // split order, round once, scatter into the latent.
        const int R = 128 / p.splits;             // rows per CTA
        const int per_row = kDeBN / 4;            // float4 per row
        const int P = p.P, PP = P * P;
        const size_t plane = (size_t)p.Hl * p.Wl;
        for (int q = threadIdx.x; q < R * per_row; q += kThreads) {
            const int row = split * R + q / per_row;
            const int c4 = q % per_row;
            const int m = mt * 128 + row;
            // All splits' partials requested before the first add (remote
            // shared-memory loads are independent), summed in split order.
            float4 v[kDeMaxSplits];
#pragma unroll
            for (int sp = 0; sp < kDeMaxSplits; ++sp)
                v[sp] = sp < p.splits ? ptx::ld_cluster_f4(part + row * kDePartStride + 4 * c4, (uint32_t)sp)
                                      : make_float4(0.f, 0.f, 0.f, 0.f);
            float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
            for (int sp = 0; sp < kDeMaxSplits; ++sp) {
                acc.x += v[sp].x;
                acc.y += v[sp].y;
                acc.z += v[sp].z;
                acc.w += v[sp].w;
            }
            if (m < p.M && p.rows_out) {
                const float sc = p.rows_scale;
                uint2 v2;
                v2.x = ptx::pack_bf16(sc * acc.x, sc * acc.y);
                v2.y = ptx::pack_bf16(sc * acc.z, sc * acc.w);
                *reinterpret_cast<uint2*>(p.rows_out + (size_t)b * p.rows_bstride + (size_t)m * p.rows_ld +
                                          nt * kDeBN + 4 * c4) = v2;
            } else if (m < p.M) {
                const int i = m / p.gw, jj = m % p.gw;
                __nv_bfloat16* lat =
                    p.latent + (size_t)b * p.C * plane + (size_t)(P * i) * p.Wl + (size_t)P * jj;
                const float vals[4] = {acc.x, acc.y, acc.z, acc.w};
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const int f = nt * kDeBN + 4 * c4 + e;
                    const int ch = f / PP, dy = (f % PP) / P, dx = f % P;
                    lat[(size_t)ch * plane + (size_t)dy * p.Wl + dx] = __float2bfloat16_rn(vals[e]);
                }
            }
        }
    }
    // No CTA leaves while another may still read its shared memory.
    ptx::cluster_sync();
    __syncthreads();
    if (warp == 2) {
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tbase, kDeBN);
    }
}

constexpr int kDeSmem = kDeStages * (kChunkA + kDeBN * 128) + 1024;
static_assert(128 * kDePartStride * 4 <= kDeStages * (kChunkA + kDeBN * 128), "partial tile fits the ring");

constexpr int kEmbedSmem = kEmbedStages * (kChunkA + kEmbedBN * 128) + 1024;

}  // namespace

bool msp_embed_supported(const MspEmbedRun* runs, int n, int E) {
    if (n < 1 || n > kMaxGemmProblems || E % 64 != 0 || E <= 0) return false;
    for (int i = 0; i < n; ++i) {
        const MspEmbedRun& r = runs[i];
        if (r.K % 64 != 0 || r.P < 1 || 64 % r.P != 0 || ((uintptr_t)r.w & 15) || r.M <= 0) return false;
        if (r.w_rows < 0 || r.w_rows > E) return false;
        if (r.lora_up && (r.rank < 8 || r.rank > 64 || r.rank % 8 != 0 || !r.codes ||
                          ((uintptr_t)r.lora_up & 15) || ((uintptr_t)r.codes & 15) || r.codes_bstride % 8))
            return false;
    }
    return true;
}

cudaError_t launch_msp_embed(const MspEmbedRun* runs, int n, const MspShape& sh, int E, const void* latent,
                             void* tokens, long long tok_bstride, int batch, unsigned int* status,
                             cudaStream_t st, const PoolBatch* pool, int pool_ctas) {
    EmbedMaps maps;
    memset(&maps, 0, sizeof(maps));
    EmbedParams p;
    memset(&p, 0, sizeof(p));
    int tiles = 0;
    for (int i = 0; i < n; ++i) {
        const MspEmbedRun& r = runs[i];
        if (!encode_2d(&maps.w[i], r.w, r.K, r.w_rows > 0 ? r.w_rows : E, (long long)r.K * 2, 64, kEmbedBN))
            return cudaErrorInvalidValue;
        if (r.lora_up) {
            EncodeTiledFn enc = encoder();
            if (!encode_2d(&maps.up[i], r.lora_up, r.rank, E, (long long)r.rank * 2, 64, kEmbedBN))
                return cudaErrorInvalidValue;
            cuuint64_t dims[3] = {64, (cuuint64_t)r.M, (cuuint64_t)batch};
            cuuint64_t strides[2] = {128, (cuuint64_t)r.codes_bstride * 2};
            cuuint32_t box[3] = {64, 128, 1};
            cuuint32_t es[3] = {1, 1, 1};
            if (!enc || enc(&maps.codes[i], CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(r.codes), dims,
                            strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
                return cudaErrorInvalidValue;
        }
        {
            EncodeTiledFn enc = encoder();
            cuuint64_t dims[3] = {(cuuint64_t)E, (cuuint64_t)r.M, (cuuint64_t)batch};
            cuuint64_t strides[2] = {(cuuint64_t)E * 2, (cuuint64_t)tok_bstride * 2};
            cuuint32_t box[3] = {64, 128, 1};
            cuuint32_t es[3] = {1, 1, 1};
            if (!enc || enc(&maps.out[i], CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3,
                            (char*)tokens + (size_t)r.tok_off * E * 2, dims, strides, box, es,
                            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
                return cudaErrorInvalidValue;
        }
        EmbedRun& R = p.run[i];
        R.tile_base = tiles;
        R.m_tiles = (r.M + 127) / 128;
        R.M = r.M;
        R.l0 = r.l0;
        R.n_l = r.n_l;
        R.gw = r.gw;
        R.P = r.P;
        R.K = r.K;
        R.tok_off = r.tok_off;
        R.lora = r.lora_up ? 1 : 0;
        R.scale = r.scale;
        tiles += R.m_tiles * ((E + kEmbedBN - 1) / kEmbedBN);
    }
    p.n_tiles_n = (E + kEmbedBN - 1) / kEmbedBN;
    p.n_runs = n;
    p.T = sh.T;
    p.C = sh.C;
    p.Hl = sh.Hl;
    p.Wl = sh.Wl;
    p.E = E;
    p.latent = (const __nv_bfloat16*)latent;
    p.tokens = (__nv_bfloat16*)tokens;
    p.tok_bstride = tok_bstride;
    p.status = status;
    cudaError_t e = set_smem_attr((const void*)msp_embed_kernel, kEmbedSmem, 100);
    if (e != cudaSuccess) return e;
    p.n_embed_tiles = tiles;
    PoolBatch pb;
    if (pool && pool->n > 0) {
        pb = *pool;
        int max_n = 0;
        for (int k = 0; k < pb.n; ++k) max_n = pb.j[k].out_n > max_n ? pb.j[k].out_n : max_n;
        p.pool_tasks = max_n * (pb.row_vecs / 2);
        p.pool_ctas = pool_ctas > 0 ? pool_ctas : 1;
    } else {
        memset(&pb, 0, sizeof(pb));
    }
    return launch_pdl(msp_embed_kernel, dim3((unsigned)(tiles + p.pool_ctas), 1, (unsigned)batch), dim3(kThreads),
                      kEmbedSmem, st, maps, p, pb);
}


bool msp_deembed_supported(int M, int F, int E) {
    return M > 0 && F % kDeBN == 0 && E % 64 == 0 && E >= 64;
}

cudaError_t launch_msp_deembed(const void* tokens, long long tok_bstride_elems, int tok_rows, int tok_row0,
                               const void* w_out, int M, int F, int E, const MspShape& sh, int P, void* latent,
                               int batch, unsigned int* status, cudaStream_t st, const DeembedTier* tier) {
    DeembedMaps maps;
    memset(&maps, 0, sizeof(maps));
    EncodeTiledFn enc = encoder();
    if (!enc) return cudaErrorNotSupported;
    {
        cuuint64_t dims[3] = {(cuuint64_t)E, (cuuint64_t)tok_rows, (cuuint64_t)batch};
        cuuint64_t strides[2] = {(cuuint64_t)E * 2, (cuuint64_t)tok_bstride_elems * 2};
        cuuint32_t box[3] = {64, 128, 1};
        cuuint32_t es[3] = {1, 1, 1};
        if (enc(&maps.a, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(tokens), dims, strides, box, es,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return cudaErrorInvalidValue;
    }
    if (!encode_2d(&maps.b, w_out, E, F, (long long)E * 2, 64, kDeBN)) return cudaErrorInvalidValue;
    const bool lora = tier && tier->up;
    const bool res = tier && tier->residual;
    if (lora) {
        EncodeTiledFn enc = encoder();
        cuuint64_t dims[3] = {64, (cuuint64_t)tok_rows, (cuuint64_t)batch};
        cuuint64_t strides[2] = {128, (cuuint64_t)tier->codes_bstride * 2};
        cuuint32_t box[3] = {64, 128, 1};
        cuuint32_t es[3] = {1, 1, 1};
        if (!enc || enc(&maps.codes, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(tier->codes), dims,
                        strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return cudaErrorInvalidValue;
        if (!encode_2d(&maps.up, tier->up, tier->rank, F, (long long)tier->rank * 2, 64, kDeBN))
            return cudaErrorInvalidValue;
    }
    if (res) {
        EncodeTiledFn enc = encoder();
        cuuint64_t dims[3] = {(cuuint64_t)F, (cuuint64_t)M, (cuuint64_t)batch};
        cuuint64_t strides[2] = {(cuuint64_t)F * 2, (cuuint64_t)tier->xraw_bstride * 2};
        cuuint32_t box[3] = {64, 128, 1};
        cuuint32_t es[3] = {1, 1, 1};
        if (!enc || enc(&maps.xraw, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(tier->xraw), dims,
                        strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return cudaErrorInvalidValue;
        if (!encode_2d(&maps.res, tier->residual, F, F, (long long)F * 2, 64, kDeBN)) return cudaErrorInvalidValue;
    }
    const int nk_all = E / 64 + (lora ? 1 : 0) + (res ? F / 64 : 0);
    // The largest power of two <= 8 that leaves each split at least one K chunk.
    int splits = 8;
    while (splits > 1 && splits > nk_all) splits /= 2;
    DeembedParams p;
    memset(&p, 0, sizeof(p));
    p.M = M;
    p.K = E;
    p.nk_all = nk_all;
    p.lora = lora ? 1 : 0;
    p.nk_res = res ? F / 64 : 0;
    p.m_tiles = (M + 127) / 128;
    p.splits = splits;
    p.P = P;
    p.gw = sh.Wl / P;
    p.C = sh.C;
    p.Hl = sh.Hl;
    p.Wl = sh.Wl;
    p.tok_row0 = tok_row0;
    p.latent = (__nv_bfloat16*)latent;
    p.status = status;
    cudaError_t e = set_smem_attr((const void*)msp_deembed_kernel, kDeSmem);
    if (e != cudaSuccess) return e;
    const dim3 grid((unsigned)(p.m_tiles * (F / kDeBN)), (unsigned)splits, (unsigned)batch);
    return launch_pdl_cluster(msp_deembed_kernel, grid, dim3(kThreads), kDeSmem, st, dim3(1, splits, 1), maps, p);
}

cudaError_t launch_msp_rows_splitk(const void* tokens, long long tok_bstride_elems, int tok_rows, int tok_row0,
                                   const void* w, int w_rows, int M, int E, void* out, long long out_bstride,
                                   int out_ld, float scale, int batch, unsigned int* status, cudaStream_t st) {
    DeembedMaps maps;
    memset(&maps, 0, sizeof(maps));
    EncodeTiledFn enc = encoder();
    if (!enc) return cudaErrorNotSupported;
    {
        cuuint64_t dims[3] = {(cuuint64_t)E, (cuuint64_t)tok_rows, (cuuint64_t)batch};
        cuuint64_t strides[2] = {(cuuint64_t)E * 2, (cuuint64_t)tok_bstride_elems * 2};
        cuuint32_t box[3] = {64, 128, 1};
        cuuint32_t es[3] = {1, 1, 1};
        if (enc(&maps.a, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(tokens), dims, strides, box, es,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return cudaErrorInvalidValue;
    }
    if (!encode_2d(&maps.b, w, E, w_rows, (long long)E * 2, 64, kDeBN)) return cudaErrorInvalidValue;
    const int nk_all = E / 64;
    int splits = 8;
    while (splits > 1 && splits > nk_all) splits /= 2;
    DeembedParams p;
    memset(&p, 0, sizeof(p));
    p.M = M;
    p.K = E;
    p.nk_all = nk_all;
    p.m_tiles = (M + 127) / 128;
    p.splits = splits;
    p.P = 1;
    p.gw = 1;
    p.tok_row0 = tok_row0;
    p.status = status;
    p.rows_out = (__nv_bfloat16*)out;
    p.rows_bstride = out_bstride;
    p.rows_ld = out_ld;
    p.rows_scale = scale;
    cudaError_t e = set_smem_attr((const void*)msp_deembed_kernel, kDeSmem);
    if (e != cudaSuccess) return e;
    const dim3 grid((unsigned)p.m_tiles, (unsigned)splits, (unsigned)batch);
    return launch_pdl_cluster(msp_deembed_kernel, grid, dim3(kThreads), kDeSmem, st, dim3(1, splits, 1), maps, p);
}

}  // namespace msf
