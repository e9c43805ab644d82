// MSSA attention on the sm_103a tensor cores (Eq. 4 context, bf16 operands,
// fp32 online softmax and accumulation).
//
// Work: an item is one 256-row query block (two 128-row tiles Q0, Q1) of one
// (stream, head, query group); it walks that group's context segments (sink,
// history or pyramid part, window suffix) in 128-row K/V tiles. All items'
// tiles form one sequence (longest contexts first). While the longest group
// has at least one item per CTA, a persistent grid takes its items whole in
// data-parallel rounds; the rest of the sequence is split into equal
// contiguous ranges, one per CTA (stream-K), which each CTA runs before its
// whole items. A piece is the part of one item inside one CTA's range. A
// piece that is a whole item writes its normalised output; a piece of a
// split item writes its unnormalised output with the running max and sum to
// a partial slot, and the piece that counts itself finished last (per-item
// counter word in the workspace: pieces finished | partials written, reset
// by the merge) has all of them merged in piece order.
//
// Roles inside a CTA (384 threads):
//   warp 0      TMA producer: Q0/Q1 per piece, then K_j and V_j into a
//               2-deep K ring and a 3-deep V ring, gated by one release per tile
//   warp 1      MMA issuer (one elected lane of the converged warp):
//               S_t = Q_t K_j^T into TMEM (SS form), O_t += P_t V_j with P_t
//               read from TMEM (TS form, V MN-major)
//   warp 2      TMEM allocation (all 512 columns)
//   warps 2-3   merge helpers: combine the pieces of the split items this CTA
//               finished last while the softmax warps run the whole items
//   warps 4-7   softmax of tile 0, warps 8-11 softmax of tile 1: one thread
//               per query row; tcgen05.ld of S, exp2 against a running max
//               that may lag, row sum, P as bf16 written over S's first 64
//               columns, rescale of O only when a tile's sum passes 2^32
// TMEM columns: S0 [0,128) S1 [128,256) O0 [256,384) O1 [384,512).
// The MMA thread issues S_t(j+1) right after PV_t(j), so the commit that
// signals S_t(j+1) also covers PV_t(j): a softmax warp that sees S ready may
// rescale O_t in place. Every segment has its own tensor map whose extent is
// the segment's end, so rows past it load as zeros; their scores are masked.
// Every wait is bounded; a wait that gives up raises the CTA's abort flag and
// the device status word, and every role winds down without hanging.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdlib.h>
#include <string.h>

#include "attn_tc.h"
#include "pool.cuh"
#include "ptx.cuh"

namespace msf {

namespace {

constexpr int kBlockM = 128;   // query rows per tile
constexpr int kBlockN = 128;   // context rows per K/V tile
constexpr int kStages = 2;     // K ring depth
constexpr int kVStages = 3;    // V ring depth
constexpr int kThreads = 384;  // 12 warps
// Registers: 168 per thread at launch (12 warps x 168 = 64512 of 65536). The
// producer/MMA warpgroup drops to 120 and the two softmax warpgroups rise to
// 192: 4 x 120 + 8 x 192 = 12 x 168, so the increase is always satisfiable.
// The launcher refuses to run if the compiled kernel does not use exactly
// kLaunchRegs per thread.
constexpr int kLaunchRegs = 168;
constexpr int kCtrlRegs = 120;
constexpr int kSoftmaxRegs = 192;
static_assert(4 * kCtrlRegs + 8 * kSoftmaxRegs == 12 * kLaunchRegs, "register split");
constexpr long long kWaitLimit = 2000000000LL;  // ~1 s of SM clock
// Lead tiles per item in the stream-K sequence: the fixed cost of a piece
// (Q load and pipeline fill, epilogue or partial write) measured as ~5 K/V
// tiles, so CTAs whose ranges hold many short items get fewer tiles.
constexpr int kItemLeadTiles = 5;
// Pieces of one item that the merging CTA combines from one batch of loads.
constexpr int kMergeBatch = 8;
// Bound of the helper warps' wait for a merge job: the next job (or the stop)
// comes after at most the CTA's remaining tiles, so the bound is the CTA's
// tile count times ~0.5 ms of SM clock per tile (about 400 times what a
// 128-row K/V step costs), and at least the per-wait bound.
constexpr long long kHelperCyclesPerTile = 1LL << 20;

struct TcSeg {
    int map;
    int row0;
    int len;
    int tile0;  // first tile of this segment in the item's tile sequence
};
struct TcGroup {
    int q_begin, q_end;
    int n_qb;        // 256-row query blocks
    int n_items;     // B * H * n_qb
    int n_seg;
    int n_tiles;     // tiles per item
    int n_virt;      // item stride in the tile sequence: n_tiles + lead tiles
    long long tile_base;  // first tile of this group in the global sequence
    int item_base;        // first item index of this group (merge counters)
    TcSeg seg[kMaxSeg];
};
struct TcParams {
    int H, B;
    float scale_log2;
    int n_groups;
    long long total_tiles;
    TcGroup g[MSF_MAX_GROUPS];  // longest context first
    __nv_bfloat16* out;
    long long out_bstride;  // elements
    int out_v8;             // output rows 32-byte aligned: 32-byte stores
    unsigned int* status;
    unsigned int* counters;  // per item
    float* partials;         // 2 slots per CTA
    long long wait_limit;
    int dp_rounds;           // whole items of group 0 per CTA before the stream-K range
    long long dp_stride;     // group 0's tiles per item in the sequence (n_virt)
    long long t_sk;          // first sequence position of the stream-K part
    float* lse;              // optional [B, H, N] row log-sum-exp (natural log)
    int N;                   // query rows per stream
    // The launch's own K/V pyramid (0 tasks: none): vector-pair tasks of the
    // pool batch, pool_per_stream = jobs * pool_tasks per stream. pyr_sync[0]
    // counts the CTAs whose share is written, pyr_sync[1] the CTAs that have
    // finished; the last CTA to finish zeroes both.
    long long pool_total;
    int pool_per_stream;
    int pool_tasks;
    int pool_ring;  // the batch also writes the history ring (the staged head)
    unsigned int* pyr_sync;
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
    static constexpr int kSmem = (2 + kStages + kVStages) * kTileBytes + 1024;
    // Partial slot: output as [D/4 float4][256 rows] then [2][256 rows] (running
    // max, running sum), so that the 32 rows of a warp touch consecutive words.
    static constexpr int kSlotFloats = 2 * kBlockM * (D + 2);
    static constexpr int kSlotML = 2 * kBlockM * D;
};

__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

__device__ __forceinline__ unsigned int ld_acquire(const unsigned int* p) {
    unsigned int v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

// One piece of work: tiles [u0, u1) of one item.
struct Piece {
    int gi, item, b, h, q_row0, u0, u1;
    bool whole;
    long long item_start;  // global index of the item's first real tile
    long long t_next;      // sequence position after this piece
};

// A merge handed from the softmax warps to the helper warps.
struct MergeJob {
    long long item_rel;  // sequence position of the item's first real tile, relative to t_sk
    long long c1, c2;    // CTAs holding its pieces
    unsigned int* cnt;   // the item's counter word
    int q_row0, q_end, b, h;
    int stop;            // no more jobs
};

__device__ __forceinline__ long long cta_begin(long long c, long long T, long long n) {
    return c * T / n;
}
// The CTA whose range [cta_begin(c), cta_begin(c+1)) holds tile t.
__device__ __forceinline__ long long cta_of(long long t, long long T, long long n) {
    return ((t + 1) * n - 1) / T;
}

__device__ __forceinline__ Piece locate(const TcParams& p, long long t, long long r1) {
    Piece pc;
    int gi = 0;
    while (gi < p.n_groups - 1 && t >= p.g[gi + 1].tile_base) ++gi;
    const TcGroup& G = p.g[gi];
    const long long rel = t - G.tile_base;
    const int item = (int)(rel / G.n_virt);
    const int v0 = (int)(rel - (long long)item * G.n_virt);
    long long v1 = v0 + (r1 - t);
    if (v1 > G.n_virt) v1 = G.n_virt;
    // Each item starts with lead tiles that stand for the fixed cost of a
    // piece (Q load, pipeline fill, epilogue); they carry no work.
    const int lead = G.n_virt - G.n_tiles;
    pc.gi = gi;
    pc.item = item;
    const int qb = item % G.n_qb;
    pc.h = (item / G.n_qb) % p.H;
    pc.b = item / (G.n_qb * p.H);
    pc.q_row0 = G.q_begin + qb * 2 * kBlockM;
    pc.u0 = v0 > lead ? v0 - lead : 0;
    pc.u1 = (int)v1 > lead ? (int)v1 - lead : 0;
    pc.whole = (pc.u0 == 0 && pc.u1 == G.n_tiles);
    pc.item_start = G.tile_base + (long long)item * G.n_virt + lead;
    pc.t_next = t + (v1 - v0);
    return pc;
}

// Segment, context row and valid row count of tile u of an item of group G.
__device__ __forceinline__ void tile_info(const TcGroup& G, int u, int& seg, int& row, int& valid) {
    int s = 0;
    while (s < G.n_seg - 1 && u >= G.seg[s + 1].tile0) ++s;
    const int kt = u - G.seg[s].tile0;
    seg = s;
    row = G.seg[s].row0 + kt * kBlockN;
    valid = min(kBlockN, G.seg[s].len - kt * kBlockN);
}

// Partial slot of the piece of an item that CTA c holds: a CTA's first piece
// uses slot 2c, a later (last) piece slot 2c+1.
__device__ __forceinline__ int slot_of(long long c, long long c1, long long item_start, long long T,
                                       long long n) {
    return 2 * (int)c + ((c == c1 && cta_begin(c, T, n) < item_start) ? 1 : 0);
}

// The kernel body; kPool: the launch also builds its K/V pyramid (`pool`),
// compiled as its own kernel so that the plain attention carries none of it.
template <int D, bool kPool>
__device__ __forceinline__ void mssa_tc_body(const TcMaps& maps, const TcParams& p, const PoolBatch* pool) {
    using C = Cfg<D>;
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    unsigned char* smem = (unsigned char*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    unsigned char* sQ = smem;                                  // [2][tile]
    unsigned char* sK = smem + 2 * C::kTileBytes;              // [kStages][tile]
    unsigned char* sV = sK + kStages * C::kTileBytes;          // [kVStages][tile]

    __shared__ uint64_t q_full, q_empty, o_full, drain_bar;
    __shared__ uint64_t k_full[kStages], k_empty[kStages], v_full[kVStages];
    __shared__ uint64_t s_full[2], p_full[2];
    __shared__ uint64_t epi_written, epi_decided;
    __shared__ uint64_t job_full, job_empty, job_ready;
    __shared__ MergeJob job;
    __shared__ uint32_t tmem_base_sh;
    __shared__ int abort_flag;
    __shared__ int merge_flag;

    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const long long T = p.total_tiles;
    const long long ncta = gridDim.x;
    // Work of this CTA: its equal share of the stream-K part of the sequence
    // (which starts at t_sk) first, then dp_rounds whole items of the first
    // group (items blockIdx.x, blockIdx.x + ncta, ...). Split items thus end
    // early, and their merges run on the helper warps beside the whole items.
    const long long Tsk = T - p.t_sk;
    const long long r0 = p.t_sk + cta_begin(blockIdx.x, Tsk, ncta);
    const long long r1 = p.t_sk + cta_begin(blockIdx.x + 1, Tsk, ncta);
    auto phase_range = [&](int ph, long long& a0, long long& a1) {
        if (ph == 0) {
            a0 = r0;
            a1 = r1;
        } else {
            a0 = ((long long)blockIdx.x + (long long)(ph - 1) * ncta) * p.dp_stride;
            a1 = a0 + p.dp_stride;
        }
    };
    // Merges of split items go to the helper warps while whole items follow.
    const bool helper_merges = p.dp_rounds > 0;


    if (threadIdx.x == 0) {
        abort_flag = 0;
        merge_flag = 0;
        ptx::mbar_init(&q_full, 1);
        ptx::mbar_init(&q_empty, 1);
        ptx::mbar_init(&o_full, 1);
        ptx::mbar_init(&drain_bar, 1);
        for (int s = 0; s < kStages; ++s) {
            ptx::mbar_init(&k_full[s], 1);
            ptx::mbar_init(&k_empty[s], 1);
        }
        for (int s = 0; s < kVStages; ++s) ptx::mbar_init(&v_full[s], 1);
        for (int t = 0; t < 2; ++t) {
            ptx::mbar_init(&s_full[t], 1);
            ptx::mbar_init(&p_full[t], 4);   // one arrival per softmax warp
        }
        ptx::mbar_init(&epi_written, 8);
        ptx::mbar_init(&epi_decided, 1);
        ptx::mbar_init(&job_full, 1);
        ptx::mbar_init(&job_empty, 2);  // one arrival per helper warp
        ptx::mbar_init(&job_ready, 1);  // the pieces of the job are all written
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
    ptx::grid_dep_wait();  // q/k/v and the pyramid of the previous kernels are visible
    ptx::grid_dep_launch();

    if (warp < 4) {
        ptx::setmaxnreg_dec<kCtrlRegs>();
        if (warp == 0) {
        // =========================== TMA producer ===========================
        if (lane == 0) {
            ptx::prefetch_tmap(&maps.q);
            bool ok = true;
            long long js = 0;  // global K/V step
            int piece = 0;
            bool q_in_flight = false;
            bool pyr_ready = !kPool || p.pool_total == 0;
            // K(j) and V(j) wait for one release: the commit that follows S1 of
            // tile j-2. It covers the last reader of K(j)'s slot (S of tile
            // j-2) and of V(j)'s slot in the 3-deep V ring (PV1 of tile j-3).
            for (int ph = 0; ph <= p.dp_rounds && ok; ++ph) {
            long long a0, a1;
            phase_range(ph, a0, a1);
            for (long long t = a0; t < a1 && ok;) {
                const Piece pc = locate(p, t, a1);
                t = pc.t_next;
                if (pc.u0 == pc.u1) continue;  // lead tiles only
                const TcGroup& G = p.g[pc.gi];
                if (!ptx::mbar_wait_bounded(&q_empty, (uint32_t)((piece & 1) ^ 1), abort_p,
                                            p.wait_limit)) {
                    ok = false;
                    break;
                }
                ptx::mbar_arrive_expect_tx(&q_full, 2 * C::kTileBytes);
                for (int qt = 0; qt < 2; ++qt)
                    for (int c = 0; c < C::kChunks; ++c)
                        ptx::tma_load_4d(sQ + qt * C::kTileBytes + c * (kBlockM * 128), &maps.q,
                                         &q_full, c * 64, pc.h, pc.q_row0 + qt * kBlockM, pc.b);
                q_in_flight = true;
                for (int u = pc.u0; u < pc.u1; ++u, ++js) {
                    int seg, row, valid;
                    tile_info(G, u, seg, row, valid);
                    if (kPool && !pyr_ready &&
                        (G.seg[seg].map >= kMapPyr0 || (p.pool_ring && G.seg[seg].map == kMapHist))) {
                        // The first tile of this CTA that the launch's pooling
                        // writes (a pyramid segment, or the history ring that
                        // holds the staged head): every CTA's share is written
                        // (their rows are read here through TMA, the async proxy).
                        const long long w0 = clock64();
                        while (ld_acquire(p.pyr_sync) < (unsigned int)ncta) {
                            if (*abort_p || clock64() - w0 > p.wait_limit) {
                                *abort_p = 1;
                                ok = false;
                                break;
                            }
                        }
                        if (!ok) break;
                        asm volatile("fence.proxy.async.global;" ::: "memory");
                        pyr_ready = true;
                    }
                    const CUtensorMap* mk = &maps.k[G.seg[seg].map];
                    const int st = (int)(js % kStages);
                    const uint32_t ph = (uint32_t)((js / kStages) & 1);
                    if (!ptx::mbar_wait_bounded(&k_empty[st], ph ^ 1u, abort_p, p.wait_limit)) {
                        ok = false;
                        break;
                    }
                    ptx::mbar_arrive_expect_tx(&k_full[st], C::kTileBytes);
                    for (int c = 0; c < C::kChunks; ++c)
                        ptx::tma_load_4d(sK + st * C::kTileBytes + c * (kBlockN * 128), mk,
                                         &k_full[st], c * 64, pc.h, row, pc.b);
                    const int sv = (int)(js % kVStages);
                    ptx::mbar_arrive_expect_tx(&v_full[sv], C::kTileBytes);
                    for (int c = 0; c < C::kChunks; ++c)
                        ptx::tma_load_4d(sV + sv * C::kTileBytes + c * (kBlockN * 128),
                                         &maps.v[G.seg[seg].map], &v_full[sv], c * 64, pc.h, row, pc.b);
                    if (js == 0) {
                        // Cold start: every CTA asks HBM for its first tiles at
                        // once. The ring's deeper tiles wait until Q has landed,
                        // so the first tile's bytes are not queued behind them.
                        if (!ptx::mbar_wait_bounded(&q_full, 0, abort_p, p.wait_limit)) {
                            ok = false;
                            ++js;  // tile 0's copies are in flight: drain them
                            break;
                        }
                    }
                }
                ++piece;
            }
            }
            if (!ok) {
                // Drain: every copy issued must land before the CTA exits.
                if (q_in_flight)
                    ptx::mbar_wait_bounded(&q_full, (uint32_t)((piece - 1) & 1), &never, kWaitLimit);
                for (long long j = (js > kStages ? js - kStages : 0); j < js; ++j)
                    ptx::mbar_wait_bounded(&k_full[j % kStages], (uint32_t)((j / kStages) & 1), &never,
                                           kWaitLimit);
                for (long long j = (js > kVStages ? js - kVStages : 0); j < js; ++j)
                    ptx::mbar_wait_bounded(&v_full[j % kVStages], (uint32_t)((j / kVStages) & 1), &never,
                                           kWaitLimit);
                atomicOr(p.status, kDevTimeout);
            }
        }
        } else if (warp == 1) {
        // ============================ MMA issuer ============================
        // The whole warp runs the loop, so its control flow, barrier waits and
        // descriptors stay warp-uniform; one elected lane (the same lane every
        // time in a converged warp, so every commit covers every MMA before
        // it) issues the MMAs and commits. The tensor pipe queues only a few
        // MMAs, so the loop waits at two points per K/V step and issues 16
        // MMAs after each.
        {
            constexpr uint32_t idS = ptx::idesc_bf16(kBlockM, kBlockN, false, false);
            constexpr uint32_t idO = ptx::idesc_bf16(kBlockM, D, false, true);
            // Descriptors are built once; a K step or another stage only adds a
            // constant to the 14-bit start-address field (shared memory offsets
            // stay below 256 KB, so the field never carries).
            constexpr uint64_t kTileDesc = (uint64_t)(C::kTileBytes >> 4);
            const uint64_t q_desc = ptx::sdesc_sw128(ptx::smem_u32(sQ), 16, 1024);
            const uint64_t k_desc = ptx::sdesc_sw128(ptx::smem_u32(sK), 16, 1024);
            const uint64_t v_desc = ptx::sdesc_sw128(ptx::smem_u32(sV), kBlockN * 128, 1024);
            auto issue_s = [&](int t, int st) {
                const uint64_t qd = q_desc + (uint64_t)t * kTileDesc;
                const uint64_t kd = k_desc + (uint64_t)st * kTileDesc;
                const uint32_t d = tbase + t * 128;
#pragma unroll
                for (int kk = 0; kk < D / 16; ++kk) {
                    constexpr int kChunk = kBlockM * 128;
                    const uint64_t off = (uint64_t)(((kk / 4) * kChunk + (kk % 4) * 32) >> 4);
                    ptx::mma_ss(d, qd + off, kd + off, idS, kk > 0 ? 1u : 0u);
                }
                ptx::mma_commit(&s_full[t]);
            };
            auto issue_pv = [&](int t, int st, bool acc) {
                const uint64_t vd = v_desc + (uint64_t)st * kTileDesc;
                const uint32_t d = tbase + 256 + t * 128, a = tbase + t * 128;
#pragma unroll
                for (int kk = 0; kk < kBlockN / 16; ++kk)
                    ptx::mma_ts(d, a + kk * 8, vd + (uint64_t)(kk * (2048 >> 4)), idO,
                                (acc || kk > 0) ? 1u : 0u);
            };
            // Warp-wide bounded wait: every lane waits, the warp agrees.
            auto wait_all = [&](uint64_t* bar, uint32_t parity) {
                const bool r = ptx::mbar_wait_bounded(bar, parity, abort_p, p.wait_limit);
                return __all_sync(0xffffffffu, r);
            };
            bool ok = true;
            // Ring positions of the next K/V tile: K slot and phase (2-deep),
            // V slot and phase (3-deep), P/S phase (one per tile).
            int ks = 0, vs = 0;
            uint32_t kph = 0, vph = 0, pph = 0;
            int piece = 0;
            for (int ph = 0; ph <= p.dp_rounds && ok; ++ph) {
            long long a0, a1;
            phase_range(ph, a0, a1);
            for (long long t = a0; t < a1 && ok;) {
                const Piece pc = locate(p, t, a1);
                t = pc.t_next;
                const int n = pc.u1 - pc.u0;
                if (n == 0) continue;  // lead tiles only
                ok = wait_all(&q_full, (uint32_t)(piece & 1)) && wait_all(&k_full[ks], kph);
                if (!ok) break;
                ptx::tc_fence_after();
                if (ptx::elect_one_sync()) {
                    issue_s(0, ks);
                    issue_s(1, ks);
                    ptx::mma_commit(&k_empty[ks]);
                    if (n == 1) ptx::mma_commit(&q_empty);
                }
                __syncwarp();
                for (int jl = 0; jl < n; ++jl) {
                    const bool more = jl + 1 < n;
                    const int ks1 = ks ^ 1;
                    const uint32_t kph1 = ks1 == 0 ? kph ^ 1u : kph;
                    // V of this tile, K of the next one and P0 of this tile: the
                    // three probes go out together; the bounded waits run only
                    // if one of them is not ready yet.
                    {
                        const bool rv = ptx::mbar_try_wait(&v_full[vs], vph);
                        const bool rk = !more || ptx::mbar_try_wait(&k_full[ks1], kph1);
                        const bool rp = ptx::mbar_try_wait(&p_full[0], pph);
                        if (!__all_sync(0xffffffffu, rv && rk && rp))
                            ok = wait_all(&v_full[vs], vph) && (!more || wait_all(&k_full[ks1], kph1)) &&
                                 wait_all(&p_full[0], pph);
                    }
                    if (!ok) break;
                    ptx::tc_fence_after();
                    if (ptx::elect_one_sync()) {
                        issue_pv(0, vs, jl > 0);
                        if (more) issue_s(0, ks1);
                    }
                    __syncwarp();
                    ok = wait_all(&p_full[1], pph);
                    if (!ok) break;
                    ptx::tc_fence_after();
                    if (ptx::elect_one_sync()) {
                        issue_pv(1, vs, jl > 0);
                        if (more) {
                            issue_s(1, ks1);
                            ptx::mma_commit(&k_empty[ks1]);
                            if (jl + 2 == n) ptx::mma_commit(&q_empty);  // last use of Q issued
                        }
                    }
                    __syncwarp();
                    ks = ks1;
                    kph = kph1;
                    pph ^= 1u;
                    if (++vs == kVStages) {
                        vs = 0;
                        vph ^= 1u;
                    }
                }
                if (!ok) break;
                if (ptx::elect_one_sync()) ptx::mma_commit(&o_full);
                __syncwarp();
                ++piece;
            }
            }
            if (!ok) {
                // drain_bar covers every MMA issued: TMEM is never released under one.
                if (ptx::elect_one_sync()) ptx::mma_commit(&drain_bar);
                __syncwarp();
                ptx::mbar_wait_bounded(&drain_bar, 0, &never, kWaitLimit);
                if (lane == 0) atomicOr(p.status, kDevTimeout);
            }
        }
        } else if (helper_merges) {
        // ========================== merge helpers ===========================
        // Warps 2 and 3 merge the split items whose last piece this CTA
        // finished, while the softmax warps go on with whole items: every
        // piece's partial result is in its slot, and each of the 64 threads
        // combines four rows, in piece order (the same bits whichever CTA
        // merges). Loads go out in batches (m and l of every piece, then one
        // 16-column chunk of two pieces), as each round trip to L2 costs
        // about a microsecond.
        const int ht = (warp - 2) * 32 + lane;
        long long helper_limit = ((r1 - r0) + (long long)p.dp_rounds * p.dp_stride) * kHelperCyclesPerTile;
        if (helper_limit < p.wait_limit) helper_limit = p.wait_limit;
        for (int jn = 0;; ++jn) {
            // The next job may come only after this CTA's whole items (or its
            // stop at the end), so this wait's bound scales with the CTA's
            // tiles; the softmax warps' own waits are bounded and raise the
            // abort flag, which ends it at once.
            bool okj = ptx::mbar_wait_bounded(&job_full, (uint32_t)(jn & 1), abort_p, helper_limit);
            okj = __all_sync(0xffffffffu, okj);
            if (!okj) break;
            const volatile MergeJob& vj = job;
            if (vj.stop) break;
            const long long c1 = vj.c1, item_rel = vj.item_rel;
            const int n = (int)(vj.c2 - c1) + 1;
            const int q_row0 = vj.q_row0, q_end = vj.q_end, jb = vj.b, jh = vj.h;
            unsigned int* const jcnt = vj.cnt;
            // The other pieces have finished their tiles; wait (bounded) until
            // their partial results are written and fenced, then reset the
            // counter for the next launch.
            if (warp == 2) {
                if (lane == 0) {
                    const long long w0 = clock64();
                    while ((*(volatile unsigned int*)jcnt >> 16) != (unsigned int)(n - 1)) {
                        if (*abort_p || clock64() - w0 > p.wait_limit) {
                            *abort_p = 1;
                            atomicOr(p.status, kDevTimeout);
                            break;
                        }
                    }
                    atomicExch(jcnt, 0u);
                    __threadfence();
                    ptx::mbar_arrive(&job_ready);
                }
                __syncwarp();
            } else {
                okj = ptx::mbar_wait_bounded(&job_ready, (uint32_t)(jn & 1), abort_p, p.wait_limit);
                okj = __all_sync(0xffffffffu, okj);
                if (!okj) break;
            }
            if (*abort_p) break;
            int off[kMergeBatch];
#pragma unroll
            for (int k = 0; k < kMergeBatch; ++k)
                off[k] = k < n ? slot_of(c1 + k, c1, item_rel, Tsk, ncta) * C::kSlotFloats : 0;
#pragma unroll 1
            for (int i = 0; i < 4; ++i) {
                const int rr = i * 64 + ht;
                const int qrow = q_row0 + rr;
                float mv[kMergeBatch], lv[kMergeBatch];
#pragma unroll
                for (int k = 0; k < kMergeBatch; ++k) {
                    mv[k] = k < n ? __ldcg(p.partials + off[k] + C::kSlotML + rr) : -INFINITY;
                    lv[k] = k < n ? __ldcg(p.partials + off[k] + C::kSlotML + 2 * kBlockM + rr) : 0.f;
                }
                float M = -INFINITY;
#pragma unroll
                for (int k = 0; k < kMergeBatch; ++k) M = fmaxf(M, mv[k]);
                float L = 0.f;
#pragma unroll
                for (int k = 0; k < kMergeBatch; ++k) {
                    mv[k] = k < n ? ex2(mv[k] - M) : 0.f;  // piece k's weight
                    L = fmaf(mv[k], lv[k], L);
                }
                const float inv = 1.0f / L;
                const bool store = qrow < q_end;
                if (store && p.lse)
                    p.lse[((size_t)jb * p.H + jh) * p.N + qrow] = (M + log2f(L)) * 0.6931471805599453f;
                __nv_bfloat16* dst = p.out + (size_t)jb * p.out_bstride + ((size_t)qrow * p.H + jh) * D;
#pragma unroll 1
                for (int ch = 0; ch < D / 16; ++ch) {
                    float acc[16];
#pragma unroll
                    for (int e = 0; e < 16; ++e) acc[e] = 0.f;
#pragma unroll
                    for (int k = 0; k < kMergeBatch; k += 2) {
                        if (k >= n) break;
                        const bool two = k + 1 < n;
                        const float4* sa = reinterpret_cast<const float4*>(p.partials + off[k]) + rr;
                        const float4* sb = reinterpret_cast<const float4*>(p.partials + off[k + 1]) + rr;
                        float4 va[4], vb[4];
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            const size_t q = (size_t)(ch * 4 + e) * 2 * kBlockM;
                            va[e] = __ldcg(sa + q);
                            vb[e] = two ? __ldcg(sb + q) : make_float4(0.f, 0.f, 0.f, 0.f);
                        }
                        const float wa = mv[k], wb = mv[k + 1];
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            acc[4 * e] = fmaf(wa, va[e].x, acc[4 * e]);
                            acc[4 * e + 1] = fmaf(wa, va[e].y, acc[4 * e + 1]);
                            acc[4 * e + 2] = fmaf(wa, va[e].z, acc[4 * e + 2]);
                            acc[4 * e + 3] = fmaf(wa, va[e].w, acc[4 * e + 3]);
                            if (two) {
                                acc[4 * e] = fmaf(wb, vb[e].x, acc[4 * e]);
                                acc[4 * e + 1] = fmaf(wb, vb[e].y, acc[4 * e + 1]);
                                acc[4 * e + 2] = fmaf(wb, vb[e].z, acc[4 * e + 2]);
                                acc[4 * e + 3] = fmaf(wb, vb[e].w, acc[4 * e + 3]);
                            }
                        }
                    }
                    if (store) {
                        uint4* d4 = reinterpret_cast<uint4*>(dst + ch * 16);
#pragma unroll
                        for (int e = 0; e < 2; ++e)
                            d4[e] = make_uint4(ptx::pack_bf16(acc[8 * e] * inv, acc[8 * e + 1] * inv),
                                               ptx::pack_bf16(acc[8 * e + 2] * inv, acc[8 * e + 3] * inv),
                                               ptx::pack_bf16(acc[8 * e + 4] * inv, acc[8 * e + 5] * inv),
                                               ptx::pack_bf16(acc[8 * e + 6] * inv, acc[8 * e + 7] * inv));
                    }
                }
            }
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&job_empty);
        }
        }
    } else {
        ptx::setmaxnreg_inc<kSoftmaxRegs>();
        if (kPool && p.pool_total > 0) {
            // =================== the launch's K/V pyramid ===================
            // Eq. 4's Subsample of the window states (and the history, and the
            // staged head) before the first softmax: the 256 softmax threads of
            // every CTA take a strided share of the vector-pair tasks while the
            // producer and the MMA issuer start on the first tiles. Only tiles
            // of a pyramid segment wait for the count.
            const int ti = (int)threadIdx.x - 128;
            for (long long tk = (long long)blockIdx.x * 256 + ti; tk < p.pool_total;
                 tk += (long long)gridDim.x * 256) {
                const int b = (int)(tk / p.pool_per_stream);
                const int rr = (int)(tk - (long long)b * p.pool_per_stream);
                pool_task<__nv_bfloat16>(*pool, rr / p.pool_tasks, b, rr % p.pool_tasks);
            }
            // generic-proxy writes, read by other CTAs' TMA loads: proxy fence
            // and GPU-scope fence by every writer, then one count per CTA
            asm volatile("fence.proxy.async.global;" ::: "memory");
            __threadfence();
            ptx::named_bar_sync(1, 256);
            if (threadIdx.x == 128) atomicAdd(p.pyr_sync, 1u);
        }
        // ============================== softmax =============================
        const int t = (warp - 4) / 4;
        const int wq = warp % 4;
        const int r = wq * 32 + lane;
        const uint32_t lane_off = (uint32_t)(wq * 32) << 16;
        const uint32_t tS = tbase + t * 128 + lane_off;
        const uint32_t tO = tbase + 256 + t * 128 + lane_off;
        const float sl2 = p.scale_log2;
        bool ok = true;
        long long js = 0;
        int piece = 0, nsplit = 0, nwritten = 0, njob = 0;
        for (int ph = 0; ph <= p.dp_rounds && ok; ++ph) {
        long long a0, a1;
        phase_range(ph, a0, a1);
        for (long long tt = a0; tt < a1 && ok;) {
            const Piece pc = locate(p, tt, a1);
            tt = pc.t_next;
            if (pc.u0 == pc.u1) continue;  // lead tiles only
            const TcGroup& G = p.g[pc.gi];
            float m_used = -INFINITY, l = 0.f;
            // A split piece counts itself finished as its last tile starts (one
            // thread, its result used only in the epilogue, so the atomic's
            // round trip overlaps that tile): the last to count in merges.
            unsigned int fin_old = 0;
            unsigned int* const cnt = p.counters + G.item_base + pc.item;
            for (int u = pc.u0; u < pc.u1; ++u, ++js) {
                int seg, row, valid;
                tile_info(G, u, seg, row, valid);
                if (!pc.whole && u == pc.u1 - 1 && warp == 4 && lane == 0) fin_old = atomicAdd(cnt, 1u);
                ok = ptx::mbar_wait_bounded(&s_full[t], (uint32_t)(js & 1), abort_p, p.wait_limit);
                ok = __all_sync(0xffffffffu, ok);
                if (!ok) break;
                ptx::tc_fence_after();
                uint32_t s[4][32];
#pragma unroll
                for (int q4 = 0; q4 < 4; ++q4) ptx::tmem_ld32(tS + 32 * q4, s[q4]);
                ptx::tmem_wait_ld();
                if (valid < kBlockN) {
                    // Rows past the segment's end: score -inf, probability 0.
#pragma unroll
                    for (int c = 0; c < 128; ++c)
                        if (c >= valid) s[c >> 5][c & 31] = 0xff800000u;
                }
                // Exponentials use the running maximum m_used, which may lag
                // the row's true maximum: P = 2^(s - m_used) then exceeds 1,
                // which changes nothing but a power-of-two scale common to
                // P, O and l. The tile's sum shows how far it lags; only when
                // it passes 2^32 (or is not finite) is the exact maximum found
                // and O rescaled, so most tiles skip the max pass entirely.
                // The first tile of a piece starts from its exact maximum.
                auto tile_max = [&]() -> float {
                    float mx[8];
#pragma unroll
                    for (int e = 0; e < 8; ++e) mx[e] = -INFINITY;
#pragma unroll
                    for (int c = 0; c < 128; c += 2)
                        mx[(c >> 1) & 7] = ptx::fmax3(mx[(c >> 1) & 7], __uint_as_float(s[c >> 5][c & 31]),
                                                      __uint_as_float(s[c >> 5][(c & 31) + 1]));
                    return fmaxf(ptx::fmax3(mx[0], mx[1], mx[2]),
                                 fmaxf(ptx::fmax3(mx[3], mx[4], mx[5]), fmaxf(mx[6], mx[7]))) * sl2;
                };
                if (u == pc.u0) m_used = tile_max();
                uint64_t sum2[2];
#pragma unroll 1
                for (int pass = 0; pass < 2; ++pass) {
                    const float nm = -m_used;
                    const uint64_t sl2x2 = ptx::f2_pack(sl2, sl2), nmx2 = ptx::f2_pack(nm, nm);
                    sum2[0] = sum2[1] = ptx::f2_pack(0.f, 0.f);
#pragma unroll
                    for (int q4 = 0; q4 < 4; ++q4) {
                        uint32_t pk[16];
#pragma unroll
                        for (int c = 0; c < 16; ++c) {
                            const uint64_t arg = ptx::f2_fma(
                                ptx::f2_pack(__uint_as_float(s[q4][2 * c]), __uint_as_float(s[q4][2 * c + 1])),
                                sl2x2, nmx2);
                            float a0, a1;
                            ptx::f2_unpack(arg, a0, a1);
                            const float p0 = ex2(a0), p1 = ex2(a1);
                            sum2[c & 1] = ptx::f2_add(sum2[c & 1], ptx::f2_pack(p0, p1));
                            pk[c] = ptx::pack_bf16(p0, p1);
                        }
                        ptx::tmem_st16(tS + 16 * q4, pk);
                    }
                    if (pass == 1) break;
                    float a0, a1, b0, b1;
                    ptx::f2_unpack(sum2[0], a0, a1);
                    ptx::f2_unpack(sum2[1], b0, b1);
                    const float tile_sum = (a0 + a1) + (b0 + b1);
                    if (!__any_sync(0xffffffffu, !(tile_sum <= 4294967296.0f))) break;
                    // O_t holds every PV up to the previous step (the S_t commit covers it).
                    const float m_new = fmaxf(m_used, tile_max());
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
                    ptx::tmem_wait_st();  // P of the first pass is overwritten after this
                }
                {
                    float a0, a1, b0, b1;
                    ptx::f2_unpack(sum2[0], a0, a1);
                    ptx::f2_unpack(sum2[1], b0, b1);
                    l += (a0 + a1) + (b0 + b1);
                }
                ptx::tmem_wait_st();
                ptx::tc_fence_before();
                __syncwarp();
                if (lane == 0) ptx::mbar_arrive(&p_full[t]);
            }
            if (!ok) break;
            ok = ptx::mbar_wait_bounded(&o_full, (uint32_t)(piece & 1), abort_p, p.wait_limit);
            ok = __all_sync(0xffffffffu, ok);
            if (!ok) break;
            ptx::tc_fence_after();
            const int qrow = pc.q_row0 + t * kBlockM + r;
            const bool store = qrow < G.q_end;
            __nv_bfloat16* dst =
                p.out + (size_t)pc.b * p.out_bstride + ((size_t)qrow * p.H + pc.h) * D;
            if (pc.whole) {
                const float inv = 1.0f / l;
                // P, O and l share the scale 2^-m_used: ln sum exp = (m_used + log2 l) ln 2
                if (store && p.lse)
                    p.lse[((size_t)pc.b * p.H + pc.h) * p.N + qrow] =
                        (m_used + log2f(l)) * 0.6931471805599453f;
                // The whole row of O in one batch of TMEM loads and one wait (the
                // registers of S are free here), then packed and stored.
                uint32_t ob[D / 32][32];
#pragma unroll
                for (int c = 0; c < D / 32; ++c) ptx::tmem_ld32(tO + c * 32, ob[c]);
                ptx::tmem_wait_ld();
#pragma unroll
                for (int c = 0; c < D / 32; ++c) {
                    const uint32_t* o = ob[c];
                    uint32_t pk[16];
#pragma unroll
                    for (int e = 0; e < 16; ++e)
                        pk[e] = ptx::pack_bf16(__uint_as_float(o[2 * e]) * inv,
                                               __uint_as_float(o[2 * e + 1]) * inv);
                    if (store && p.out_v8) {
                        ptx::st_global_v8(dst + c * 32, pk);
                        ptx::st_global_v8(dst + c * 32 + 16, pk + 8);
                    } else if (store) {
                        uint4* d4 = reinterpret_cast<uint4*>(dst + c * 32);
#pragma unroll
                        for (int e = 0; e < 4; ++e)
                            d4[e] = make_uint4(pk[4 * e], pk[4 * e + 1], pk[4 * e + 2], pk[4 * e + 3]);
                    }
                }
            } else {
                // ---- split item (only stream-K pieces are split: positions
                // relative to t_sk). The piece that counted itself finished
                // last merges; every other piece writes its partial result.
                const long long c1 = cta_of(pc.item_start - p.t_sk, Tsk, ncta);
                const long long c2 = cta_of(pc.item_start + G.n_tiles - 1 - p.t_sk, Tsk, ncta);
                const int slot = slot_of(blockIdx.x, c1, pc.item_start - p.t_sk, Tsk, ncta);
                const int rr = t * kBlockM + r;
                const int n_pieces = (int)(c2 - c1) + 1;
                // The counter word holds the pieces finished (low 16 bits) and
                // the partial results written (high 16 bits).
                const uint32_t par = (uint32_t)(nsplit & 1);
                ++nsplit;
                if (warp == 4 && lane == 0) {
                    int last = (fin_old & 0xffffu) == (unsigned int)(n_pieces - 1);
                    // A merge handed to the helper warps waits there instead.
                    if (last && !(helper_merges && n_pieces <= kMergeBatch)) {
                        // Every other piece has finished its tiles; wait (bounded)
                        // until their partial results are written and fenced.
                        const long long w0 = clock64();
                        while ((*(volatile unsigned int*)cnt >> 16) != (unsigned int)(n_pieces - 1)) {
                            if (*abort_p || clock64() - w0 > p.wait_limit) {
                                *abort_p = 1;
                                atomicOr(p.status, kDevTimeout);
                                break;
                            }
                        }
                        atomicExch(cnt, 0u);  // no piece updates it again in this launch
                        __threadfence();
                    }
                    merge_flag = last;
                    ptx::mbar_arrive(&epi_decided);
                }
                ok = ptx::mbar_wait_bounded(&epi_decided, par, abort_p, p.wait_limit);
                ok = __all_sync(0xffffffffu, ok && !*abort_p);
                if (!ok) break;
                const bool merger = *(volatile int*)&merge_flag != 0;
                // The merge goes to the helper warps when whole items follow;
                // otherwise the merger of an item of up to kMergeBatch pieces
                // keeps its own piece in TMEM and merges here. Every other
                // piece writes its partial result.
                const bool to_helper = merger && helper_merges && n_pieces <= kMergeBatch;
                const bool fast = merger && !helper_merges && n_pieces <= kMergeBatch;
                if (!fast) {
                    float* ps = p.partials + (size_t)slot * C::kSlotFloats;
                    float4* po = reinterpret_cast<float4*>(ps) + rr;
                    uint32_t ob[D / 32][32];
#pragma unroll
                    for (int c = 0; c < D / 32; ++c) ptx::tmem_ld32(tO + c * 32, ob[c]);
                    ptx::tmem_wait_ld();
#pragma unroll
                    for (int c = 0; c < D / 32; ++c) {
                        const uint32_t* o = ob[c];
#pragma unroll
                        for (int e = 0; e < 8; ++e)
                            po[(size_t)(c * 8 + e) * 2 * kBlockM] =
                                make_float4(__uint_as_float(o[4 * e]), __uint_as_float(o[4 * e + 1]),
                                            __uint_as_float(o[4 * e + 2]), __uint_as_float(o[4 * e + 3]));
                    }
                    ps[C::kSlotML + rr] = m_used;
                    ps[C::kSlotML + 2 * kBlockM + rr] = l;
                    __syncwarp();
                    if (lane == 0) ptx::mbar_arrive(&epi_written);  // release, CTA scope
                    const uint32_t pw = (uint32_t)(nwritten & 1);
                    ++nwritten;
                    if (warp == 4 && lane == 0 && (!merger || to_helper)) {
                        // All 256 rows are written (acquired through the barrier);
                        // one GPU-scope fence, which is cumulative over the writes
                        // of the eight warps, orders them before the count or the
                        // hand-over to the helper warps.
                        bool okw = ptx::mbar_wait_bounded(&epi_written, pw, abort_p, p.wait_limit);
                        if (okw) __threadfence();
                        if (okw && !merger) atomicAdd(cnt, 1u << 16);
                        if (okw && to_helper) {
                            okw = ptx::mbar_wait_bounded(&job_empty, (uint32_t)((njob & 1) ^ 1), abort_p,
                                                         p.wait_limit);
                            if (okw) {
                                job.item_rel = pc.item_start - p.t_sk;
                                job.c1 = c1;
                                job.c2 = c2;
                                job.cnt = cnt;
                                job.q_row0 = pc.q_row0;
                                job.q_end = G.q_end;
                                job.b = pc.b;
                                job.h = pc.h;
                                job.stop = 0;
                                ptx::mbar_arrive(&job_full);
                            }
                        }
                        if (!okw) atomicOr(p.status, kDevTimeout);
                    }
                    if (to_helper) ++njob;
                }
                if (fast) {
                    // ---- last piece: merge every piece of this item, in piece
                    // order whichever CTA merges (the same bits on every run).
                    // Its own piece is still in TMEM (O) and registers
                    // (m_used, l); the others come from L2, and each batch of
                    // loads (m and l of every piece, then one 32-column chunk
                    // of two other pieces) is issued before its first use: a
                    // round trip to L2 costs about a microsecond, so the merge
                    // takes a few round trips instead of one per piece and
                    // chunk. Other piece k is piece k + (k >= own) in order.
                    const int own = (int)((long long)blockIdx.x - c1);
                    const int n_oth = n_pieces - 1;
                    int off[kMergeBatch];  // even length: the pairs below never index past it
                    float mv[kMergeBatch], lv[kMergeBatch];
#pragma unroll
                    for (int k = 0; k < kMergeBatch; ++k) {
                        off[k] = 0;
                        mv[k] = -INFINITY;
                        lv[k] = 0.f;
                        if (k < n_oth) {
                            off[k] = slot_of(c1 + k + (k >= own ? 1 : 0), c1, pc.item_start - p.t_sk, Tsk,
                                             ncta) * C::kSlotFloats;
                            mv[k] = __ldcg(p.partials + off[k] + C::kSlotML + rr);
                            lv[k] = __ldcg(p.partials + off[k] + C::kSlotML + 2 * kBlockM + rr);
                        }
                    }
                    float M = m_used;
#pragma unroll
                    for (int k = 0; k < kMergeBatch; ++k) M = fmaxf(M, mv[k]);
                    const float w_own = ex2(m_used - M);
                    float L = 0.f;
#pragma unroll
                    for (int k = 0; k < kMergeBatch; ++k) {
                        if (k == own) L = fmaf(w_own, l, L);
                        mv[k] = k < n_oth ? ex2(mv[k] - M) : 0.f;  // other piece k's weight
                        if (k < n_oth) L = fmaf(mv[k], lv[k], L);
                    }
                    const float inv = 1.0f / L;
                    if (store && p.lse)
                        p.lse[((size_t)pc.b * p.H + pc.h) * p.N + qrow] =
                            (M + log2f(L)) * 0.6931471805599453f;
#pragma unroll 1
                    for (int ch = 0; ch < D / 32; ++ch) {
                        uint32_t o[32];
                        ptx::tmem_ld32(tO + ch * 32, o);
                        ptx::tmem_wait_ld();
                        float acc[32];
#pragma unroll
                        for (int e = 0; e < 32; ++e) acc[e] = 0.f;
#pragma unroll
                        for (int k = 0; k < kMergeBatch; k += 2) {
                            if (k >= n_oth) break;
                            const bool two = k + 1 < n_oth;
                            const float4* sa = reinterpret_cast<const float4*>(p.partials + off[k]) + rr;
                            const float4* sb = reinterpret_cast<const float4*>(p.partials + off[k + 1]) + rr;
                            float4 va[8], vb[8];
#pragma unroll
                            for (int e = 0; e < 8; ++e) {
                                const size_t q = (size_t)(ch * 8 + e) * 2 * kBlockM;
                                va[e] = __ldcg(sa + q);
                                vb[e] = two ? __ldcg(sb + q) : make_float4(0.f, 0.f, 0.f, 0.f);
                            }
                            const float wa = mv[k], wb = mv[k + 1];
#pragma unroll
                            for (int e = 0; e < 8; ++e) {
                                const float a4[4] = {va[e].x, va[e].y, va[e].z, va[e].w};
                                const float b4[4] = {vb[e].x, vb[e].y, vb[e].z, vb[e].w};
#pragma unroll
                                for (int x = 0; x < 4; ++x) {
                                    float v = acc[4 * e + x];
                                    const float ov = __uint_as_float(o[4 * e + x]);
                                    if (own == k) v = fmaf(w_own, ov, v);
                                    v = fmaf(wa, a4[x], v);
                                    if (two && own == k + 1) v = fmaf(w_own, ov, v);
                                    if (two) v = fmaf(wb, b4[x], v);
                                    acc[4 * e + x] = v;
                                }
                            }
                        }
                        if (own == n_oth) {  // the own piece is the item's last one
#pragma unroll
                            for (int e = 0; e < 32; ++e) acc[e] = fmaf(w_own, __uint_as_float(o[e]), acc[e]);
                        }
                        if (store) {
                            uint4* d4 = reinterpret_cast<uint4*>(dst + ch * 32);
#pragma unroll
                            for (int e = 0; e < 4; ++e)
                                d4[e] = make_uint4(ptx::pack_bf16(acc[8 * e] * inv, acc[8 * e + 1] * inv),
                                                   ptx::pack_bf16(acc[8 * e + 2] * inv, acc[8 * e + 3] * inv),
                                                   ptx::pack_bf16(acc[8 * e + 4] * inv, acc[8 * e + 5] * inv),
                                                   ptx::pack_bf16(acc[8 * e + 6] * inv, acc[8 * e + 7] * inv));
                        }
                    }
                } else if (merger && !to_helper) {
                    // ---- last piece of an item cut into more pieces than one
                    // batch holds: merge every piece from its partial slot
                    const int rr = t * kBlockM + r;
                    float M = -INFINITY;
                    for (long long c = c1; c <= c2; ++c) {
                        const float* q = p.partials +
                                         (size_t)slot_of(c, c1, pc.item_start - p.t_sk, Tsk, ncta) * C::kSlotFloats;
                        M = fmaxf(M, __ldcg(q + C::kSlotML + rr));
                    }
                    float L = 0.f;
                    for (long long c = c1; c <= c2; ++c) {
                        const float* q = p.partials +
                                         (size_t)slot_of(c, c1, pc.item_start - p.t_sk, Tsk, ncta) * C::kSlotFloats;
                        L += ex2(__ldcg(q + C::kSlotML + rr) - M) * __ldcg(q + C::kSlotML + 2 * kBlockM + rr);
                    }
                    const float inv = 1.0f / L;
                    if (store && p.lse)
                        p.lse[((size_t)pc.b * p.H + pc.h) * p.N + qrow] =
                            (M + log2f(L)) * 0.6931471805599453f;
#pragma unroll 1
                    for (int ch = 0; ch < D / 32; ++ch) {
                        float acc[32];
#pragma unroll
                        for (int e = 0; e < 32; ++e) acc[e] = 0.f;
                        for (long long c = c1; c <= c2; ++c) {
                            const float* base =
                                p.partials + (size_t)slot_of(c, c1, pc.item_start - p.t_sk, Tsk, ncta) * C::kSlotFloats;
                            const float w = ex2(__ldcg(base + C::kSlotML + rr) - M);
                            const float4* src = reinterpret_cast<const float4*>(base) + rr;
#pragma unroll
                            for (int e = 0; e < 8; ++e) {
                                const float4 v = __ldcg(src + (size_t)(ch * 8 + e) * 2 * kBlockM);
                                acc[4 * e] = fmaf(w, v.x, acc[4 * e]);
                                acc[4 * e + 1] = fmaf(w, v.y, acc[4 * e + 1]);
                                acc[4 * e + 2] = fmaf(w, v.z, acc[4 * e + 2]);
                                acc[4 * e + 3] = fmaf(w, v.w, acc[4 * e + 3]);
                            }
                        }
                        if (store) {
                            uint4* d4 = reinterpret_cast<uint4*>(dst + ch * 32);
#pragma unroll
                            for (int e = 0; e < 4; ++e)
                                d4[e] = make_uint4(ptx::pack_bf16(acc[8 * e] * inv, acc[8 * e + 1] * inv),
                                                   ptx::pack_bf16(acc[8 * e + 2] * inv, acc[8 * e + 3] * inv),
                                                   ptx::pack_bf16(acc[8 * e + 4] * inv, acc[8 * e + 5] * inv),
                                                   ptx::pack_bf16(acc[8 * e + 6] * inv, acc[8 * e + 7] * inv));
                        }
                    }
                }
            }
            ++piece;
        }
        }
        if (!ok && lane == 0) atomicOr(p.status, kDevTimeout);
        if (helper_merges && warp == 4 && lane == 0) {
            // No more merges: let the helper warps finish.
            if (ptx::mbar_wait_bounded(&job_empty, (uint32_t)((njob & 1) ^ 1), abort_p, p.wait_limit)) {
                job.stop = 1;
                ptx::mbar_arrive(&job_full);
            }
        }
    }

    ptx::tc_fence_before();
    __syncthreads();
    if (warp == 2) {
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tbase, 512);
    }
    if (kPool && p.pool_total > 0 && threadIdx.x == 0) {
        // The last CTA to finish resets the pyramid counts for the next
        // launch: no CTA of this one waits on them any more.
        __threadfence();
        if (atomicAdd(p.pyr_sync + 1, 1u) == (unsigned int)ncta - 1) {
            atomicExch(p.pyr_sync, 0u);
            atomicExch(p.pyr_sync + 1, 0u);
        }
    }
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    mssa_tc_kernel(const __grid_constant__ TcMaps maps, const __grid_constant__ TcParams p) {
    mssa_tc_body<D, false>(maps, p, nullptr);
}

// The same attention with the launch's own pyramid (bf16 D = 128 plans).
__global__ void __launch_bounds__(kThreads, 1)
    mssa_tc_pool_kernel(const __grid_constant__ TcMaps maps, const __grid_constant__ TcParams p,
                        const __grid_constant__ PoolBatch pool) {
    mssa_tc_body<128, true>(maps, p, &pool);
}

// ---------------------------------------------------------------- host side

}  // namespace

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

namespace {

struct TcCache {
    TcMaps maps;
    // what the maps were built from
    const void* key_ptr[2 * kNumMaps + 1];
    int key_rows[2 * kNumMaps + 1];
    bool valid[2 * kNumMaps + 1];
    bool attr_set[3];  // register count of the compiled kernel checked (D 64, D 128, D 128 + pool)
    int num_sms;
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
        c->num_sms = 0;
    }
}

msf_status launch_attn_tc(msf_plan_t plan, const AttnArgs& a, cudaStream_t st, const PoolBatch* pool) {
    Plan& P = *plan;
    if (!P.tc_cache) {
        P.tc_cache = calloc(1, sizeof(TcCache));
        if (!P.tc_cache) return MSF_ERR_INVALID_ARG;
    }
    TcCache& cache = *(TcCache*)P.tc_cache;
    const long long row = (long long)P.H * P.D * 2;
    cudaError_t e;
    if (cache.num_sms == 0) {
        int dev = 0, sms = 0;
        e = cudaGetDevice(&dev);
        if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        if (e != cudaSuccess) {
            set_cuda_error((int)e);
            return MSF_ERR_CUDA;
        }
        cache.num_sms = sms;
    }

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
    // Rows of one head are D * 2 bytes (a multiple of 32): with a 32-byte
    // aligned output the epilogue stores whole 32-byte sectors.
    tp.out_v8 = ((uintptr_t)a.out % 32 == 0 && (tp.out_bstride * 2) % 32 == 0) ? 1 : 0;
    tp.status = a.status;
    tp.counters = attn_counters(P);
    tp.partials = attn_partials(P);
    tp.wait_limit = kWaitLimit;
    tp.lse = a.lse;
    tp.N = P.N;

    if (!ensure(2 * kNumMaps, &cache.maps.q, a.q, P.N, a.q_bstride)) {
        set_cuda_error((int)cudaErrorInvalidValue);
        return MSF_ERR_CUDA;
    }
    // Order groups by context length, longest first.
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
    long long total_tiles = 0;
    int item_base = 0;
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
            ts.tile0 = tg.n_tiles;
            tg.n_tiles += (sg.len + kBlockN - 1) / kBlockN;
        }
        tg.n_virt = tg.n_tiles + kItemLeadTiles;
        tg.tile_base = total_tiles;
        tg.item_base = item_base;
        total_tiles += (long long)tg.n_items * tg.n_virt;
        item_base += tg.n_items;
    }
    tp.n_groups = a.n_groups;
    tp.total_tiles = total_tiles;
    if (total_tiles == 0) return MSF_OK;
    if (item_base > P.attn_items) return MSF_ERR_STATE;
    long long ncta = cache.num_sms;
    if (ncta > P.attn_max_ctas) ncta = P.attn_max_ctas;
    if (ncta > total_tiles) ncta = total_tiles;
    if (ncta < 1) ncta = 1;
    // Data-parallel rounds: while the longest group has at least one item per
    // CTA, each CTA first takes whole items of it (no partial results), and
    // only the rest of the sequence is split evenly (stream-K).
    tp.dp_rounds = 0;
    if (tp.n_groups > 0) tp.dp_rounds = (int)(tp.g[0].n_items / ncta);
    tp.dp_stride = tp.g[0].n_virt;
    tp.t_sk = (long long)tp.dp_rounds * ncta * tp.dp_stride;
    // The launch's own pyramid (D = 128): vector-pair tasks of every job and
    // stream. Other head sizes run the pool kernel first.
    const bool own_pool = pool && pool->n > 0 && P.D == 128;
    if (pool && pool->n > 0 && !own_pool) {
        e = launch_pool(*pool, P.B, true, st);
        if (e != cudaSuccess) {
            set_cuda_error((int)e);
            return MSF_ERR_CUDA;
        }
    }
    if (own_pool) {
        int max_n = 0;
        for (int k = 0; k < pool->n; ++k) max_n = pool->j[k].out_n > max_n ? pool->j[k].out_n : max_n;
        tp.pool_tasks = max_n * (pool->row_vecs / 2);
        tp.pool_per_stream = pool->n * tp.pool_tasks;
        tp.pool_total = (long long)P.B * tp.pool_per_stream;
        tp.pyr_sync = attn_pyr_sync(P);
        for (int k = 0; k < pool->n; ++k)
            if (pool->j[k].copy_k || pool->j[k].dst_k == P.k_hist) tp.pool_ring = 1;
    }

    if (own_pool) {
        if (!cache.attr_set[2]) {
            cudaFuncAttributes fa;
            e = cudaFuncGetAttributes(&fa, mssa_tc_pool_kernel);
            if (e != cudaSuccess) {
                set_cuda_error((int)e);
                return MSF_ERR_CUDA;
            }
            if (fa.numRegs != kLaunchRegs) return MSF_ERR_UNSUPPORTED;
            cache.attr_set[2] = true;
        }
        e = set_smem_attr((const void*)mssa_tc_pool_kernel, Cfg<128>::kSmem);
        if (e != cudaSuccess) {
            set_cuda_error((int)e);
            return MSF_ERR_CUDA;
        }
        e = launch_pdl(mssa_tc_pool_kernel, dim3((unsigned)ncta), dim3(kThreads), Cfg<128>::kSmem, st,
                       cache.maps, tp, *pool);
    } else if (P.D == 128) {
        if (!cache.attr_set[1]) {
            // The warpgroup register split assumes exactly kLaunchRegs per thread.
            cudaFuncAttributes fa;
            e = cudaFuncGetAttributes(&fa, mssa_tc_kernel<128>);
            if (e != cudaSuccess) {
                set_cuda_error((int)e);
                return MSF_ERR_CUDA;
            }
            if (fa.numRegs != kLaunchRegs) return MSF_ERR_UNSUPPORTED;
            cache.attr_set[1] = true;
        }
        e = set_smem_attr((const void*)mssa_tc_kernel<128>, Cfg<128>::kSmem);
        if (e != cudaSuccess) {
            set_cuda_error((int)e);
            return MSF_ERR_CUDA;
        }
        e = launch_pdl(mssa_tc_kernel<128>, dim3((unsigned)ncta), dim3(kThreads), Cfg<128>::kSmem, st,
                       cache.maps, tp);
    } else {
        if (!cache.attr_set[0]) {
            cudaFuncAttributes fa;
            e = cudaFuncGetAttributes(&fa, mssa_tc_kernel<64>);
            if (e != cudaSuccess) {
                set_cuda_error((int)e);
                return MSF_ERR_CUDA;
            }
            if (fa.numRegs != kLaunchRegs) return MSF_ERR_UNSUPPORTED;
            cache.attr_set[0] = true;
        }
        e = set_smem_attr((const void*)mssa_tc_kernel<64>, Cfg<64>::kSmem);
        if (e != cudaSuccess) {
            set_cuda_error((int)e);
            return MSF_ERR_CUDA;
        }
        e = launch_pdl(mssa_tc_kernel<64>, dim3((unsigned)ncta), dim3(kThreads), Cfg<64>::kSmem, st,
                       cache.maps, tp);
    }
    if (e == cudaSuccess) e = cudaGetLastError();
    if (e != cudaSuccess) {
        set_cuda_error((int)e);
        return MSF_ERR_CUDA;
    }
    return MSF_OK;
}

}  // namespace msf
