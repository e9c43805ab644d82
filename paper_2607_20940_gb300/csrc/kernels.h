// Launch interfaces of the CUDA kernels (host side of each .cu file).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "internal.h"

namespace msf {

// Set the dynamic shared-memory limit of kernel `fn` to `bytes` (and, if
// carveout >= 0, its preferred shared-memory carveout in percent) on the
// current device, once per (kernel, device): the attribute belongs to a
// device's context, so a process that launches on several devices needs it on
// each. Thread-safe.
cudaError_t set_smem_attr(const void* fn, int bytes, int carveout = -1);

// One block that waits, with the bounded wait of the tcgen05 kernels, on an
// mbarrier nothing arrives at, then raises the TIMEOUT bit of *status.
cudaError_t launch_wait_timeout_selftest(unsigned int* status, long long limit_cycles, cudaStream_t st);

// Launch with programmatic stream serialisation (see grid_dep_wait in
// ptx.cuh): the kernel's launch and prologue may overlap the previous kernel.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t st, Args... args) {
    cudaLaunchConfig_t cfg;
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    note_launch();
    return cudaLaunchKernelEx(&cfg, kernel, args...);
}

// The same with thread-block clusters of `cluster` CTAs.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl_cluster(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                               cudaStream_t st, dim3 cluster, Args... args) {
    cudaLaunchConfig_t cfg;
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = cluster.x;
    attr[1].val.clusterDim.y = cluster.y;
    attr[1].val.clusterDim.z = cluster.z;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    note_launch();
    return cudaLaunchKernelEx(&cfg, kernel, args...);
}

// ------------------------------------------------------------------ pooling
struct PoolJob {
    const char* src_k;      // source block, stream 0
    const char* src_v;
    char* dst_k;            // destination block, stream 0
    char* dst_v;
    long long src_bstride;  // bytes between streams
    long long dst_bstride;
    int src_gw;             // source grid width (tokens)
    int out_gw;             // pooled grid width
    int out_n;              // pooled tokens
    int sigma;              // stride (1 = copy)
    // Optional: also write every source token read to this block (same token
    // index as in the source, so the whole source is copied when the pooled
    // blocks tile it). NULL = no copy. Requires sigma <= 4.
    char* copy_k;
    char* copy_v;
    long long copy_bstride;
};
constexpr int kMaxPoolJobs = 40;
struct PoolBatch {
    PoolJob j[kMaxPoolJobs];
    int n;
    int row_vecs;  // 16-byte vectors per token row (H*D*elem/16)
    int mode;      // msf_resample_mode
};
cudaError_t launch_pool(const PoolBatch& jobs, int batch, bool bf16, cudaStream_t st);

// -------------------------------------------------------------------- MSP
struct MspShape {
    int T, C, Hl, Wl, patch;
    int scales[MSF_MAX_STATES];
};
// Raw patchify of states [l0, l0 + n_states) (n_states < 0: to the end) into
// their blocks of the [B, T, C*Hl*Wl] raw layout.
cudaError_t launch_patchify_raw(const void* latent, void* raw, const MspShape& sh, int batch,
                                bool bf16, cudaStream_t st, int l0 = 0, int n_states = -1);
cudaError_t launch_unpatchify_raw(const void* raw, void* latent, const MspShape& sh, int position,
                                  long long raw_bstride, int raw_offset, int batch, bool bf16,
                                  cudaStream_t st);

// Sum `splits` fp32 partial token blocks [split][B][N_l * C*P^2] (fixed
// order), round once to bf16 and rearrange into the latent [B, C, Hl, Wl].
cudaError_t launch_unpatchify_splitk(const float* part, int splits, void* latent, const MspShape& sh,
                                     int position, int batch, cudaStream_t st);

struct GemmArgs {
    const void* A;  // [M, K] (+ a_bstride per batch), element strides
    const void* B;  // [N, K]
    void* C;        // [M, N]
    int M, N, K;
    long long lda, ldb, ldc;
    long long a_bstride, c_bstride;
};
cudaError_t launch_gemm_nt_simt(const GemmArgs& g, int batch, bool bf16, cudaStream_t st);

// --------------------------------------------------------------- attention
// One context segment of a query group: rows [row0, row0 + len) of a
// [B, rows_total, H, D] tensor pair.
struct Segment {
    const char* k;
    const char* v;
    long long bstride;  // bytes between streams
    int row0;
    int len;
    int rows_total;     // rows of the underlying tensor (TMA extent)
    int map_id;         // which tensor map (tensor-core kernel)
};
constexpr int kMaxSeg = 3;
struct AttnGroup {
    int q_begin, q_end;
    int n_seg;
    Segment seg[kMaxSeg];
};
struct AttnArgs {
    const char* q;
    char* out;
    long long q_bstride;  // bytes between streams of q/out/k_win
    int H, D, B;
    float scale_log2;     // softmax scale * log2(e)
    int n_groups;
    AttnGroup g[MSF_MAX_GROUPS];
    unsigned int* status;
    float* lse;           // optional [B, H, N] row log-sum-exp (natural log); NULL = none
    int N;                // query rows per stream
};
cudaError_t launch_attn_simt(const AttnArgs& a, bool bf16, cudaStream_t st);

// ---------------------------------------------------------- MSSA backward
//
// Context rows whose key/value gradients flow back to window tokens: rows
// [row0, row0 + len) of a [B, rows_total, H, D] tensor pair (k, v). Their
// gradients go to rows [crow0, crow0 + len) of the context-gradient buffers
// (one run after another, all groups). sigma 1: row row0 + r is window token
// dst0 + r. sigma > 1: row r is token (r / out_gw, r % out_gw) of a pooled
// state whose fine grid (src_gw wide) starts at window token dst0.
struct GradSeg {
    const char* k;
    const char* v;
    long long bstride;  // bytes between streams
    int row0, len, rows_total, map_id;
    int sigma, dst0, src_gw, out_gw;
    int crow0;
};
constexpr int kMaxGradSeg = MSF_MAX_STATES + 1;
struct BwdGroup {
    int q_begin, q_end;
    int n_gseg;
    GradSeg gseg[kMaxGradSeg];
};
// Per-launch arguments shared by the backward kernels.
struct BwdCommon {
    const char* q;      // [B, N, H, D]
    const char* dout;   // [B, N, H, D]
    const char* out;    // [B, N, H, D]
    const float* lse;   // [B, H, N], natural log
    float* delta;       // [B, H, N]: rowsum(dout * out)
    float* dk_ctx;      // [B, R, H, D] fp32 gradients of the window-derived context
    float* dv_ctx;      //   rows of every group (GradSeg.crow0 places each run)
    int R;
    long long bstride;  // bytes between streams of q/dout/out/dq
    int H, D, B, N;
    float scale;        // softmax scale
    float scale_log2;   // scale * log2(e)
};
// The adjoint of Subsample, summed over groups: window token t of state l
// receives, from each entry of state l, context-gradient row
//   sigma 1:  crow0 + (t - dst0)
//   sigma > 1: crow0 + (i / sigma) * out_gw + j / sigma, weight 1/sigma^2 (AVG),
//              or only when sigma divides i and j, weight 1 (STRIDED),
// where (i, j) is t's position on the state's grid (src_gw wide).
struct GatherEntry {
    int crow0, dst0, sigma, src_gw, out_gw;
};
struct GatherArgs {
    int T;
    int st_off[MSF_MAX_STATES + 1];
    int n_ent[MSF_MAX_STATES];
    GatherEntry e[MSF_MAX_STATES][MSF_MAX_GROUPS];
    int mode;  // msf_resample_mode
};
cudaError_t launch_bwd_delta(const BwdCommon& c, bool bf16, cudaStream_t st);
// dq for every query of every group (context of each group as in the forward).
cudaError_t launch_bwd_dq_simt(const BwdCommon& c, const AttnArgs& a, void* dq, bool bf16,
                               cudaStream_t st);
// Context-row gradients of one group's window-derived rows.
cudaError_t launch_bwd_dkdv_simt(const BwdCommon& c, const BwdGroup& g, bool bf16,
                                 cudaStream_t st);
// dk_win, dv_win from the context-row gradients (adjoint of Subsample, sum
// over groups, one rounding to the dtype).
cudaError_t launch_bwd_gather(const BwdCommon& c, const GatherArgs& g, void* dk, void* dv,
                              bool bf16, cudaStream_t st);

}  // namespace msf
