// Fused MSP kernels (patchify + tier embedding, de-embedding + unpatchify) on
// the sm_103a tensor cores; see msp_tc.cu.
#pragma once
#include <cuda_runtime.h>

#include "kernels.h"

namespace msf {

// One run of consecutive window states of one tier (same patch edge, same
// weight): their tokens are contiguous in the output.
struct MspEmbedRun {
    const void* w;  // [w_rows, K] bf16 tier weight, K = C * P * P contiguous
    int M;          // tokens of the run per stream
    int l0;         // first state
    int n_l;        // tokens per state
    int gw;         // tokens per grid row (Wl / P)
    int P;          // patch edge in latent pixels
    int K;          // C * P * P
    int tok_off;    // first token row of the run
    int w_rows = 0;             // rows of w (0: E); output columns past them are zero
    float scale = 1.0f;         // applied to the accumulator before rounding
    // LoRA adapter of the tier (Sec. 4.1): one more K chunk whose A operand is
    // the run's rank-r codes (64-wide bf16 rows, zero past r; the codes of
    // the run's token m of stream b at codes + b * codes_bstride + m * 64)
    // and whose B operand is the up projection [E, r] (columns past r read
    // as zeros).
    const void* lora_up = nullptr;
    int rank = 0;
    const void* codes = nullptr;
    long long codes_bstride = 0;  // elements
};

bool msp_embed_supported(const MspEmbedRun* runs, int n, int E);
// Up to kMaxGemmProblems runs in one launch. With `pool` (bf16 jobs) the
// same launch also runs those K/V pyramid jobs on `pool_ctas` more CTAs per
// stream after the embedding tiles: they read and write buffers the
// embedding does not touch, so the two share the SMs of one launch.
cudaError_t launch_msp_embed(const MspEmbedRun* runs, int n, const MspShape& sh, int E, const void* latent,
                             void* tokens, long long tok_bstride, int batch, unsigned int* status,
                             cudaStream_t st, const PoolBatch* pool = nullptr, int pool_ctas = 0);

// The coarse tier's extras of a de-embedding (Sec. 4.1): K chunks added to
// the E / 64 token chunks of the same accumulation.
struct DeembedTier {
    // LoRA: codes (64-wide bf16 rows laid out like the tokens: row t of
    // stream b at codes + b * codes_bstride + t * 64, zero past the rank) times
    // the up projection [F, rank]. NULL up: no LoRA chunk.
    const void* codes = nullptr;
    long long codes_bstride = 0;  // elements
    const void* up = nullptr;
    int rank = 0;
    // Latent residual: the state's raw patch vectors [M, F] (stream b at
    // xraw + b * xraw_bstride) times residual [F, F]. NULL residual: none.
    const void* xraw = nullptr;
    long long xraw_bstride = 0;  // elements
    const void* residual = nullptr;
};

// De-embedding + unpatchify of M tokens (F = C*P*P features, E = K) of one
// window position; the split-K reduction stays inside a thread-block cluster.
bool msp_deembed_supported(int M, int F, int E);
cudaError_t launch_msp_deembed(const void* tokens, long long tok_bstride_elems, int tok_rows, int tok_row0,
                               const void* w_out, int M, int F, int E, const MspShape& sh, int P, void* latent,
                               int batch, unsigned int* status, cudaStream_t st,
                               const DeembedTier* tier = nullptr);

// The same cluster split-K kernel with a plain row output: out[b][m][0, 64)
// = scale * sum_k tokens[b][tok_row0 + m][k] * w[n][k] for the 64 output
// columns n (w has w_rows <= 64 rows; the others read as zeros), rounded once
// to bf16; E a multiple of 64.
cudaError_t launch_msp_rows_splitk(const void* tokens, long long tok_bstride_elems, int tok_rows, int tok_row0,
                                   const void* w, int w_rows, int M, int E, void* out, long long out_bstride,
                                   int out_ld, float scale, int batch, unsigned int* status, cudaStream_t st);

}  // namespace msf
