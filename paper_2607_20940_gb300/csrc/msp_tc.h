// Fused MSP kernels (patchify + tier embedding, de-embedding + unpatchify) on
// the sm_103a tensor cores; see msp_tc.cu.
#pragma once
#include <cuda_runtime.h>

#include "kernels.h"

namespace msf {

// One run of consecutive window states of one tier (same patch edge, same
// weight): their tokens are contiguous in the output.
struct MspEmbedRun {
    const void* w;  // [E, K] bf16 tier weight, K = C * P * P contiguous
    int M;          // tokens of the run per stream
    int l0;         // first state
    int n_l;        // tokens per state
    int gw;         // tokens per grid row (Wl / P)
    int P;          // patch edge in latent pixels
    int K;          // C * P * P
    int tok_off;    // first token row of the run
};

bool msp_embed_supported(const MspEmbedRun* runs, int n, int E);
// Up to kMaxGemmProblems runs in one launch.
cudaError_t launch_msp_embed(const MspEmbedRun* runs, int n, const MspShape& sh, int E, const void* latent,
                             void* tokens, long long tok_bstride, int batch, unsigned int* status,
                             cudaStream_t st);

// De-embedding + unpatchify of M tokens (F = C*P*P features, E = K) of one
// window position; the split-K reduction stays inside a thread-block cluster.
bool msp_deembed_supported(int M, int F, int E);
cudaError_t launch_msp_deembed(const void* tokens, long long tok_bstride_elems, int tok_rows, int tok_row0,
                               const void* w_out, int M, int F, int E, const MspShape& sh, int P, void* latent,
                               int batch, unsigned int* status, cudaStream_t st);

}  // namespace msf
