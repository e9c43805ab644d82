// Tensor-core MSSA attention (tcgen05 + TMA) launcher interface.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>

#include "internal.h"
#include "kernels.h"

namespace msf {

// Tensor-map slots of the context segments.
enum : int { kMapSink = 0, kMapHist = 1, kMapWin = 2, kMapPyr0 = 3 };
// Segments of groups with a pyramid part use map kMapPyr0 + group index;
// build_attn_args marks them kMapPyr and the launcher resolves the slot.
constexpr int kMapPyr = -1;
constexpr int kNumMaps = kMapPyr0 + MSF_MAX_GROUPS;

// With `pool` (bf16 jobs), the launch also builds that K/V pyramid: every CTA
// pools a share of it first, and tiles of pyramid segments wait until all
// shares are written.
msf_status launch_attn_tc(msf_plan_t plan, const AttnArgs& a, cudaStream_t st,
                          const PoolBatch* pool = nullptr);
// Tensor map of a [B, rows, H, D] bf16 tensor as 4-D {D, H, rows, B}, boxes of
// 64 x 1 x 128 x 1 with 128-byte swizzle (one K-major MMA chunk); rows past
// `rows` load as zeros.
bool encode_rows(CUtensorMap* m, const void* base, int D, int H, int rows, int B,
                 long long bstride_bytes);
void tc_cache_free(msf_plan_t plan);
void tc_cache_invalidate(msf_plan_t plan);

}  // namespace msf
