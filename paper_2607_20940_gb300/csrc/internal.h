// Internal plan state shared by the host plan code and the kernel launchers.
#pragma once

#include <stddef.h>
#include <stdint.h>

#include "../../include/msf.h"

namespace msf {

struct Group {
    int scale;       // g
    int q_begin, q_end;
    int n_finer;     // window states with s_l < g (pooled into the pyramid)
    int pooled;      // G / g^2 tokens per pooled frame at this scale
    int pyr_offset;  // token offset of the group's pyramid part (per stream), -1 for g == 1
    int pyr_cap;     // tokens reserved: (history_capacity + n_finer) * pooled
};

}  // namespace msf

// The opaque plan of the C ABI.
struct msf_plan {
    msf_plan_desc d;
    int T, G, N, H, D, B;
    bool fused;      // fused_append: history update folded into the resample
    int ring_slots;  // history ring slots: capacity (+1 spare with fused_append)
    int F;   // latent frames per state
    int gh;  // rows of a fine state's grid: F latent frames stacked (F * grid_h)
    int elem;  // bytes per element
    int st_off[MSF_MAX_STATES], st_n[MSF_MAX_STATES];
    int st_gh[MSF_MAX_STATES], st_gw[MSF_MAX_STATES];
    int n_groups;
    msf::Group groups[MSF_MAX_GROUPS];
    int pyr_tokens;   // per stream
    // tensor-core attention scheduling state in the workspace
    int attn_items;     // 256-row query blocks over all groups, streams and heads
    int attn_max_ctas;  // persistent CTAs the partial-result slots are sized for
    size_t ws_bytes;
    float scale;      // softmax scale

    // history ring state (host side)
    int hist_count;
    int hist_oldest;
    int hist_spare;   // fused_append: ring slot the next resample stages the head in

    // bound buffers
    bool bound;
    void* ws;
    size_t ws_size;
    const void* k_sink;
    const void* v_sink;
    void* k_hist;
    void* v_hist;

    // opaque per-kernel caches (tensor maps etc.)
    void* tc_cache;
};

namespace msf {
using Plan = ::msf_plan;

// Workspace layout: [status area | pyramid K | pyramid V | MSP scratch | attention
// merge counters | attention partial slots | de-embedding split partials | tier codes]
constexpr size_t kStatusBytes = 256;
inline size_t round256(size_t x) { return (x + 255) / 256 * 256; }
inline size_t pyramid_bytes(const Plan& p) {
    return round256((size_t)p.B * p.pyr_tokens * p.H * p.D * p.elem);
}
// Raw MSP tokens of every state: [B, T, C*Hl*Wl].
inline size_t msp_scratch_bytes(const Plan& p) {
    if (p.d.latent_channels <= 0 || p.d.patch <= 0) return 0;
    size_t per = (size_t)p.d.latent_channels * p.d.patch * p.gh * p.d.patch * p.d.grid_w;
    return round256((size_t)p.B * p.T * per * p.elem);
}
// Tensor-core attention (bf16 plans): one merge counter per query block, and
// two partial-result slots per persistent CTA, each [256 rows][D] fp32 output
// followed by [256 rows][2] fp32 (running max, running sum).
constexpr int kAttnMaxCtas = 160;
constexpr int kAttnBlockRows = 256;
// After the counters, two words of a launch that builds its own pyramid
// (CTAs whose pooled share is written, CTAs finished; reset by its last CTA).
inline size_t attn_counter_bytes(const Plan& p) {
    return p.elem == 2 ? round256((size_t)p.attn_items * 4 + 8) : 0;
}
inline size_t attn_slot_floats(const Plan& p) { return (size_t)kAttnBlockRows * (p.D + 2); }
inline size_t attn_partial_bytes(const Plan& p) {
    return p.elem == 2 ? round256((size_t)2 * p.attn_max_ctas * attn_slot_floats(p) * 4) : 0;
}
// fp32 partial sums of a split-K de-embedding: [splits][B][C*Hl*Wl].
constexpr int kMaxDeembedSplits = 8;
inline size_t msp_split_bytes(const Plan& p) {
    if (p.d.latent_channels <= 0 || p.d.patch <= 0 || p.elem != 2) return 0;
    size_t per = (size_t)p.d.latent_channels * p.d.patch * p.gh * p.d.patch * p.d.grid_w;
    return round256((size_t)kMaxDeembedSplits * p.B * per * 4);
}
// LoRA codes of the tier modules (msf_patchify_tiers, msf_unpatchify_tier):
// [B, N, 64] bf16, the rank-r code of every window token zero-padded to 64.
constexpr int kTierCodeCols = 64;
inline size_t tier_codes_bytes(const Plan& p) {
    if (p.d.latent_channels <= 0 || p.d.patch <= 0 || p.elem != 2 || p.d.embed_dim <= 0) return 0;
    return round256((size_t)p.B * p.N * kTierCodeCols * 2);
}
// Backward workspace (caller-provided per msf_mssa_backward call):
// [delta fp32 [B, H, N] | dk_ctx fp32 [B, R, H, D] | dv_ctx fp32 [B, R, H, D]],
// R = rows of every group's context that come from the window (the rows
// that receive key/value gradients): N for g = 1, n_finer * G/g^2 + the
// window suffix for g > 1.
inline int bwd_ctx_rows(const Plan& p) {
    int r = 0;
    for (int gi = 0; gi < p.n_groups; ++gi) {
        const Group& g = p.groups[gi];
        r += g.scale == 1 ? p.N : g.n_finer * g.pooled + (p.N - g.q_begin);
    }
    return r;
}
inline size_t bwd_delta_bytes(const Plan& p) { return round256((size_t)p.B * p.H * p.N * 4); }
inline size_t bwd_ctx_bytes(const Plan& p) {
    return round256((size_t)p.B * bwd_ctx_rows(p) * p.H * p.D * 4);
}
inline size_t bwd_workspace_bytes(const Plan& p) { return bwd_delta_bytes(p) + 2 * bwd_ctx_bytes(p); }
inline size_t workspace_bytes(const Plan& p) {
    return kStatusBytes + 2 * pyramid_bytes(p) + msp_scratch_bytes(p) + attn_counter_bytes(p) +
           attn_partial_bytes(p) + msp_split_bytes(p) + tier_codes_bytes(p);
}
inline unsigned int* status_word(const Plan& p) { return (unsigned int*)p.ws; }
inline char* pyr_k(const Plan& p) { return (char*)p.ws + kStatusBytes; }
inline char* pyr_v(const Plan& p) { return (char*)p.ws + kStatusBytes + pyramid_bytes(p); }
inline char* msp_scratch(const Plan& p) {
    return (char*)p.ws + kStatusBytes + 2 * pyramid_bytes(p);
}
inline unsigned int* attn_counters(const Plan& p) {
    return (unsigned int*)(msp_scratch(p) + msp_scratch_bytes(p));
}
inline unsigned int* attn_pyr_sync(const Plan& p) { return attn_counters(p) + p.attn_items; }
inline float* attn_partials(const Plan& p) {
    return (float*)((char*)attn_counters(p) + attn_counter_bytes(p));
}
inline float* msp_split(const Plan& p) {
    return (float*)((char*)attn_partials(p) + attn_partial_bytes(p));
}
inline char* tier_codes(const Plan& p) { return (char*)msp_split(p) + msp_split_bytes(p); }

// Number of context tokens of group gi with the current history count.
inline int group_nkv(const Plan& p, int gi) {
    const Group& g = p.groups[gi];
    int n = p.d.sink_tokens + p.hist_count * g.pooled;
    for (int l = 0; l < p.T; ++l) {
        int s = p.d.scales[l];
        n += (s < g.scale) ? g.pooled : p.st_n[l];
    }
    return n;
}
// Tokens of the pyramid part of group gi (history@g + finer window states).
inline int group_npyr(const Plan& p, int gi) {
    const Group& g = p.groups[gi];
    return (p.hist_count + g.n_finer) * g.pooled;
}

void set_cuda_error(int e);
// Count one kernel launch (see msf_kernel_launches).
void note_launch();

// Device status codes written into the status word.
constexpr unsigned int kDevTimeout = 1u;

}  // namespace msf
