// Host-side static schedule: Eq. 3 token counts, Eq. 4 query groups and
// context layout, workspace sizing, index maps. No CUDA calls here.
#include <math.h>
#include <stdlib.h>
#include <string.h>

#include <atomic>
#include <new>

#include "internal.h"

namespace msf {
static thread_local int g_last_cuda_error = 0;
static std::atomic<uint64_t> g_launches{0};
void set_cuda_error(int e) { g_last_cuda_error = e; }
void note_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }
}  // namespace msf

extern "C" uint64_t msf_kernel_launches(void) { return msf::g_launches.load(); }

using msf::Plan;

extern "C" const char* msf_status_string(msf_status s) {
    switch (s) {
        case MSF_OK: return "ok";
        case MSF_ERR_INVALID_ARG: return "invalid argument";
        case MSF_ERR_UNSUPPORTED: return "unsupported schedule or shape";
        case MSF_ERR_CUDA: return "CUDA runtime error";
        case MSF_ERR_TIMEOUT: return "device wait timed out";
        case MSF_ERR_STATE: return "invalid plan state";
        case MSF_ERR_WORKSPACE: return "workspace too small";
    }
    return "unknown status";
}

extern "C" int msf_last_cuda_error(void) { return msf::g_last_cuda_error; }

static bool is_pow2(int x) { return x >= 1 && (x & (x - 1)) == 0; }

extern "C" msf_status msf_plan_create(const msf_plan_desc* desc, msf_plan_t* out) {
    if (!desc || !out) return MSF_ERR_INVALID_ARG;
    *out = nullptr;
    const msf_plan_desc& d = *desc;
    if (d.T < 1 || d.T > MSF_MAX_STATES) return MSF_ERR_INVALID_ARG;
    if (d.grid_h < 1 || d.grid_w < 1 || d.heads < 1 || d.batch < 1) return MSF_ERR_INVALID_ARG;
    if (d.sink_tokens < 0 || d.history_frames < 0 || d.history_capacity < d.history_frames)
        return MSF_ERR_INVALID_ARG;
    if (d.dtype != MSF_DTYPE_BF16 && d.dtype != MSF_DTYPE_F32) return MSF_ERR_INVALID_ARG;
    if (d.resample != MSF_RESAMPLE_AVG && d.resample != MSF_RESAMPLE_STRIDED)
        return MSF_ERR_INVALID_ARG;
    if (d.head_dim != 64 && d.head_dim != 128) return MSF_ERR_UNSUPPORTED;
    if (d.softmax_scale < 0.f || !isfinite(d.softmax_scale)) return MSF_ERR_INVALID_ARG;
    if (d.latent_channels < 0 || d.patch < 0 || d.embed_dim < 0 || d.frames_per_state < 0)
        return MSF_ERR_INVALID_ARG;
    // Chunked states (Sec. 5.1): F latent frames per state, patches and
    // Subsample spatial. Since every stride divides one frame's grid_h, no
    // patch or pooling block crosses a frame boundary, so a chunk is handled
    // as one grid of F * grid_h rows (frames stacked in order).
    const int F = d.frames_per_state > 0 ? d.frames_per_state : 1;
    // Sec. 4.1: p_l in {p, 2p, 4p, ...}, p_1 <= ... <= p_T.
    int smax = 1;
    for (int l = 0; l < d.T; ++l) {
        if (!is_pow2(d.scales[l])) return MSF_ERR_UNSUPPORTED;
        if (l > 0 && d.scales[l] < d.scales[l - 1]) return MSF_ERR_UNSUPPORTED;
        if (d.scales[l] > smax) smax = d.scales[l];
    }
    if (d.grid_h % smax || d.grid_w % smax) return MSF_ERR_UNSUPPORTED;
    if (d.fused_append != 0 && d.fused_append != 1) return MSF_ERR_INVALID_ARG;
    // The staged head is the fine state at position 1 and needs a spare slot.
    if (d.fused_append && (d.scales[0] != 1 || d.history_capacity < 1)) return MSF_ERR_UNSUPPORTED;
    // Index arithmetic in the kernels is 32-bit per stream; keep every
    // per-stream element count well inside that range.
    long long G = (long long)F * d.grid_h * d.grid_w;
    long long row = (long long)d.heads * d.head_dim;
    if (G * row * (d.T + d.history_capacity + 8) > (1LL << 31)) return MSF_ERR_UNSUPPORTED;
    if ((long long)d.sink_tokens * row > (1LL << 31)) return MSF_ERR_UNSUPPORTED;

    Plan* p = new (std::nothrow) Plan();
    if (!p) return MSF_ERR_INVALID_ARG;
    memset((void*)p, 0, sizeof(Plan));
    p->d = d;
    p->fused = d.fused_append != 0;
    p->ring_slots = d.history_capacity + (p->fused ? 1 : 0);
    p->F = F;
    p->gh = F * d.grid_h;
    p->T = d.T;
    p->G = (int)G;
    p->H = d.heads;
    p->D = d.head_dim;
    p->B = d.batch;
    p->elem = d.dtype == MSF_DTYPE_BF16 ? 2 : 4;
    p->scale = d.softmax_scale > 0.f ? d.softmax_scale : 1.0f / sqrtf((float)d.head_dim);

    // Eq. 3: N_l = G / s_l^2, states concatenated in position order.
    int acc = 0;
    for (int l = 0; l < d.T; ++l) {
        int s = d.scales[l];
        p->st_gh[l] = p->gh / s;
        p->st_gw[l] = d.grid_w / s;
        p->st_n[l] = p->st_gh[l] * p->st_gw[l];
        p->st_off[l] = acc;
        acc += p->st_n[l];
    }
    p->N = acc;

    // Query groups: states sharing one scale are contiguous (monotone schedule).
    int ng = 0;
    for (int l = 0; l < d.T; ++l) {
        if (l == 0 || d.scales[l] != d.scales[l - 1]) {
            if (ng == MSF_MAX_GROUPS) {
                delete p;
                return MSF_ERR_UNSUPPORTED;
            }
            msf::Group& g = p->groups[ng++];
            g.scale = d.scales[l];
            g.q_begin = p->st_off[l];
            g.n_finer = l;  // every earlier state is finer
            g.pooled = p->G / (g.scale * g.scale);
        }
        p->groups[ng - 1].q_end = p->st_off[l] + p->st_n[l];
    }
    p->n_groups = ng;

    // Pyramid: per group g > 1, room for every history slot and every finer
    // window state, all pooled to G / g^2 tokens. With fused_append the part
    // is [finer states 2..n_finer | ring slots 0..capacity] (the head's level
    // lives in the ring's spare slot): the same size.
    int pyr = 0;
    for (int gi = 0; gi < ng; ++gi) {
        msf::Group& g = p->groups[gi];
        if (g.scale == 1) {
            g.pyr_offset = -1;
            g.pyr_cap = 0;
        } else {
            g.pyr_offset = pyr;
            g.pyr_cap = (d.history_capacity + g.n_finer) * g.pooled;
            pyr += g.pyr_cap;
        }
    }
    p->pyr_tokens = pyr;
    // Attention work: 256-row query blocks and 128-row context tiles, counted
    // at full history (the most tiles the schedule can ever hold).
    {
        long long items = 0, tiles = 0;
        for (int gi = 0; gi < ng; ++gi) {
            const msf::Group& g = p->groups[gi];
            long long it = (long long)p->B * p->H * ((g.q_end - g.q_begin + 255) / 256);
            long long nt = (d.sink_tokens + 127) / 128 + (p->N - g.q_begin + 127) / 128;
            if (g.scale == 1)
                nt += ((long long)p->ring_slots * p->G + 127) / 128;
            else
                nt += ((long long)(d.history_capacity + g.n_finer) * g.pooled + 127) / 128;
            items += it;
            tiles += it * nt;
        }
        if (items > (1 << 30)) {
            delete p;
            return MSF_ERR_UNSUPPORTED;
        }
        p->attn_items = (int)items;
        p->attn_max_ctas = (int)(tiles < msf::kAttnMaxCtas ? tiles : msf::kAttnMaxCtas);
    }
    p->ws_bytes = msf::workspace_bytes(*p);
    p->hist_count = d.history_frames;
    p->hist_oldest = 0;
    p->hist_spare = d.history_frames;
    *out = p;
    return MSF_OK;
}

extern "C" void msf_plan_destroy_caches(msf_plan_t plan);

extern "C" void msf_plan_destroy(msf_plan_t plan) {
    if (!plan) return;
    msf_plan_destroy_caches(plan);
    delete plan;
}

static uint64_t flops_for(const Plan& p) {
    uint64_t pairs = 0;
    for (int gi = 0; gi < p.n_groups; ++gi) {
        const msf::Group& g = p.groups[gi];
        pairs += (uint64_t)(g.q_end - g.q_begin) * (uint64_t)msf::group_nkv(p, gi);
    }
    return 4ull * p.D * p.H * p.B * pairs;
}

extern "C" msf_status msf_plan_query(msf_plan_t plan, msf_plan_info* info) {
    if (!plan || !info) return MSF_ERR_INVALID_ARG;
    const Plan& p = *plan;
    memset(info, 0, sizeof(*info));
    info->T = p.T;
    info->n_tokens = p.N;
    info->n_tokens_fine = p.T * p.G;
    info->fine_tokens = p.G;
    for (int l = 0; l < p.T; ++l) {
        info->state_offset[l] = p.st_off[l];
        info->state_tokens[l] = p.st_n[l];
        info->state_grid_h[l] = p.st_gh[l];
        info->state_grid_w[l] = p.st_gw[l];
    }
    info->n_groups = p.n_groups;
    for (int gi = 0; gi < p.n_groups; ++gi) {
        const msf::Group& g = p.groups[gi];
        msf_group_info& o = info->groups[gi];
        o.scale = g.scale;
        o.q_begin = g.q_begin;
        o.q_end = g.q_end;
        o.n_kv = msf::group_nkv(p, gi);
        o.n_pyramid = g.scale == 1 ? 0 : msf::group_npyr(p, gi);
        o.pyr_offset = g.pyr_offset;
    }
    info->history_count = p.hist_count;
    info->history_next_slot = p.fused ? p.hist_spare
                                      : (p.hist_count < p.d.history_capacity ? p.hist_count
                                                                             : p.hist_oldest);
    info->pyramid_tokens = p.pyr_tokens;
    info->frames_per_state = p.F;
    info->workspace_bytes = p.ws_bytes;
    info->backward_workspace_bytes = msf::bwd_workspace_bytes(p);
    {
        uint64_t f = 0;
        for (int gi = 0; gi < p.n_groups; ++gi) {
            const msf::Group& g = p.groups[gi];
            const uint64_t nkv = (uint64_t)msf::group_nkv(p, gi);
            const uint64_t cache = (uint64_t)p.d.sink_tokens + (uint64_t)p.hist_count * g.pooled;
            f += (uint64_t)(g.q_end - g.q_begin) * (6ull * p.D * nkv + 4ull * p.D * (nkv - cache));
        }
        info->backward_flops = f * p.H * p.B;
    }
    info->attention_flops = flops_for(p);
    // Dense reference: every state fine, every query sees sink + history + T*G.
    uint64_t nd = (uint64_t)p.T * p.G;
    info->dense_flops = 4ull * p.D * p.H * p.B * nd *
                        (uint64_t)(p.d.sink_tokens + (uint64_t)p.hist_count * p.G + nd);
    // Full resample traffic: every pooled frame reads its source and writes
    // G/g^2 tokens, for K and V.
    uint64_t bytes = 0;
    uint64_t row = (uint64_t)p.H * p.D * p.elem;
    for (int gi = 0; gi < p.n_groups; ++gi) {
        const msf::Group& g = p.groups[gi];
        if (g.scale == 1) continue;
        for (int f = 0; f < p.hist_count; ++f) bytes += (uint64_t)(p.G + g.pooled) * row;
        for (int l = 0; l < g.n_finer; ++l) bytes += (uint64_t)(p.st_n[l] + g.pooled) * row;
    }
    info->resample_bytes = 2 * bytes * p.B;
    info->pyramid_k_offset = msf::kStatusBytes;
    info->pyramid_v_offset = msf::kStatusBytes + msf::pyramid_bytes(p);
    info->attention_counter_offset =
        msf::kStatusBytes + 2 * msf::pyramid_bytes(p) + msf::msp_scratch_bytes(p);
    info->attention_counter_bytes = msf::attn_counter_bytes(p);
    return MSF_OK;
}

extern "C" msf_status msf_plan_index_map(msf_plan_t plan, int32_t group, int32_t* out,
                                         size_t cap_rows, size_t* n_rows) {
    if (!plan || !n_rows) return MSF_ERR_INVALID_ARG;
    const Plan& p = *plan;
    if (group < 0 || group >= p.n_groups) return MSF_ERR_INVALID_ARG;
    if (cap_rows > 0 && !out) return MSF_ERR_INVALID_ARG;
    const int g = p.groups[group].scale;
    size_t n = 0;
    auto put = [&](int kind, int frame, int stride, int r, int c) {
        if (n < cap_rows) {
            int32_t* o = out + 5 * n;
            o[0] = kind;
            o[1] = frame;
            o[2] = stride;
            o[3] = r;
            o[4] = c;
        }
        ++n;
    };
    for (int t = 0; t < p.d.sink_tokens; ++t) put(0, 0, 1, t, 0);
    auto put_frame = [&](int kind, int frame, int st, int gh, int gw) {
        for (int i = 0; i < gh; ++i)
            for (int j = 0; j < gw; ++j) put(kind, frame, st, i, j);
    };
    if (!p.fused) {
        for (int f = 0; f < p.hist_count; ++f) put_frame(1, f, g, p.gh / g, p.d.grid_w / g);
        for (int l = 0; l < p.T; ++l) {
            int s = p.d.scales[l];
            int st = s < g ? g / s : 1;
            put_frame(2, l, st, p.st_gh[l] / st, p.st_gw[l] / st);
        }
    } else {
        // Kernel order: [finer states 2.. pooled | ring slots 0..count | window from k_win].
        const int first_win = g == 1 ? 1 : 0;
        if (g > 1)
            for (int l = 1; l < p.groups[group].n_finer; ++l)
                put_frame(2, l, g / p.d.scales[l], p.gh / g, p.d.grid_w / g);
        for (int slot = 0; slot <= p.hist_count; ++slot) {
            if (slot == p.hist_spare)
                put_frame(2, 0, g, p.gh / g, p.d.grid_w / g);
            else
                put_frame(1, slot, g, p.gh / g, p.d.grid_w / g);
        }
        for (int l = first_win; l < p.T; ++l) {
            int s = p.d.scales[l];
            if (s < g) continue;
            put_frame(2, l, 1, p.st_gh[l], p.st_gw[l]);
        }
    }
    *n_rows = n;
    return MSF_OK;
}
