// C ABI entry points that touch the device: binding, MSP, KV pyramid,
// attention, history update, device status.
#include <cuda_runtime.h>
#include <string.h>

#include <mutex>
#include <utility>
#include <vector>

#include "attn_bwd_tc.h"
#include "attn_tc.h"
#include "gemm_tc.h"
#include "msp_tc.h"
#include "internal.h"
#include "kernels.h"
#include "ptx.cuh"

using msf::Plan;

namespace msf {

cudaError_t set_smem_attr(const void* fn, int bytes, int carveout) {
    static std::mutex mu;
    static std::vector<std::pair<const void*, int>> done;  // (kernel, device)
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    std::lock_guard<std::mutex> lock(mu);
    for (const auto& d : done)
        if (d.first == fn && d.second == dev) return cudaSuccess;
    e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (e == cudaSuccess && carveout >= 0)
        e = cudaFuncSetAttribute(fn, cudaFuncAttributePreferredSharedMemoryCarveout, carveout);
    if (e == cudaSuccess) done.emplace_back(fn, dev);
    return e;
}

}  // namespace msf

namespace {

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

msf_status cuda_status(cudaError_t e) {
    if (e == cudaSuccess) return MSF_OK;
    msf::set_cuda_error((int)e);
    return MSF_ERR_CUDA;
}

size_t row_bytes(const Plan& p) { return (size_t)p.H * p.D * p.elem; }

// Jobs that pool the history frames (full mode) and the window states finer
// than each group's scale into that group's pyramid part.
void add_window_jobs(const Plan& p, const void* k_win, const void* v_win, bool with_history,
                     msf::PoolBatch& jb) {
    const size_t row = row_bytes(p);
    const long long win_bs = (long long)p.N * row;
    const long long hist_bs = (long long)p.ring_slots * p.G * row;
    const long long pyr_bs = (long long)p.pyr_tokens * row;
    auto job = [&](const char* sk, const char* sv, long long sbs, char* dk, char* dv,
                   int src_gw, int out_gw, int out_n, int sigma) -> msf::PoolJob& {
        msf::PoolJob& j = jb.j[jb.n++];
        j.src_k = sk;
        j.src_v = sv;
        j.dst_k = dk;
        j.dst_v = dv;
        j.src_bstride = sbs;
        j.dst_bstride = pyr_bs;
        j.src_gw = src_gw;
        j.out_gw = out_gw;
        j.out_n = out_n;
        j.sigma = sigma;
        return j;
    };
    // With fused_append the pyramid part of g is [finer states 2.. | ring slots]
    // and the head (state 1) is staged in the ring's spare slot.
    bool head_copied = false;
    for (int gi = 0; gi < p.n_groups; ++gi) {
        const msf::Group& g = p.groups[gi];
        if (g.scale == 1) continue;
        const int ring0 = p.fused ? g.n_finer - 1 : 0;  // pyramid slot of ring slot 0
        if (with_history) {
            for (int f = 0; f < (p.fused ? p.hist_count + 1 : p.hist_count); ++f) {
                if (p.fused && f == p.hist_spare) continue;
                size_t so = (size_t)f * p.G * row;
                size_t dof = (size_t)(g.pyr_offset + (ring0 + f) * g.pooled) * row;
                job((const char*)p.k_hist + so, (const char*)p.v_hist + so, hist_bs,
                    msf::pyr_k(p) + dof, msf::pyr_v(p) + dof, p.d.grid_w, p.d.grid_w / g.scale,
                    g.pooled, g.scale);
            }
        }
        for (int l = 0; l < g.n_finer; ++l) {
            int slot;  // pyramid slot of this pooled state
            if (!p.fused)
                slot = p.hist_count + l;
            else
                slot = l == 0 ? ring0 + p.hist_spare : l - 1;
            size_t so = (size_t)p.st_off[l] * row;
            size_t dof = (size_t)(g.pyr_offset + slot * g.pooled) * row;
            msf::PoolJob& j = job((const char*)k_win + so, (const char*)v_win + so, win_bs,
                                  msf::pyr_k(p) + dof, msf::pyr_v(p) + dof, p.st_gw[l],
                                  p.d.grid_w / g.scale, g.pooled, g.scale / p.d.scales[l]);
            if (p.fused && l == 0 && !head_copied && g.scale <= 4) {
                // the same read also writes the fine head into the spare ring slot
                const size_t ro = (size_t)p.hist_spare * p.G * row;
                j.copy_k = (char*)p.k_hist + ro;
                j.copy_v = (char*)p.v_hist + ro;
                j.copy_bstride = hist_bs;
                head_copied = true;
            }
        }
    }
    if (p.fused && !head_copied) {
        // no coarser level: a plain copy of the head into the spare slot
        const size_t ro = (size_t)p.hist_spare * p.G * row;
        msf::PoolJob& j = job((const char*)k_win, (const char*)v_win, win_bs, (char*)p.k_hist + ro,
                              (char*)p.v_hist + ro, p.d.grid_w, p.d.grid_w, p.G, 1);
        j.dst_bstride = hist_bs;
    }
}

int count_window_jobs(const Plan& p, bool with_history) {
    int n = p.fused ? 1 : 0;
    for (int gi = 0; gi < p.n_groups; ++gi) {
        const msf::Group& g = p.groups[gi];
        if (g.scale == 1) continue;
        n += g.n_finer + (with_history ? p.hist_count : 0);
    }
    return n;
}

// The context segments of every query group (Eq. 4 order: sink, history,
// window), pointing at the bound buffers, the pyramid and k_win/v_win.
void build_attn_args(const Plan& p, const void* q, const void* k_win, const void* v_win,
                     void* out, msf::AttnArgs& a) {
    memset(&a, 0, sizeof(a));
    const size_t row = row_bytes(p);
    a.q = (const char*)q;
    a.out = (char*)out;
    a.q_bstride = (long long)p.N * row;
    a.H = p.H;
    a.D = p.D;
    a.B = p.B;
    a.scale_log2 = p.scale * 1.4426950408889634f;
    a.n_groups = p.n_groups;
    a.status = msf::status_word(p);
    a.N = p.N;
    for (int gi = 0; gi < p.n_groups; ++gi) {
        const msf::Group& g = p.groups[gi];
        msf::AttnGroup& ag = a.g[gi];
        ag.q_begin = g.q_begin;
        ag.q_end = g.q_end;
        int ns = 0;
        if (p.d.sink_tokens > 0) {
            msf::Segment& s = ag.seg[ns++];
            s.k = (const char*)p.k_sink;
            s.v = (const char*)p.v_sink;
            s.bstride = (long long)p.d.sink_tokens * row;
            s.row0 = 0;
            s.len = p.d.sink_tokens;
            s.rows_total = p.d.sink_tokens;
            s.map_id = msf::kMapSink;
        }
        // fused_append: the head (state 1) is read from the ring's spare slot,
        // which sits inside the used slots [0, count]; the window part starts
        // after it.
        const int ring_used = p.fused ? p.hist_count + 1 : p.hist_count;
        int win0 = g.q_begin;
        if (g.scale == 1) {
            if (ring_used > 0) {
                msf::Segment& s = ag.seg[ns++];
                s.k = (const char*)p.k_hist;
                s.v = (const char*)p.v_hist;
                s.bstride = (long long)p.ring_slots * p.G * row;
                s.row0 = 0;
                s.len = ring_used * p.G;
                s.rows_total = p.ring_slots * p.G;
                s.map_id = msf::kMapHist;
            }
            if (p.fused) win0 = p.st_n[0];
        } else {
            int n = msf::group_npyr(p, gi);
            if (n > 0) {
                msf::Segment& s = ag.seg[ns++];
                s.k = msf::pyr_k(p);
                s.v = msf::pyr_v(p);
                s.bstride = (long long)p.pyr_tokens * row;
                s.row0 = g.pyr_offset;
                s.len = n;
                s.rows_total = p.pyr_tokens;
                s.map_id = msf::kMapPyr;
            }
        }
        if (win0 < p.N) {
            msf::Segment& s = ag.seg[ns++];
            s.k = (const char*)k_win;
            s.v = (const char*)v_win;
            s.bstride = (long long)p.N * row;
            s.row0 = win0;
            s.len = p.N - win0;
            s.rows_total = p.N;
            s.map_id = msf::kMapWin;
        }
        ag.n_seg = ns;
    }
}

}  // namespace

extern "C" void msf_plan_destroy_caches(msf_plan_t plan) { msf::tc_cache_free(plan); }

extern "C" msf_status msf_plan_bind(msf_plan_t plan, void* workspace, size_t workspace_bytes,
                                    const void* k_sink, const void* v_sink, void* k_hist,
                                    void* v_hist) {
    if (!plan || !workspace) return MSF_ERR_INVALID_ARG;
    Plan& p = *plan;
    if (workspace_bytes < p.ws_bytes) return MSF_ERR_WORKSPACE;
    if (!aligned16(workspace)) return MSF_ERR_INVALID_ARG;
    if (p.d.sink_tokens > 0 && (!k_sink || !v_sink || !aligned16(k_sink) || !aligned16(v_sink)))
        return MSF_ERR_INVALID_ARG;
    if (p.d.history_capacity > 0 &&
        (!k_hist || !v_hist || !aligned16(k_hist) || !aligned16(v_hist)))
        return MSF_ERR_INVALID_ARG;
    p.ws = workspace;
    p.ws_size = workspace_bytes;
    p.k_sink = k_sink;
    p.v_sink = v_sink;
    p.k_hist = k_hist;
    p.v_hist = v_hist;
    p.hist_count = p.d.history_frames;
    p.hist_oldest = 0;
    p.hist_spare = p.d.history_frames;
    p.bound = true;
    msf::tc_cache_invalidate(plan);
    cudaError_t e = cudaMemset(msf::status_word(p), 0, msf::kStatusBytes);
    if (e == cudaSuccess && msf::attn_counter_bytes(p) > 0)
        e = cudaMemset(msf::attn_counters(p), 0, msf::attn_counter_bytes(p));
    if (e == cudaSuccess) e = cudaDeviceSynchronize();
    return cuda_status(e);
}

extern "C" msf_status msf_kv_resample(msf_plan_t plan, const void* k_win, const void* v_win,
                                      int32_t flags, void* stream) {
    if (!plan || !k_win || !v_win) return MSF_ERR_INVALID_ARG;
    const Plan& p = *plan;
    if (!p.bound) return MSF_ERR_STATE;
    if (!aligned16(k_win) || !aligned16(v_win)) return MSF_ERR_INVALID_ARG;
    if (flags != MSF_RESAMPLE_FULL && flags != MSF_RESAMPLE_WINDOW_ONLY) return MSF_ERR_INVALID_ARG;
    const bool with_hist = flags == MSF_RESAMPLE_FULL;
    if (count_window_jobs(p, with_hist) > msf::kMaxPoolJobs) return MSF_ERR_UNSUPPORTED;
    msf::PoolBatch jb;
    memset(&jb, 0, sizeof(jb));
    jb.row_vecs = (int)(row_bytes(p) / 16);
    jb.mode = p.d.resample;
    add_window_jobs(p, k_win, v_win, with_hist, jb);
    return cuda_status(msf::launch_pool(jb, p.B, p.elem == 2, (cudaStream_t)stream));
}

extern "C" msf_status msf_history_append(msf_plan_t plan, const void* k_win, const void* v_win,
                                         void* stream) {
    if (!plan || !k_win || !v_win) return MSF_ERR_INVALID_ARG;
    Plan& p = *plan;
    if (!p.bound || p.d.history_capacity == 0 || p.d.scales[0] != 1 || p.fused)
        return MSF_ERR_STATE;
    if (!aligned16(k_win) || !aligned16(v_win)) return MSF_ERR_INVALID_ARG;
    const int slot = p.hist_count < p.d.history_capacity ? p.hist_count : p.hist_oldest;
    const size_t row = row_bytes(p);
    msf::PoolBatch jb;
    memset(&jb, 0, sizeof(jb));
    jb.row_vecs = (int)(row / 16);
    jb.mode = p.d.resample;
    {
        // the head state (position 1, fine) into its ring slot
        msf::PoolJob& j = jb.j[jb.n++];
        j.src_k = (const char*)k_win;
        j.src_v = (const char*)v_win;
        j.dst_k = (char*)p.k_hist + (size_t)slot * p.G * row;
        j.dst_v = (char*)p.v_hist + (size_t)slot * p.G * row;
        j.src_bstride = (long long)p.N * row;
        j.dst_bstride = (long long)p.d.history_capacity * p.G * row;
        j.src_gw = p.d.grid_w;
        j.out_gw = p.d.grid_w;
        j.out_n = p.G;
        j.sigma = 1;
    }
    for (int gi = 0; gi < p.n_groups; ++gi) {
        const msf::Group& g = p.groups[gi];
        if (g.scale == 1) continue;
        // and, pooled, into the same slot of every coarser level
        msf::PoolJob& j = jb.j[jb.n++];
        size_t dof = (size_t)(g.pyr_offset + slot * g.pooled) * row;
        j.src_k = (const char*)k_win;
        j.src_v = (const char*)v_win;
        j.dst_k = msf::pyr_k(p) + dof;
        j.dst_v = msf::pyr_v(p) + dof;
        j.src_bstride = (long long)p.N * row;
        j.dst_bstride = (long long)p.pyr_tokens * row;
        j.src_gw = p.d.grid_w;
        j.out_gw = p.d.grid_w / g.scale;
        j.out_n = g.pooled;
        j.sigma = g.scale;
    }
    msf_status st = cuda_status(msf::launch_pool(jb, p.B, p.elem == 2, (cudaStream_t)stream));
    if (st != MSF_OK) return st;
    if (p.hist_count < p.d.history_capacity) {
        ++p.hist_count;
    } else {
        p.hist_oldest = (p.hist_oldest + 1) % p.d.history_capacity;
    }
    return MSF_OK;
}

extern "C" msf_status msf_history_commit(msf_plan_t plan) {
    if (!plan) return MSF_ERR_INVALID_ARG;
    Plan& p = *plan;
    if (!p.bound || !p.fused) return MSF_ERR_STATE;
    // The staged head joins the live frames (slot order: frames stay where
    // they were written). Below capacity the next free slot becomes the spare;
    // at capacity the oldest frame is evicted and its slot becomes the spare.
    if (p.hist_count < p.d.history_capacity) {
        ++p.hist_count;
        p.hist_spare = p.hist_count;
    } else {
        p.hist_spare = p.hist_oldest;
        p.hist_oldest = (p.hist_oldest + 1) % p.ring_slots;
    }
    return MSF_OK;
}

extern "C" msf_status msf_history_get(msf_plan_t plan, msf_history_state* out) {
    if (!plan || !out) return MSF_ERR_INVALID_ARG;
    out->count = plan->hist_count;
    out->oldest = plan->hist_oldest;
    out->spare = plan->fused ? plan->hist_spare : -1;
    out->_pad = 0;
    return MSF_OK;
}

extern "C" msf_status msf_history_set(msf_plan_t plan, const msf_history_state* st) {
    if (!plan || !st) return MSF_ERR_INVALID_ARG;
    Plan& p = *plan;
    if (!p.bound) return MSF_ERR_STATE;
    const int cap = p.d.history_capacity;
    if (st->count < 0 || st->count > cap) return MSF_ERR_INVALID_ARG;
    if (st->oldest < 0 || st->oldest >= (p.fused ? cap + 1 : (cap > 0 ? cap : 1)))
        return MSF_ERR_INVALID_ARG;
    if (st->count < cap && st->oldest != 0) return MSF_ERR_INVALID_ARG;
    if (p.fused) {
        // below capacity the live frames are slots [0, count) and the spare
        // is slot count; at capacity the spare is the slot just before the
        // oldest frame (the one evicted last)
        const int want = st->count < cap ? st->count : (st->oldest + cap) % (cap + 1);
        if (st->spare != want) return MSF_ERR_INVALID_ARG;
        p.hist_spare = st->spare;
    }
    p.hist_count = st->count;
    p.hist_oldest = st->oldest;
    return MSF_OK;
}

static msf_status check_attn_args(const Plan& p, const void* q, const void* k_win,
                                  const void* v_win, void* out) {
    if (!q || !k_win || !v_win || !out) return MSF_ERR_INVALID_ARG;
    if (!p.bound) return MSF_ERR_STATE;
    if (!aligned16(q) || !aligned16(k_win) || !aligned16(v_win) || !aligned16(out))
        return MSF_ERR_INVALID_ARG;
    if (out == q || out == k_win || out == v_win) return MSF_ERR_INVALID_ARG;
    return MSF_OK;
}

extern "C" msf_status msf_mssa_forward_simt(msf_plan_t plan, const void* q, const void* k_win,
                                            const void* v_win, void* out, void* stream) {
    if (!plan) return MSF_ERR_INVALID_ARG;
    const Plan& p = *plan;
    msf_status st = check_attn_args(p, q, k_win, v_win, out);
    if (st != MSF_OK) return st;
    msf::AttnArgs a;
    build_attn_args(p, q, k_win, v_win, out, a);
    return cuda_status(msf::launch_attn_simt(a, p.elem == 2, (cudaStream_t)stream));
}

extern "C" msf_status msf_mssa_forward_lse(msf_plan_t plan, const void* q, const void* k_win,
                                           const void* v_win, void* out, float* lse,
                                           void* stream) {
    if (!plan) return MSF_ERR_INVALID_ARG;
    Plan& p = *plan;
    msf_status st = check_attn_args(p, q, k_win, v_win, out);
    if (st != MSF_OK) return st;
    if (lse && !aligned16(lse)) return MSF_ERR_INVALID_ARG;
    msf::AttnArgs a;
    build_attn_args(p, q, k_win, v_win, out, a);
    a.lse = lse;
    if (p.elem == 2) return msf::launch_attn_tc(plan, a, (cudaStream_t)stream);
    return cuda_status(msf::launch_attn_simt(a, false, (cudaStream_t)stream));
}

extern "C" msf_status msf_mssa_forward(msf_plan_t plan, const void* q, const void* k_win,
                                       const void* v_win, void* out, void* stream) {
    if (!plan) return MSF_ERR_INVALID_ARG;
    Plan& p = *plan;
    msf_status st = check_attn_args(p, q, k_win, v_win, out);
    if (st != MSF_OK) return st;
    msf::AttnArgs a;
    build_attn_args(p, q, k_win, v_win, out, a);
    if (p.elem == 2) return msf::launch_attn_tc(plan, a, (cudaStream_t)stream);
    return cuda_status(msf::launch_attn_simt(a, false, (cudaStream_t)stream));
}

extern "C" msf_status msf_mssa_forward_resample(msf_plan_t plan, const void* q, const void* k_win,
                                                const void* v_win, void* out, int32_t flags, void* stream) {
    if (!plan) return MSF_ERR_INVALID_ARG;
    Plan& p = *plan;
    msf_status st = check_attn_args(p, q, k_win, v_win, out);
    if (st != MSF_OK) return st;
    if (flags != MSF_RESAMPLE_FULL && flags != MSF_RESAMPLE_WINDOW_ONLY) return MSF_ERR_INVALID_ARG;
    const bool with_hist = flags == MSF_RESAMPLE_FULL;
    if (count_window_jobs(p, with_hist) > msf::kMaxPoolJobs) return MSF_ERR_UNSUPPORTED;
    msf::PoolBatch jb;
    memset(&jb, 0, sizeof(jb));
    jb.row_vecs = (int)(row_bytes(p) / 16);
    jb.mode = p.d.resample;
    add_window_jobs(p, k_win, v_win, with_hist, jb);
    msf::AttnArgs a;
    build_attn_args(p, q, k_win, v_win, out, a);
    cudaStream_t s = (cudaStream_t)stream;
    if (p.elem == 2) return msf::launch_attn_tc(plan, a, s, &jb);
    if (jb.n > 0) {
        st = cuda_status(msf::launch_pool(jb, p.B, false, s));
        if (st != MSF_OK) return st;
    }
    return cuda_status(msf::launch_attn_simt(a, false, s));
}

// Gradient rows of group gi: the context rows that come from the window,
// each run with the window token its rows map back to (Eq. 4's Subsample
// undone by the adjoint). Mirrors the context layout of build_attn_args.
static void build_bwd_group(const Plan& p, int gi, const void* k_win, const void* v_win,
                            msf::BwdGroup& bg, int& crow) {
    memset(&bg, 0, sizeof(bg));
    const msf::Group& g = p.groups[gi];
    const size_t row = row_bytes(p);
    bg.q_begin = g.q_begin;
    bg.q_end = g.q_end;
    auto add = [&](const char* k, const char* v, long long bs, int row0, int len, int rows_total,
                   int map_id, int sigma, int dst0, int src_gw, int out_gw) {
        if (len <= 0) return;
        msf::GradSeg& s = bg.gseg[bg.n_gseg++];
        s.k = k;
        s.v = v;
        s.bstride = bs;
        s.row0 = row0;
        s.len = len;
        s.rows_total = rows_total;
        s.map_id = map_id;
        s.sigma = sigma;
        s.dst0 = dst0;
        s.src_gw = src_gw;
        s.out_gw = out_gw;
        s.crow0 = crow;
        crow += len;
    };
    const long long win_bs = (long long)p.N * row;
    const long long pyr_bs = (long long)p.pyr_tokens * row;
    const long long ring_bs = (long long)p.ring_slots * p.G * row;
    if (g.scale == 1) {
        if (p.fused) {
            // the head is read from the ring's spare slot
            add((const char*)p.k_hist, (const char*)p.v_hist, ring_bs, p.hist_spare * p.G, p.G,
                p.ring_slots * p.G, msf::kMapHist, 1, 0, 0, 0);
            add((const char*)k_win, (const char*)v_win, win_bs, p.st_n[0], p.N - p.st_n[0], p.N,
                msf::kMapWin, 1, p.st_n[0], 0, 0);
        } else {
            add((const char*)k_win, (const char*)v_win, win_bs, 0, p.N, p.N, msf::kMapWin, 1, 0, 0,
                0);
        }
        return;
    }
    const int out_gw = p.d.grid_w / g.scale;
    for (int l = 0; l < g.n_finer; ++l) {
        int slot;  // pyramid slot of pooled state l (same rule as the resample jobs)
        if (!p.fused)
            slot = p.hist_count + l;
        else
            slot = l == 0 ? g.n_finer - 1 + p.hist_spare : l - 1;
        add(msf::pyr_k(p), msf::pyr_v(p), pyr_bs, g.pyr_offset + slot * g.pooled, g.pooled,
            p.pyr_tokens, msf::kMapPyr, g.scale / p.d.scales[l], p.st_off[l], p.st_gw[l], out_gw);
    }
    add((const char*)k_win, (const char*)v_win, win_bs, g.q_begin, p.N - g.q_begin, p.N,
        msf::kMapWin, 1, g.q_begin, 0, 0);
}

static msf_status mssa_backward(msf_plan_t plan, const void* q, const void* k_win,
                                const void* v_win, const void* out, const void* dout,
                                const float* lse, void* dq, void* dk_win, void* dv_win,
                                void* bwd_ws, size_t bwd_ws_bytes, void* stream, bool tc) {
    if (!plan) return MSF_ERR_INVALID_ARG;
    Plan& p = *plan;
    if (!q || !k_win || !v_win || !out || !dout || !lse || !dq || !dk_win || !dv_win || !bwd_ws)
        return MSF_ERR_INVALID_ARG;
    if (!p.bound) return MSF_ERR_STATE;
    const void* in[] = {q, k_win, v_win, out, dout, lse, dq, dk_win, dv_win, bwd_ws};
    for (const void* x : in)
        if (!aligned16(x)) return MSF_ERR_INVALID_ARG;
    const void* outs[] = {dq, dk_win, dv_win};
    const void* ins[] = {q, k_win, v_win, out, dout, lse};
    for (const void* o : outs)
        for (const void* i : ins)
            if (o == i) return MSF_ERR_INVALID_ARG;
    if (dq == dk_win || dq == dv_win || dk_win == dv_win) return MSF_ERR_INVALID_ARG;
    if (bwd_ws_bytes < msf::bwd_workspace_bytes(p)) return MSF_ERR_WORKSPACE;
    cudaStream_t s = (cudaStream_t)stream;
    const bool bf16 = p.elem == 2;
    msf::BwdCommon c;
    memset(&c, 0, sizeof(c));
    c.q = (const char*)q;
    c.dout = (const char*)dout;
    c.out = (const char*)out;
    c.lse = lse;
    c.delta = (float*)bwd_ws;
    c.dk_ctx = (float*)((char*)bwd_ws + msf::bwd_delta_bytes(p));
    c.dv_ctx = (float*)((char*)bwd_ws + msf::bwd_delta_bytes(p) + msf::bwd_ctx_bytes(p));
    c.R = msf::bwd_ctx_rows(p);
    c.bstride = (long long)p.N * row_bytes(p);
    c.H = p.H;
    c.D = p.D;
    c.B = p.B;
    c.N = p.N;
    c.scale = p.scale;
    c.scale_log2 = p.scale * 1.4426950408889634f;
    cudaError_t e = msf::launch_bwd_delta(c, bf16, s);
    if (e != cudaSuccess) return cuda_status(e);
    msf::AttnArgs a;
    build_attn_args(p, q, k_win, v_win, (void*)out, a);
    msf::BwdGroup bg[MSF_MAX_GROUPS];
    int crow = 0;
    for (int gi = 0; gi < p.n_groups; ++gi) build_bwd_group(p, gi, k_win, v_win, bg[gi], crow);
    if (crow != c.R) return MSF_ERR_STATE;
    // The adjoint of Subsample per window state: the runs of every group
    // that hold the state, as is (sigma 1) or pooled.
    msf::GatherArgs ga;
    memset(&ga, 0, sizeof(ga));
    ga.T = p.T;
    ga.mode = p.d.resample;
    for (int l = 0; l < p.T; ++l) ga.st_off[l] = p.st_off[l];
    ga.st_off[p.T] = p.N;
    for (int gi = 0; gi < p.n_groups; ++gi)
        for (int si = 0; si < bg[gi].n_gseg; ++si) {
            const msf::GradSeg& gs = bg[gi].gseg[si];
            for (int l = 0; l < p.T; ++l) {
                const int lo = p.st_off[l], hi = p.st_off[l] + p.st_n[l];
                const bool holds = gs.sigma == 1 ? (gs.dst0 <= lo && hi <= gs.dst0 + gs.len)
                                                 : gs.dst0 == lo;
                if (!holds) continue;
                if (ga.n_ent[l] == MSF_MAX_GROUPS) return MSF_ERR_STATE;
                msf::GatherEntry& en = ga.e[l][ga.n_ent[l]++];
                en.crow0 = gs.crow0;
                en.dst0 = gs.dst0;
                en.sigma = gs.sigma;
                en.src_gw = gs.src_gw;
                en.out_gw = gs.out_gw;
            }
        }
    if (tc && bf16) {
        msf::BwdTcInput in;
        in.a = &a;
        in.g = bg;
        in.q = q;
        in.dout = dout;
        in.lse = lse;
        in.delta = c.delta;
        in.dq = dq;
        in.dk_ctx = c.dk_ctx;
        in.dv_ctx = c.dv_ctx;
        in.R = c.R;
        msf_status st = msf::launch_bwd_tc(plan, in, s);
        if (st != MSF_OK) return st;
    } else {
        e = msf::launch_bwd_dq_simt(c, a, dq, bf16, s);
        if (e != cudaSuccess) return cuda_status(e);
        for (int gi = 0; gi < p.n_groups; ++gi) {
            e = msf::launch_bwd_dkdv_simt(c, bg[gi], bf16, s);
            if (e != cudaSuccess) return cuda_status(e);
        }
    }
    return cuda_status(msf::launch_bwd_gather(c, ga, dk_win, dv_win, bf16, s));
}

extern "C" msf_status msf_mssa_backward(msf_plan_t plan, const void* q, const void* k_win,
                                        const void* v_win, const void* out, const void* dout,
                                        const float* lse, void* dq, void* dk_win, void* dv_win,
                                        void* bwd_ws, size_t bwd_ws_bytes, void* stream) {
    return mssa_backward(plan, q, k_win, v_win, out, dout, lse, dq, dk_win, dv_win, bwd_ws,
                         bwd_ws_bytes, stream, true);
}

extern "C" msf_status msf_mssa_backward_simt(msf_plan_t plan, const void* q, const void* k_win,
                                             const void* v_win, const void* out, const void* dout,
                                             const float* lse, void* dq, void* dk_win,
                                             void* dv_win, void* bwd_ws, size_t bwd_ws_bytes,
                                             void* stream) {
    return mssa_backward(plan, q, k_win, v_win, out, dout, lse, dq, dk_win, dv_win, bwd_ws,
                         bwd_ws_bytes, stream, false);
}

static msf::MspShape msp_shape(const Plan& p) {
    msf::MspShape sh;
    memset(&sh, 0, sizeof(sh));
    sh.T = p.T;
    sh.C = p.d.latent_channels;
    sh.patch = p.d.patch;
    sh.Hl = p.gh * p.d.patch;  // F latent frames stacked: [C, F, Hl, Wl] = [C, F*Hl, Wl]
    sh.Wl = p.d.grid_w * p.d.patch;
    for (int l = 0; l < p.T; ++l) sh.scales[l] = p.d.scales[l];
    return sh;
}

extern "C" msf_status msf_patchify(msf_plan_t plan, const void* latent, const void* const* w_tier,
                                   void* tokens, void* stream) {
    if (!plan || !latent || !tokens) return MSF_ERR_INVALID_ARG;
    const Plan& p = *plan;
    if (p.d.latent_channels <= 0 || p.d.patch <= 0) return MSF_ERR_UNSUPPORTED;
    if (!aligned16(latent) || !aligned16(tokens)) return MSF_ERR_INVALID_ARG;
    const msf::MspShape sh = msp_shape(p);
    cudaStream_t s = (cudaStream_t)stream;
    const bool bf16 = p.elem == 2;
    if (!w_tier) return cuda_status(msf::launch_patchify_raw(latent, tokens, sh, p.B, bf16, s));
    if (p.d.embed_dim <= 0) return MSF_ERR_UNSUPPORTED;
    if (!p.bound) return MSF_ERR_STATE;  // the raw tokens go through the workspace
    for (int l = 0; l < p.T; ++l)
        if (!w_tier[l] || !aligned16(w_tier[l])) return MSF_ERR_INVALID_ARG;
    const long long per = (long long)sh.C * sh.Hl * sh.Wl;
    const int E = p.d.embed_dim;
    if (bf16) {
        // Fused gather + embedding: one problem per run of consecutive states
        // that share a tier (same scale, same weight), all runs in one launch.
        msf::MspEmbedRun runs[MSF_MAX_STATES];
        int n_runs = 0;
        for (int l0 = 0; l0 < p.T;) {
            int l1 = l0 + 1;
            while (l1 < p.T && p.d.scales[l1] == p.d.scales[l0] && w_tier[l1] == w_tier[l0]) ++l1;
            msf::MspEmbedRun& r = runs[n_runs++];
            r.w = w_tier[l0];
            r.P = p.d.patch * p.d.scales[l0];
            r.K = sh.C * r.P * r.P;
            r.l0 = l0;
            r.n_l = p.st_n[l0];
            r.M = p.st_off[l1 - 1] + p.st_n[l1 - 1] - p.st_off[l0];
            r.gw = sh.Wl / r.P;
            r.tok_off = p.st_off[l0];
            l0 = l1;
        }
        bool fused = true;
        for (int r0 = 0; r0 < n_runs && fused; r0 += msf::kMaxGemmProblems) {
            const int n = n_runs - r0 < msf::kMaxGemmProblems ? n_runs - r0 : msf::kMaxGemmProblems;
            fused = msf::msp_embed_supported(runs + r0, n, E);
        }
        if (fused) {
            for (int r0 = 0; r0 < n_runs; r0 += msf::kMaxGemmProblems) {
                const int n = n_runs - r0 < msf::kMaxGemmProblems ? n_runs - r0 : msf::kMaxGemmProblems;
                cudaError_t e = msf::launch_msp_embed(runs + r0, n, sh, E, latent, tokens, (long long)p.N * E,
                                                      p.B, msf::status_word(p), s);
                if (e != cudaSuccess) return cuda_status(e);
            }
            return MSF_OK;
        }
    }
    char* raw = msf::msp_scratch(p);
    cudaError_t e = msf::launch_patchify_raw(latent, raw, sh, p.B, bf16, s);
    if (e != cudaSuccess) return cuda_status(e);
    if (bf16) {
        // One tensor-core GEMM problem per run of consecutive states that
        // share a tier (same scale, same weight): their raw blocks and output
        // rows are contiguous. All runs go out in one grouped launch.
        msf::GemmTcArgs runs[MSF_MAX_STATES];
        int n_runs = 0;
        bool all_tc = true;
        for (int l0 = 0; l0 < p.T && all_tc;) {
            int l1 = l0 + 1;
            while (l1 < p.T && p.d.scales[l1] == p.d.scales[l0] && w_tier[l1] == w_tier[l0]) ++l1;
            const int P = p.d.patch * p.d.scales[l0];
            msf::GemmTcArgs& g = runs[n_runs++];
            g.K = sh.C * P * P;
            g.A = raw + (size_t)l0 * per * p.elem;
            g.B = w_tier[l0];
            g.C = (char*)tokens + (size_t)p.st_off[l0] * E * p.elem;
            g.M = p.st_off[l1 - 1] + p.st_n[l1 - 1] - p.st_off[l0];
            g.N = E;
            g.lda = g.K;
            g.ldb = g.K;
            g.ldc = E;
            g.a_bstride = (long long)p.T * per;
            g.c_bstride = (long long)p.N * E;
            g.status = msf::status_word(p);
            all_tc = msf::gemm_tc_supported(g);
            l0 = l1;
        }
        if (all_tc) {
            for (int r0 = 0; r0 < n_runs; r0 += msf::kMaxGemmProblems) {
                const int n = n_runs - r0 < msf::kMaxGemmProblems ? n_runs - r0 : msf::kMaxGemmProblems;
                e = msf::launch_gemm_tc_grouped(runs + r0, n, p.B, s);
                if (e != cudaSuccess) return cuda_status(e);
            }
            return MSF_OK;
        }
    }
    for (int l = 0; l < p.T; ++l) {
        const int P = p.d.patch * p.d.scales[l];
        const int F = sh.C * P * P;
        msf::GemmArgs g;
        g.A = raw + (size_t)l * per * p.elem;
        g.B = w_tier[l];
        g.C = (char*)tokens + (size_t)p.st_off[l] * E * p.elem;
        g.M = p.st_n[l];
        g.N = E;
        g.K = F;
        g.lda = F;
        g.ldb = F;
        g.ldc = E;
        g.a_bstride = (long long)p.T * per;
        g.c_bstride = (long long)p.N * E;
        e = msf::launch_gemm_nt_simt(g, p.B, bf16, s);
        if (e != cudaSuccess) return cuda_status(e);
    }
    return MSF_OK;
}

extern "C" msf_status msf_patchify_resample(msf_plan_t plan, const void* latent, const void* const* w_tier,
                                            void* tokens, const void* k_win, const void* v_win, int32_t flags,
                                            void* stream) {
    if (!plan || !latent || !tokens || !w_tier || !k_win || !v_win) return MSF_ERR_INVALID_ARG;
    const Plan& p = *plan;
    if (p.d.latent_channels <= 0 || p.d.patch <= 0 || p.d.embed_dim <= 0 || p.elem != 2)
        return MSF_ERR_UNSUPPORTED;
    if (!p.bound) return MSF_ERR_STATE;
    if (!aligned16(latent) || !aligned16(tokens) || !aligned16(k_win) || !aligned16(v_win))
        return MSF_ERR_INVALID_ARG;
    for (int l = 0; l < p.T; ++l)
        if (!w_tier[l] || !aligned16(w_tier[l])) return MSF_ERR_INVALID_ARG;
    if (flags != MSF_RESAMPLE_FULL && flags != MSF_RESAMPLE_WINDOW_ONLY) return MSF_ERR_INVALID_ARG;
    const bool with_hist = flags == MSF_RESAMPLE_FULL;
    if (count_window_jobs(p, with_hist) > msf::kMaxPoolJobs) return MSF_ERR_UNSUPPORTED;
    const msf::MspShape sh = msp_shape(p);
    const int E = p.d.embed_dim;
    msf::MspEmbedRun runs[MSF_MAX_STATES];
    int n_runs = 0, tiles = 0;
    for (int l0 = 0; l0 < p.T;) {
        int l1 = l0 + 1;
        while (l1 < p.T && p.d.scales[l1] == p.d.scales[l0] && w_tier[l1] == w_tier[l0]) ++l1;
        msf::MspEmbedRun& r = runs[n_runs++];
        r.w = w_tier[l0];
        r.P = p.d.patch * p.d.scales[l0];
        r.K = sh.C * r.P * r.P;
        r.l0 = l0;
        r.n_l = p.st_n[l0];
        r.M = p.st_off[l1 - 1] + p.st_n[l1 - 1] - p.st_off[l0];
        r.gw = sh.Wl / r.P;
        r.tok_off = p.st_off[l0];
        if (n_runs <= msf::kMaxGemmProblems) tiles += ((r.M + 127) / 128) * ((E + 255) / 256);
        l0 = l1;
    }
    // Runs with the widest patch vectors (most K chunks, the longest tiles)
    // first in the grid, so that the block scheduler starts them first.
    for (int i = 1; i < n_runs; ++i)
        for (int k = i; k > 0 && runs[k].K > runs[k - 1].K; --k) {
            const msf::MspEmbedRun t = runs[k];
            runs[k] = runs[k - 1];
            runs[k - 1] = t;
        }
    for (int r0 = 0; r0 < n_runs; r0 += msf::kMaxGemmProblems) {
        const int n = n_runs - r0 < msf::kMaxGemmProblems ? n_runs - r0 : msf::kMaxGemmProblems;
        if (!msf::msp_embed_supported(runs + r0, n, E)) return MSF_ERR_UNSUPPORTED;
    }
    msf::PoolBatch jb;
    memset(&jb, 0, sizeof(jb));
    jb.row_vecs = (int)(row_bytes(p) / 16);
    jb.mode = p.d.resample;
    add_window_jobs(p, k_win, v_win, with_hist, jb);
    // Pool CTAs per stream: one 256-thread block per 256 tasks, as the pool
    // kernel launches them, after the embedding tiles in the grid (the
    // longest tiles, those of the widest patch vectors, first).
    int max_n = 0;
    for (int k = 0; k < jb.n; ++k) max_n = jb.j[k].out_n > max_n ? jb.j[k].out_n : max_n;
    long long pool_ctas = ((long long)jb.n * max_n * (jb.row_vecs / 2) + 255) / 256;
    if (pool_ctas < 1) pool_ctas = 1;
    (void)tiles;
    cudaError_t e = cudaSuccess;
    cudaStream_t s = (cudaStream_t)stream;
    for (int r0 = 0; r0 < n_runs; r0 += msf::kMaxGemmProblems) {
        const int n = n_runs - r0 < msf::kMaxGemmProblems ? n_runs - r0 : msf::kMaxGemmProblems;
        e = msf::launch_msp_embed(runs + r0, n, sh, E, latent, tokens, (long long)p.N * E, p.B, msf::status_word(p), s,
                                  r0 == 0 && jb.n > 0 ? &jb : nullptr, (int)pool_ctas);
        if (e != cudaSuccess) return cuda_status(e);
    }
    return MSF_OK;
}

extern "C" msf_status msf_unpatchify(msf_plan_t plan, int32_t position, const void* tokens,
                                     const void* w_out, void* latent_out, void* stream) {
    if (!plan || !tokens || !latent_out) return MSF_ERR_INVALID_ARG;
    const Plan& p = *plan;
    if (p.d.latent_channels <= 0 || p.d.patch <= 0) return MSF_ERR_UNSUPPORTED;
    if (position < 0 || position >= p.T) return MSF_ERR_INVALID_ARG;
    if (!aligned16(tokens) || !aligned16(latent_out)) return MSF_ERR_INVALID_ARG;
    const msf::MspShape sh = msp_shape(p);
    cudaStream_t s = (cudaStream_t)stream;
    const bool bf16 = p.elem == 2;
    const long long per = (long long)sh.C * sh.Hl * sh.Wl;
    if (!w_out)
        return cuda_status(msf::launch_unpatchify_raw(tokens, latent_out, sh, position,
                                                      (long long)p.T * per, (int)(position * per),
                                                      p.B, bf16, s));
    if (p.d.embed_dim <= 0) return MSF_ERR_UNSUPPORTED;
    if (!p.bound) return MSF_ERR_STATE;
    if (!aligned16(w_out)) return MSF_ERR_INVALID_ARG;
    const int P = p.d.patch * p.d.scales[position];
    const int F = sh.C * P * P;
    const int E = p.d.embed_dim;
    char* raw = msf::msp_scratch(p);
    if (bf16 && msf::msp_deembed_supported(p.st_n[position], F, E)) {
        return cuda_status(msf::launch_msp_deembed(tokens, (long long)p.N * E, p.N, p.st_off[position], w_out,
                                                   p.st_n[position], F, E, sh, P, latent_out, p.B,
                                                   msf::status_word(p), s));
    }
    if (bf16) {
        msf::GemmTcArgs t;
        t.A = (const char*)tokens + (size_t)p.st_off[position] * E * p.elem;
        t.B = w_out;
        t.C = raw;
        t.M = p.st_n[position];
        t.N = F;
        t.K = E;
        t.lda = E;
        t.ldb = E;
        t.ldc = F;
        t.a_bstride = (long long)p.N * E;
        t.c_bstride = per;
        t.status = msf::status_word(p);
        t.C32 = msf::msp_split(p);
        t.max_splits = msf::kMaxDeembedSplits;
        if (msf::gemm_tc_supported(t)) {
            cudaError_t e = msf::launch_gemm_tc(t, p.B, s);
            if (e != cudaSuccess) return cuda_status(e);
            if (t.splits_used > 1)
                return cuda_status(msf::launch_unpatchify_splitk(msf::msp_split(p), t.splits_used,
                                                                 latent_out, sh, position, p.B, s));
            return cuda_status(
                msf::launch_unpatchify_raw(raw, latent_out, sh, position, per, 0, p.B, bf16, s));
        }
    }
    msf::GemmArgs g;
    g.A = (const char*)tokens + (size_t)p.st_off[position] * E * p.elem;
    g.B = w_out;
    g.C = raw;
    g.M = p.st_n[position];
    g.N = F;
    g.K = E;
    g.lda = E;
    g.ldb = E;
    g.ldc = F;
    g.a_bstride = (long long)p.N * E;
    g.c_bstride = per;
    cudaError_t e = msf::launch_gemm_nt_simt(g, p.B, bf16, s);
    if (e != cudaSuccess) return cuda_status(e);
    return cuda_status(msf::launch_unpatchify_raw(raw, latent_out, sh, position, per, 0, p.B, bf16, s));
}

namespace {

bool tier_lora_ok(const void* down, const void* up, int rank) {
    if (!down) return true;
    return up && rank >= 8 && rank <= msf::kTierCodeCols && rank % 8 == 0 && aligned16(down) && aligned16(up);
}

}  // namespace

extern "C" msf_status msf_patchify_tiers(msf_plan_t plan, const void* latent,
                                         const msf_tier_module* const* tiers, void* tokens, void* stream) {
    if (!plan || !latent || !tokens || !tiers) return MSF_ERR_INVALID_ARG;
    const Plan& p = *plan;
    if (p.d.latent_channels <= 0 || p.d.patch <= 0 || p.d.embed_dim <= 0 || p.elem != 2)
        return MSF_ERR_UNSUPPORTED;
    if (!p.bound) return MSF_ERR_STATE;  // the LoRA codes go through the workspace
    if (!aligned16(latent) || !aligned16(tokens)) return MSF_ERR_INVALID_ARG;
    for (int l = 0; l < p.T; ++l) {
        const msf_tier_module* t = tiers[l];
        if (!t || !t->w_embed || !aligned16(t->w_embed)) return MSF_ERR_INVALID_ARG;
        if (!tier_lora_ok(t->embed_down, t->embed_up, t->lora_rank)) return MSF_ERR_INVALID_ARG;
    }
    const msf::MspShape sh = msp_shape(p);
    cudaStream_t s = (cudaStream_t)stream;
    const int E = p.d.embed_dim;
    char* codes = msf::tier_codes(p);
    const long long codes_bstride = (long long)p.N * msf::kTierCodeCols;
    // Runs of consecutive states that share a tier module.
    msf::MspEmbedRun runs[MSF_MAX_STATES], code_runs[MSF_MAX_STATES];
    int n_runs = 0, n_code = 0;
    for (int l0 = 0; l0 < p.T;) {
        int l1 = l0 + 1;
        while (l1 < p.T && p.d.scales[l1] == p.d.scales[l0] && tiers[l1] == tiers[l0]) ++l1;
        const msf_tier_module* t = tiers[l0];
        msf::MspEmbedRun& r = runs[n_runs++];
        r.w = t->w_embed;
        r.P = p.d.patch * p.d.scales[l0];
        r.K = sh.C * r.P * r.P;
        r.l0 = l0;
        r.n_l = p.st_n[l0];
        r.M = p.st_off[l1 - 1] + p.st_n[l1 - 1] - p.st_off[l0];
        r.gw = sh.Wl / r.P;
        r.tok_off = p.st_off[l0];
        if (t->embed_down) {
            // The rank-r codes gamma * x A^T of the run's tokens, by the same
            // fused gather + GEMM kernel with A as its weight (rows past r and
            // columns past 64 are zero), then the embedding with one more K
            // chunk: codes x the up projection.
            msf::MspEmbedRun& c = code_runs[n_code++];
            c = r;
            c.w = t->embed_down;
            c.w_rows = t->lora_rank;
            c.scale = t->lora_scale;
            r.lora_up = t->embed_up;
            r.rank = t->lora_rank;
            r.codes = codes + (size_t)r.tok_off * msf::kTierCodeCols * 2;
            r.codes_bstride = codes_bstride;
        }
        l0 = l1;
    }
    for (int r0 = 0; r0 < n_code; r0 += msf::kMaxGemmProblems) {
        const int n = n_code - r0 < msf::kMaxGemmProblems ? n_code - r0 : msf::kMaxGemmProblems;
        if (!msf::msp_embed_supported(code_runs + r0, n, msf::kTierCodeCols)) return MSF_ERR_UNSUPPORTED;
    }
    for (int r0 = 0; r0 < n_runs; r0 += msf::kMaxGemmProblems) {
        const int n = n_runs - r0 < msf::kMaxGemmProblems ? n_runs - r0 : msf::kMaxGemmProblems;
        if (!msf::msp_embed_supported(runs + r0, n, E)) return MSF_ERR_UNSUPPORTED;
    }
    for (int r0 = 0; r0 < n_code; r0 += msf::kMaxGemmProblems) {
        const int n = n_code - r0 < msf::kMaxGemmProblems ? n_code - r0 : msf::kMaxGemmProblems;
        cudaError_t e = msf::launch_msp_embed(code_runs + r0, n, sh, msf::kTierCodeCols, latent, codes,
                                              codes_bstride, p.B, msf::status_word(p), s);
        if (e != cudaSuccess) return cuda_status(e);
    }
    for (int r0 = 0; r0 < n_runs; r0 += msf::kMaxGemmProblems) {
        const int n = n_runs - r0 < msf::kMaxGemmProblems ? n_runs - r0 : msf::kMaxGemmProblems;
        cudaError_t e = msf::launch_msp_embed(runs + r0, n, sh, E, latent, tokens, (long long)p.N * E, p.B,
                                              msf::status_word(p), s);
        if (e != cudaSuccess) return cuda_status(e);
    }
    return MSF_OK;
}

extern "C" msf_status msf_unpatchify_tier(msf_plan_t plan, int32_t position, const void* tokens,
                                          const void* latent_in, const msf_tier_module* tier,
                                          void* latent_out, void* stream) {
    if (!plan || !tokens || !tier || !latent_out) return MSF_ERR_INVALID_ARG;
    const Plan& p = *plan;
    if (p.d.latent_channels <= 0 || p.d.patch <= 0 || p.d.embed_dim <= 0 || p.elem != 2)
        return MSF_ERR_UNSUPPORTED;
    if (position < 0 || position >= p.T) return MSF_ERR_INVALID_ARG;
    if (!p.bound) return MSF_ERR_STATE;
    if (!aligned16(tokens) || !aligned16(latent_out) || !tier->w_out || !aligned16(tier->w_out))
        return MSF_ERR_INVALID_ARG;
    if (!tier_lora_ok(tier->out_down, tier->out_up, tier->lora_rank)) return MSF_ERR_INVALID_ARG;
    if (tier->residual && (!latent_in || !aligned16(latent_in) || !aligned16(tier->residual)))
        return MSF_ERR_INVALID_ARG;
    const msf::MspShape sh = msp_shape(p);
    cudaStream_t s = (cudaStream_t)stream;
    const int P = p.d.patch * p.d.scales[position];
    const int F = sh.C * P * P;
    const int E = p.d.embed_dim;
    const int M = p.st_n[position];
    const long long per = (long long)sh.C * sh.Hl * sh.Wl;
    if (!msf::msp_deembed_supported(M, F, E)) return MSF_ERR_UNSUPPORTED;
    char* codes = msf::tier_codes(p);
    msf::DeembedTier extra;
    if (tier->out_down) {
        // codes = gamma * h A^T for the state's tokens (columns past r zero),
        // by the de-embedding's cluster split-K kernel with a row output
        cudaError_t e = msf::launch_msp_rows_splitk(
            tokens, (long long)p.N * E, p.N, p.st_off[position], tier->out_down, tier->lora_rank, M, E,
            codes + (size_t)p.st_off[position] * msf::kTierCodeCols * 2, (long long)p.N * msf::kTierCodeCols,
            msf::kTierCodeCols, tier->lora_scale, p.B, msf::status_word(p), s);
        if (e != cudaSuccess) return cuda_status(e);
        extra.codes = codes;
        extra.codes_bstride = (long long)p.N * msf::kTierCodeCols;
        extra.up = tier->out_up;
        extra.rank = tier->lora_rank;
    }
    if (tier->residual) {
        // the state's raw patch vectors (its block of the raw layout) feed the residual
        char* raw = msf::msp_scratch(p);
        cudaError_t e = msf::launch_patchify_raw(latent_in, raw, sh, p.B, true, s, position, 1);
        if (e != cudaSuccess) return cuda_status(e);
        extra.xraw = raw + (size_t)position * per * 2;
        extra.xraw_bstride = (long long)p.T * per;
        extra.residual = tier->residual;
    }
    return cuda_status(msf::launch_msp_deembed(tokens, (long long)p.N * E, p.N, p.st_off[position], tier->w_out,
                                               M, F, E, sh, P, latent_out, p.B, msf::status_word(p), s,
                                               &extra));
}

namespace {
// Waits on a barrier that nothing arrives at; the bounded wait must give up.
__global__ void wait_timeout_selftest_kernel(unsigned int* status, long long limit) {
    __shared__ uint64_t bar;
    __shared__ int abort_flag;
    if (threadIdx.x == 0) {
        abort_flag = 0;
        msf::ptx::mbar_init(&bar, 1);
        msf::ptx::fence_mbar_init();
    }
    __syncthreads();
    volatile int* abort_p = &abort_flag;
    const bool ok = msf::ptx::mbar_wait_bounded(&bar, 0, abort_p, limit);
    if (!__all_sync(0xffffffffu, ok) && threadIdx.x == 0) atomicOr(status, msf::kDevTimeout);
}
}  // namespace

namespace msf {
cudaError_t launch_wait_timeout_selftest(unsigned int* status, long long limit_cycles, cudaStream_t st) {
    note_launch();
    wait_timeout_selftest_kernel<<<1, 32, 0, st>>>(status, limit_cycles);
    return cudaGetLastError();
}
}  // namespace msf

extern "C" msf_status msf_selftest_wait_timeout(msf_plan_t plan, int64_t limit_cycles, void* stream) {
    if (!plan || limit_cycles < 1 || limit_cycles > (int64_t(1) << 31)) return MSF_ERR_INVALID_ARG;
    const Plan& p = *plan;
    if (!p.bound) return MSF_ERR_STATE;
    return cuda_status(msf::launch_wait_timeout_selftest(msf::status_word(p), (long long)limit_cycles,
                                                         (cudaStream_t)stream));
}

extern "C" msf_status msf_plan_device_status(msf_plan_t plan, void* stream) {
    if (!plan) return MSF_ERR_INVALID_ARG;
    const Plan& p = *plan;
    if (!p.bound) return MSF_ERR_STATE;
    cudaStream_t s = (cudaStream_t)stream;
    unsigned int word = 0;
    cudaError_t e = cudaStreamSynchronize(s);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(&word, msf::status_word(p), sizeof(word), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaMemsetAsync(msf::status_word(p), 0, sizeof(word), s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    // A launch that gave up may have left merge counters counted: the next
    // launch's "last piece" test and its wait for the written partials would
    // then fire early or never. Zero them before anything else runs.
    if (e == cudaSuccess && word && msf::attn_counter_bytes(p) > 0) {
        e = cudaMemsetAsync(msf::attn_counters(p), 0, msf::attn_counter_bytes(p), s);
        if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    }
    if (e != cudaSuccess) return cuda_status(e);
    return word ? MSF_ERR_TIMEOUT : MSF_OK;
}
