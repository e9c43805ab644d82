/*
 * msf.h - C ABI of the Ms. Forcing multi-scale window pass on one GB300.
 *
 * The library computes, for one rolling denoising window (Sec. 3.1, Eq. 2):
 *   - Multi-Scale Patchification (MSP, Sec. 4.1, Eq. 3): latent states are
 *     cut into patches of size p_l = s_l * p, coarser for noisier positions;
 *   - the per-scale key/value pyramid that Eq. 4's Subsample() needs;
 *   - Multi-Scale Self-Attention (MSSA, Sec. 4.1, Eq. 4): queries of scale g
 *     attend to the full-resolution sink, then to every history frame and
 *     every window state, each subsampled by max(1, g / s_b);
 *   - the history-cache update after a pass (Algorithm 1, KV update with the
 *     emitted head state).
 *
 * Conventions shared by every call:
 *   - Every call returns msf_status; MSF_OK is 0. Argument and state errors
 *     are reported synchronously, before anything is launched.
 *   - The library never allocates device memory. The caller owns every
 *     device buffer, including the workspace whose size msf_plan_query
 *     reports. The library owns only the opaque host-side plan.
 *   - Device pointers must be 16-byte aligned. Tensors are contiguous,
 *     row-major, with the last index fastest.
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *     stream). Kernels run asynchronously on it; outputs are valid once the
 *     stream has reached the call.
 *   - Element type is the plan's dtype (bf16 or fp32) for every tensor.
 *   - Notation: B streams, T window states, fine token grid Gh x Gw
 *     (G = Gh*Gw tokens per fine frame), H heads, D head_dim, Ns sink tokens,
 *     N = sum_l G / s_l^2 window tokens (Eq. 3), E = embedding width.
 */
#ifndef MSF_H
#define MSF_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum msf_status {
    MSF_OK = 0,
    MSF_ERR_INVALID_ARG = 1,  /* null/misaligned pointer, bad size, bad index */
    MSF_ERR_UNSUPPORTED = 2,  /* a schedule or shape outside what is built */
    MSF_ERR_CUDA = 3,         /* a CUDA runtime call failed; see msf_last_cuda_error */
    MSF_ERR_TIMEOUT = 4,      /* a device-side wait hit its bound (kernel returned early) */
    MSF_ERR_STATE = 5,        /* plan not bound, or history operation not allowed */
    MSF_ERR_WORKSPACE = 6     /* workspace smaller than msf_plan_query reports */
} msf_status;

typedef enum msf_dtype { MSF_DTYPE_BF16 = 0, MSF_DTYPE_F32 = 1 } msf_dtype;

/* Eq. 4's Subsample(C_b, stride): AVG takes the mean of each stride x stride
 * block (the coarse-token proxy of the MSP probe, Sec. 3.2); STRIDED keeps the
 * block's top-left token (the stride-2 key/value subsampling of the MSSA
 * probe, Sec. 3.2). */
typedef enum msf_resample_mode { MSF_RESAMPLE_AVG = 0, MSF_RESAMPLE_STRIDED = 1 } msf_resample_mode;

/* msf_kv_resample flags. */
#define MSF_RESAMPLE_FULL 0         /* pool history frames and window states */
#define MSF_RESAMPLE_WINDOW_ONLY 1  /* window states only; history pyramid is kept
                                       up to date by msf_history_append */

#define MSF_MAX_STATES 16
#define MSF_MAX_GROUPS 8

/* Static schedule and shapes (Sec. 4.1: p_1 <= ... <= p_T, p_l in {p,2p,4p,...}). */
typedef struct msf_plan_desc {
    int32_t T;                        /* window states, 1..MSF_MAX_STATES */
    int32_t scales[MSF_MAX_STATES];   /* s_l = p_l / p: powers of two, non-decreasing */
    int32_t grid_h, grid_w;           /* fine token grid; divisible by max s_l */
    int32_t heads;                    /* H >= 1 */
    int32_t head_dim;                 /* D: 64 or 128 */
    int32_t sink_tokens;              /* Ns >= 0, never resampled */
    int32_t history_frames;           /* live history frames at bind time */
    int32_t history_capacity;         /* ring capacity (>= history_frames) */
    int32_t batch;                    /* B independent streams */
    int32_t dtype;                    /* msf_dtype */
    int32_t resample;                 /* msf_resample_mode */
    float softmax_scale;              /* 0 -> 1/sqrt(D) */
    int32_t latent_channels;          /* C of the latent (patchify); 0 if unused */
    int32_t patch;                    /* native patch p in latent pixels; 0 if unused */
    int32_t embed_dim;                /* E of the tier projections; 0 = raw tokens only */
    int32_t frames_per_state;         /* F latent frames per window state (a chunk, Sec. 5.1);
                                         0 or 1 = one frame. Patches are spatial: each latent
                                         frame is tokenised and subsampled on its own, a state
                                         holds F grids in frame order, G = F * grid_h * grid_w,
                                         history frames and ring slots hold whole chunks and the
                                         latent of a state is [C, F, Hl, Wl]. grid_h and grid_w
                                         are one latent frame's and must be divisible by max s_l */
    int32_t fused_append;             /* 0: the history update is its own launch
                                         (msf_history_append). 1: it is folded into
                                         msf_kv_resample: the ring has capacity + 1 slots,
                                         every resample copies the head state (position 1)
                                         into the spare slot and pools it there at every
                                         coarser level from the same read, attention reads
                                         the head from that slot, and msf_history_commit
                                         (host only, no launch) makes it a history frame.
                                         Needs s_1 = 1 and capacity >= 1 */
} msf_plan_desc;

typedef struct msf_group_info {
    int32_t scale;        /* g: scale shared by this group's query states */
    int32_t q_begin;      /* first query token (window order) */
    int32_t q_end;        /* one past the last */
    int32_t n_kv;         /* context length Nkv_g with the current history count */
    int32_t n_pyramid;    /* tokens of the resampled part (history@g + finer states) */
    int32_t pyr_offset;   /* token offset of that part in the workspace pyramid, -1 if g==1 */
} msf_group_info;

typedef struct msf_plan_info {
    int32_t T;
    int32_t n_tokens;                 /* N = N_MSP (Eq. 3) */
    int32_t n_tokens_fine;            /* T * G (all-fine window, N_RF of Eq. 3) */
    int32_t fine_tokens;              /* G (tokens of one fine state, all F latent frames) */
    int32_t state_offset[MSF_MAX_STATES];
    int32_t state_tokens[MSF_MAX_STATES];
    int32_t state_grid_h[MSF_MAX_STATES];  /* rows of the state's grid over all F latent
                                              frames: F * grid_h / s_l */
    int32_t state_grid_w[MSF_MAX_STATES];
    int32_t n_groups;
    msf_group_info groups[MSF_MAX_GROUPS];
    int32_t history_count;            /* live frames in the history ring */
    int32_t history_next_slot;        /* slot the next msf_history_append writes (with
                                         fused_append: the spare slot the head is staged in) */
    int32_t pyramid_tokens;           /* tokens per stream in the workspace pyramid */
    int32_t frames_per_state;         /* F (1 when desc.frames_per_state is 0) */
    uint64_t workspace_bytes;         /* device workspace msf_plan_bind needs */
    uint64_t attention_flops;         /* 4*D*H*B*sum_g Nq_g*Nkv_g (current history) */
    uint64_t dense_flops;             /* same window with every s_l = 1 (no MSP, no MSSA) */
    uint64_t resample_bytes;          /* bytes read+written by a full msf_kv_resample */
    uint64_t pyramid_k_offset;        /* byte offset of the K pyramid [B, pyramid_tokens, H, D]
                                         inside the workspace */
    uint64_t pyramid_v_offset;        /* byte offset of the V pyramid */
    uint64_t backward_workspace_bytes; /* scratch msf_mssa_backward needs */
    uint64_t backward_flops;          /* algorithmic FLOPs of msf_mssa_backward: per group
                                         Nq * (6*D*Nkv + 4*D*Nkv_window) * H * B (S, dP and
                                         dQ over the whole context; dK and dV over the rows
                                         that come from the window) */
    uint64_t attention_counter_offset; /* byte offset, inside the workspace, of the merge
                                          counters of the tensor-core attention (one 32-bit
                                          word per 256-row query block; zero between launches) */
    uint64_t attention_counter_bytes;  /* their size (0 for fp32 plans) */
} msf_plan_info;

typedef struct msf_plan* msf_plan_t;

/* Human-readable name of a status code. Never NULL. */
const char* msf_status_string(msf_status s);

/* The last cudaError_t value seen by a call that returned MSF_ERR_CUDA
 * (thread-local; 0 if none). */
int msf_last_cuda_error(void);

/* Validate `desc` and build the static schedule tables (Eq. 3 token counts,
 * Eq. 4 query groups and context layout). Host only; no CUDA call.
 * Errors: INVALID_ARG (null pointers, non-positive sizes), UNSUPPORTED
 * (non-monotone or non-power-of-two scales, grid not divisible by max s_l,
 * head_dim not 64/128, too many groups). On success *out owns a plan that
 * msf_plan_destroy frees. */
msf_status msf_plan_create(const msf_plan_desc* desc, msf_plan_t* out);

/* Free a plan. NULL-safe. Device buffers stay the caller's. */
void msf_plan_destroy(msf_plan_t plan);

/* Fill `info` (host memory) with the plan's tables and sizes. Host only. */
msf_status msf_plan_query(msf_plan_t plan, msf_plan_info* info);

/* Enumerate the context rows of query group `group` in the order the kernels
 * and the oracle use (Eq. 4: sink, history frames in slot order, window
 * states 1..T). Each row is 5 int32: kind (0 sink, 1 history, 2 window),
 * frame (history slot or window position, 0-based), stride (the Subsample
 * stride applied to that frame), row, col (on the pooled grid; for the sink
 * row = sink token, col = 0). With F latent frames per state the rows of
 * latent frame f follow those of frame f-1: row = f * (pooled rows of one
 * frame) + i. With fused_append the same rows come in the kernels' order:
 * sink; for g > 1 the pooled window states 2..n_finer; then ring slots
 * 0..count in slot order (live frames as history rows, the spare slot as
 * window position 0); then the window states the kernel reads from k_win
 * (from position 1 for g = 1, from the group's first state for g > 1). Writes at most `cap_rows` rows to `out` (host
 * memory, may be NULL when cap_rows is 0) and sets *n_rows to the total.
 * Host only. */
msf_status msf_plan_index_map(msf_plan_t plan, int32_t group, int32_t* out, size_t cap_rows,
                              size_t* n_rows);

/* Attach device buffers that persist across passes:
 *   workspace  >= info.workspace_bytes bytes (status word + per-scale pyramid)
 *   k_sink, v_sink [B, Ns, H, D]           (read only, never resampled)
 *   k_hist, v_hist [B, capacity, G, H, D]  history ring, fine scale; the first
 *                                          history_frames slots hold live frames
 *                                          ([B, capacity + 1, G, H, D] with
 *                                          fused_append: one spare slot)
 * Resets the history count to desc.history_frames and zeroes the device status
 * word (a cudaMemsetAsync on the legacy stream, completed before returning).
 * Builds the TMA descriptors for the bound buffers. Errors: INVALID_ARG,
 * WORKSPACE, CUDA. */
msf_status msf_plan_bind(msf_plan_t plan, void* workspace, size_t workspace_bytes,
                         const void* k_sink, const void* v_sink, void* k_hist, void* v_hist);

/* MSP patchify (Sec. 4.1). latent [B, T, C, Hl, Wl] with Hl = patch*Gh,
 * Wl = patch*Gw. Token (i, j) of state l has feature c*P^2 + dy*P + dx =
 * latent[b, l, c, P*i + dy, P*j + dx], P = patch * s_l.
 *   w_tier == NULL: tokens is the raw layout [B, T, C*Hl*Wl]; state l's block
 *                   is [G/s_l^2, C*P^2] (a permutation of its latent).
 *   w_tier != NULL: array of T device pointers, w_tier[l] = the tier's
 *                   patch-embedding weight [E, C*P^2] (the Conv2d weight
 *                   [E, C, P, P] flattened); tokens is [B, N, E] and
 *                   row off_l + i*gw_l + j holds sum_f patch[f] * w[e, f]
 *                   (fp32 accumulation, one rounding to the dtype).
 * Errors: INVALID_ARG, UNSUPPORTED (no latent_channels/patch, or E == 0 with
 * weights), CUDA. */
msf_status msf_patchify(msf_plan_t plan, const void* latent, const void* const* w_tier,
                        void* tokens, void* stream);

/* msf_patchify with tier weights (w_tier != NULL) and msf_kv_resample(k_win,
 * v_win, flags) in one launch, for bf16 plans with an embedding: the tokens,
 * the pyramid and (fused_append) the staged head are exactly those of the
 * two calls. The two read and write disjoint buffers, so the pooling runs on
 * the CTA slots of the wave that the embedding tiles leave free (the
 * embedding holds two CTAs per SM) instead of a second launch. Errors:
 * INVALID_ARG, UNSUPPORTED (fp32 plan, no embedding, a shape the fused
 * embedding kernel does not take), STATE (not bound), CUDA. */
msf_status msf_patchify_resample(msf_plan_t plan, const void* latent, const void* const* w_tier,
                                 void* tokens, const void* k_win, const void* v_win, int32_t flags,
                                 void* stream);

/* MSP unpatchify of window position `position` (0-based): the inverse of
 * msf_patchify for that state.
 *   w_out == NULL: tokens is the raw layout [B, T, C*Hl*Wl] of msf_patchify.
 *   w_out != NULL: tokens is [B, N, E] (for example the attention output viewed
 *                  as [B, N, H*D]); rows of the state are de-embedded by
 *                  w_out [C*P^2, E] (the nn.Linear weight E -> C*P^2) with fp32
 *                  accumulation, then rearranged.
 * latent_out [B, C, Hl, Wl]. Errors: INVALID_ARG, UNSUPPORTED, CUDA. */
msf_status msf_unpatchify(msf_plan_t plan, int32_t position, const void* tokens,
                          const void* w_out, void* latent_out, void* stream);

/* One tier's module (Sec. 4.1: every patch size has its own patch embedding
 * and de-embedding, LoRA adapters and a latent residual branch; the native
 * tier keeps the pretrained path). The paper does not define where the
 * adapters sit or what the residual branch computes; this library takes:
 *   embedding     t = W x + g * U (A x)          (x: the K = C*P^2 raw patch
 *                                                 vector of a token)
 *   de-embedding  y = Wo h + g * Uo (Ao h) + R x  (h: the token after the
 *                                                 backbone, x: the raw patch
 *                                                 vector of the same token of
 *                                                 the state's input latent)
 * with rank-r LoRA factors A/U, Ao/Uo, scale g and the latent residual R.
 * All device pointers, bf16, 16-byte aligned, nn.Linear layouts:
 *   w_embed [E, K], embed_down (A) [r, K], embed_up (U) [E, r],
 *   w_out [K, E], out_down (Ao) [r, E], out_up (Uo) [K, r], residual [K, K].
 * A NULL embed_down / out_down means no adapter on that projection (its up
 * pointer is then ignored), a NULL residual no residual branch. */
typedef struct msf_tier_module {
    const void* w_embed;
    const void* embed_down;
    const void* embed_up;
    const void* w_out;
    const void* out_down;
    const void* out_up;
    const void* residual;
    int32_t lora_rank;   /* r: 8..64, a multiple of 8, when an adapter is given */
    float lora_scale;    /* g */
} msf_tier_module;

/* MSP patchify with tier modules (Sec. 4.1): tokens [B, N, E] of the window
 * latent [B, T, C, Hl, Wl] (as msf_patchify), state l embedded by
 * tiers[l] (an array of T pointers; consecutive states with the same pointer
 * and scale share one run). With an embedding adapter the tokens get
 * g * U (A x): the codes g * A x (fp32 sums, rounded once to bf16) are
 * computed by one launch of the fused gather + GEMM kernel into the
 * workspace, and the embedding launch adds one K chunk (codes x U) to the
 * same fp32 accumulation. bf16 plans with an embedding, bound (the codes
 * live in the workspace). Errors: INVALID_ARG (NULL or misaligned pointers,
 * rank outside 8..64 or not a multiple of 8), UNSUPPORTED (fp32 plan, no
 * embedding, E not a multiple of 64, a patch edge that does not divide 64),
 * STATE (not bound), CUDA. */
msf_status msf_patchify_tiers(msf_plan_t plan, const void* latent, const msf_tier_module* const* tiers,
                              void* tokens, void* stream);

/* De-embedding + unpatchify of window position `position` with its tier's
 * module: tokens [B, N, E] (for example the attention output viewed as
 * [B, N, H*D]), latent_in the window latent [B, T, C, Hl, Wl] the pass
 * started from (read only when tier->residual is set), latent_out
 * [B, C, Hl, Wl]. The adapter's codes g * Ao h come from a tensor-core GEMM
 * into the workspace; the residual's raw patch vectors from the raw
 * patchify kernel into the workspace; the de-embedding kernel then sums the
 * E/64 token chunks, the code chunk and the K/64 residual chunks in one fp32
 * accumulation (split over a cluster) and rounds once. Errors: INVALID_ARG,
 * UNSUPPORTED (fp32 plan, no embedding, K or E not a multiple of 64), STATE,
 * CUDA. */
msf_status msf_unpatchify_tier(msf_plan_t plan, int32_t position, const void* tokens,
                               const void* latent_in, const msf_tier_module* tier, void* latent_out,
                               void* stream);

/* Build the per-scale key/value pyramid in the workspace: for every query
 * group g > 1, the bound history frames (fine, pooled by g) and the window
 * states with s_l < g (pooled by g/s_l), from k_win, v_win [B, N, H, D].
 * Pooling is the plan's Subsample mode; AVG sums in fp32 and rounds once.
 * flags: MSF_RESAMPLE_FULL or MSF_RESAMPLE_WINDOW_ONLY. With fused_append the
 * same launch also stages the head state (tokens [0, G) of k_win/v_win) in
 * the ring's spare slot and its pyramid levels (one read of the head for the
 * copy and the pooling). Errors: INVALID_ARG, STATE (not bound), CUDA. */
msf_status msf_kv_resample(msf_plan_t plan, const void* k_win, const void* v_win, int32_t flags,
                           void* stream);

/* MSSA (Eq. 4): out[b, t, h, :] = sum_j softmax_j(scale * q[b,t,h,:] . K_g[j]) V_g[j]
 * over the context of t's group g (sink, history, window; no mask).
 * q, k_win, v_win, out [B, N, H, D]; out may not alias q/k/v. Reads the
 * pyramid the last msf_kv_resample on the same stream produced. bf16 plans
 * run the tcgen05 tensor-core kernel (bf16 operands, fp32 softmax and
 * accumulation); fp32 plans run an fp32 CUDA-core kernel. Errors:
 * INVALID_ARG, STATE, CUDA. */
msf_status msf_mssa_forward(msf_plan_t plan, const void* q, const void* k_win, const void* v_win,
                            void* out, void* stream);

/* msf_kv_resample(k_win, v_win, flags) and msf_mssa_forward in one launch
 * (Eq. 4: the pyramid is built in the attention kernel's prologue): every CTA
 * first pools its share of the pyramid (and, with fused_append, of the staged
 * head), and a CTA's first tile of what that pooling writes (a pyramid
 * segment; with fused_append also the history ring, which holds the staged
 * head) waits (bounded) until every CTA's share is written; the pyramid, the
 * staged head and out are
 * exactly those of the two calls. fp32 plans run the two calls. flags:
 * MSF_RESAMPLE_FULL or MSF_RESAMPLE_WINDOW_ONLY. Errors: INVALID_ARG,
 * UNSUPPORTED (more pooling jobs than one launch takes), STATE (not bound),
 * CUDA; a wait that gives up raises TIMEOUT in the device status. */
msf_status msf_mssa_forward_resample(msf_plan_t plan, const void* q, const void* k_win,
                                     const void* v_win, void* out, int32_t flags, void* stream);

/* msf_mssa_forward that also writes, for every query row, the natural-log
 * log-sum-exp of its scaled scores over its context,
 *   lse[b, h, t] = ln sum_j exp(scale * q[b,t,h,:] . K_g[j]),
 * fp32 [B, H, N] (16-byte aligned, or NULL for none): the statistic
 * msf_mssa_backward needs to rebuild the softmax. Errors as msf_mssa_forward. */
msf_status msf_mssa_forward_lse(msf_plan_t plan, const void* q, const void* k_win,
                                const void* v_win, void* out, float* lse, void* stream);

/* Gradient of MSSA (Eq. 4) for training through the window: given
 * dout = dL/dout [B, N, H, D] and the forward's out and lse, writes
 *   dq, dk_win, dv_win [B, N, H, D] (plan dtype) = dL/dq, dL/dk_win, dL/dv_win,
 * with the softmax Jacobian per query group and the context gradients sent
 * back through the adjoint of Subsample (AVG: 1/s^2 of a pooled row to each
 * of its s x s source tokens; STRIDED: all of it to the top-left one); a
 * token used by several groups sums their contributions. The sink and the
 * history ring are a detached cache (Algorithm 1 updates it with a
 * stop-gradient) and get no gradient. Needs the pyramid of the forward pass
 * (the last msf_kv_resample on the stream) and the same history state (no
 * commit or append in between). bwd_workspace: >= info.backward_workspace_bytes
 * bytes, 16-byte aligned, overwritten. Output buffers may not alias inputs.
 * bf16 plans run tcgen05 tensor-core kernels (one for dq over each query
 * tile's whole context, one per query group for the window rows' dk/dv);
 * fp32 plans run CUDA-core kernels.
 * Errors: INVALID_ARG, STATE (not bound), WORKSPACE, CUDA. */
msf_status msf_mssa_backward(msf_plan_t plan, const void* q, const void* k_win, const void* v_win,
                             const void* out, const void* dout, const float* lse, void* dq,
                             void* dk_win, void* dv_win, void* bwd_workspace,
                             size_t bwd_workspace_bytes, void* stream);

/* Same gradient always on the fp32 CUDA-core kernels (a cross-check of the
 * tensor-core backward for bf16 plans). */
msf_status msf_mssa_backward_simt(msf_plan_t plan, const void* q, const void* k_win,
                                  const void* v_win, const void* out, const void* dout,
                                  const float* lse, void* dq, void* dk_win, void* dv_win,
                                  void* bwd_workspace, size_t bwd_workspace_bytes, void* stream);

/* Same computation always on the fp32 CUDA-core kernel (a cross-check of the
 * tensor-core kernel for bf16 plans). */
msf_status msf_mssa_forward_simt(msf_plan_t plan, const void* q, const void* k_win,
                                 const void* v_win, void* out, void* stream);

/* History-cache update after a pass (Algorithm 1): copy the head state's fine
 * K/V (window position 0, tokens [0, G)) into the ring slot
 * info.history_next_slot (the next free slot, else the oldest frame), and
 * pool it into that slot of every coarser pyramid level. Advances the
 * host-side count/slot state. Errors: STATE (not bound, capacity 0, s_1 != 1,
 * or a fused_append plan), INVALID_ARG, CUDA. */
msf_status msf_history_append(msf_plan_t plan, const void* k_win, const void* v_win,
                              void* stream);

/* History-cache update of a fused_append plan (Algorithm 1's KV update): the
 * head staged by the last msf_kv_resample becomes the newest history frame.
 * While the ring holds fewer than `capacity` frames the next spare slot is the
 * next free one; once it is full the oldest frame's slot becomes the spare
 * (evicted). Host only: no launch, no device access; call it after the
 * pass's msf_mssa_forward has been enqueued (the next resample overwrites the
 * new spare slot, stream order keeps that after this pass's reads).
 * Errors: INVALID_ARG, STATE (not bound, or not a fused_append plan). */
msf_status msf_history_commit(msf_plan_t plan);

/* Host-side state of the history ring, for checkpointing a streaming
 * rollout. Everything else the rollout needs lives in the caller's buffers:
 * the ring itself (k_hist, v_hist) and, for a plan that keeps its pyramid
 * incrementally, the workspace's pyramid (or rebuild it after a restore with
 * msf_kv_resample(..., MSF_RESAMPLE_FULL)). */
typedef struct msf_history_state {
    int32_t count;   /* live frames in the ring */
    int32_t oldest;  /* slot of the oldest live frame (meaningful once full) */
    int32_t spare;   /* fused_append: the slot the next head is staged in */
    int32_t _pad;
} msf_history_state;

/* Read the ring state. Host only. Errors: INVALID_ARG. */
msf_status msf_history_get(msf_plan_t plan, msf_history_state* out);

/* Restore a ring state read from a plan with the same description (for
 * example after msf_plan_bind of a new plan on restored ring buffers).
 * Checks count <= capacity, slots inside the ring, and the slot rules of the
 * plan's mode (the next free slot or the oldest frame; with fused_append the
 * spare is the free slot below capacity, else not a live one). Host only.
 * Errors: INVALID_ARG (inconsistent state), STATE (not bound). */
msf_status msf_history_set(msf_plan_t plan, const msf_history_state* st);

/* Number of kernels this library has launched in this process (all plans,
 * all devices), for accounting in benchmarks. Host only. */
uint64_t msf_kernel_launches(void);

/* Allocation-free variant of msf_unpatchify with a de-embedding weight. The
 * paper has no counterpart: this exists for callers that cannot allocate
 * device memory (hosts that hand out every device buffer from their own pool
 * and forbid libraries to call cudaMalloc), so it needs no bound workspace.
 * Same arguments and result as msf_unpatchify(plan, position, tokens, w_out,
 * latent_out, stream) with w_out != NULL, for bf16 plans with an embedding.
 * Its scratch (raw tokens and split-K fp32 partial sums) is a fixed 8 MiB
 * device array inside the library, held by every GPU that loads it until the
 * process exits; a problem needs B * C*Hl*Wl * 2 bytes (rounded up to 256)
 * plus 256 bytes of it, and larger ones are rejected with
 * MSF_ERR_UNSUPPORTED. The first call on each device looks up that array's
 * device address (cudaGetSymbolAddress, with that device current) and zeroes
 * its status word (a synchronous cudaMemset); make that first call before any
 * stream capture. It calls no cudaMalloc/cudaFree. Every call shares the one
 * array and overwrites it, so calls that overlap on the GPU (different
 * streams, or threads without ordering) race: serialise them. A device-side
 * timeout of its GEMM is recorded in the array's own status word, which
 * msf_noalloc_device_status reads (msf_plan_device_status does not see it).
 * Errors: INVALID_ARG, UNSUPPORTED (fp32 plan, no embedding, shape too
 * large, or a shape the tensor-core GEMM does not take: E a multiple of 64,
 * C*P^2 a multiple of 8), CUDA. */
msf_status msf_unpatchify_noalloc(msf_plan_t plan, int32_t position, const void* tokens,
                                  const void* w_out, void* latent_out, void* stream);

/* Synchronise `stream`, then read and clear the status word of
 * msf_unpatchify_noalloc's fixed array on the current device. Returns
 * MSF_ERR_TIMEOUT if one of its kernels gave up on a bounded wait since the
 * last read, MSF_OK otherwise. Errors: CUDA. */
msf_status msf_noalloc_device_status(void* stream);

/* Failure-path self test of that status word (no counterpart in the paper):
 * the same bounded-wait kernel as msf_selftest_wait_timeout, aimed at the
 * fixed array's status word of the current device. Errors: INVALID_ARG
 * (limit outside 1 .. 2^31), CUDA. */
msf_status msf_noalloc_selftest_wait_timeout(int64_t limit_cycles, void* stream);

/* Failure-path self test (no counterpart in the paper): launches one block
 * that waits on an mbarrier nothing ever arrives at, with the same bounded
 * wait every tcgen05 kernel of this library uses, for `limit_cycles` SM
 * clock cycles (1 .. 2^31). The wait gives up, the block raises the TIMEOUT
 * bit of the plan's device status word and returns; the next
 * msf_plan_device_status reports MSF_ERR_TIMEOUT and clears the word, and
 * the context stays usable. The plan must be bound. Asynchronous on
 * `stream`. Errors: INVALID_ARG, STATE (not bound), CUDA. */
msf_status msf_selftest_wait_timeout(msf_plan_t plan, int64_t limit_cycles, void* stream);

/* Synchronise `stream`, read and clear the device status word. Returns
 * MSF_ERR_TIMEOUT if a kernel gave up on a bounded wait since the last
 * check, MSF_OK otherwise. After a timeout it also zeroes the attention's
 * merge counters (a launch that gave up can leave them counted), so the next
 * msf_mssa_forward starts from a clean state. */
msf_status msf_plan_device_status(msf_plan_t plan, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* MSF_H */
