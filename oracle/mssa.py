"""Multi-Scale Self-Attention, written out as its definition (Eq. 4) in fp64.

Test infrastructure. The context of each query group is materialised
explicitly (sink, resampled history, resampled window states) and attention
is the naive max-subtracted softmax; numpy's matmul is the only library step.

Tensors: q, k_win, v_win [B, N, H, D] with the window's states concatenated
in position order, each state row-major over its grid; k_sink, v_sink
[B, Ns, H, D]; k_hist, v_hist [B, nh, Gh*Gw, H, D] (fine history frames in
slot order). All inputs are widened to float64 before any arithmetic.

Chunked states (Sec. 5.1, F latent frames per state): a state's tokens are
F frame grids one after the other, and Subsample acts on each latent frame
separately (spatial patches, so spatial resampling); ``frames`` = F, 1 by
default. History frames then hold F*Gh*Gw tokens each.
"""
from __future__ import annotations

import numpy as np

from . import schedule

AVG, STRIDED = 0, 1


def resample(x: np.ndarray, gh: int, gw: int, sigma: int, mode: int = AVG) -> np.ndarray:
    """Subsample(C_b, stride=sigma) of Eq. 4 on a gh x gw token grid.

    x has the grid flattened row-major on axis 1: [B, gh*gw, ...]. AVG takes
    the mean of each sigma x sigma block (the 2x2-mean proxy of the MSP probe,
    Sec. 3.2); STRIDED keeps the block's top-left token (the stride-2 key/value
    subsampling of the MSSA probe, Sec. 3.2). sigma = 1 is the identity.
    """
    x = np.asarray(x, dtype=np.float64)
    if sigma == 1:
        return x.copy()
    B = x.shape[0]
    rest = x.shape[2:]
    oh, ow = gh // sigma, gw // sigma
    grid = x.reshape((B, gh, gw) + rest)
    out = np.zeros((B, oh, ow) + rest, dtype=np.float64)
    for i in range(oh):
        for j in range(ow):
            if mode == AVG:
                acc = np.zeros((B,) + rest, dtype=np.float64)
                for dy in range(sigma):
                    for dx in range(sigma):
                        acc += grid[:, sigma * i + dy, sigma * j + dx]
                out[:, i, j] = acc / (sigma * sigma)
            else:
                out[:, i, j] = grid[:, sigma * i, sigma * j]
    return out.reshape((B, oh * ow) + rest)


def resample_frames(x: np.ndarray, frames: int, gh: int, gw: int, sigma: int,
                    mode: int = AVG) -> np.ndarray:
    """Subsample of a chunk: x [B, frames*gh*gw, ...] holds ``frames`` latent
    frame grids in order; each is resampled on its own and the results are
    concatenated in the same frame order."""
    x = np.asarray(x, dtype=np.float64)
    n = gh * gw
    return np.concatenate([resample(x[:, f * n:(f + 1) * n], gh, gw, sigma, mode)
                           for f in range(frames)], axis=1)


def group_context(kv_win, kv_sink, kv_hist, scales, grid_h, grid_w, g, mode=AVG, frames=1):
    """C_a^MSSA of Eq. 4 for query scale g: [sink || history@g || state_l@max(1,g/s_l)].

    kv_* are one of K or V. Returns [B, Nctx, H, D] float64.
    """
    offs = schedule.token_offsets(scales, grid_h, grid_w, frames)
    cnt = schedule.token_counts(scales, grid_h, grid_w, frames)
    parts = [np.asarray(kv_sink, dtype=np.float64)]
    for f in range(kv_hist.shape[1]):
        parts.append(resample_frames(kv_hist[:, f], frames, grid_h, grid_w, g, mode))
    for l, s in enumerate(scales):
        st = np.asarray(kv_win[:, offs[l]:offs[l] + cnt[l]], dtype=np.float64)
        parts.append(resample_frames(st, frames, grid_h // s, grid_w // s, max(1, g // s), mode))
    return np.concatenate(parts, axis=1)


def attention(q: np.ndarray, k: np.ndarray, v: np.ndarray, scale: float) -> np.ndarray:
    """o_i = sum_j softmax_j(scale * q_i . k_j) v_j, per (b, h); no mask.

    q [B, Nq, H, D], k/v [B, Nk, H, D]; max-subtracted exp, fp64 sums.
    """
    q = np.asarray(q, dtype=np.float64)
    k = np.asarray(k, dtype=np.float64)
    v = np.asarray(v, dtype=np.float64)
    B, Nq, H, D = q.shape
    out = np.empty((B, Nq, H, v.shape[3]), dtype=np.float64)
    for b in range(B):
        for h in range(H):
            s = (q[b, :, h, :] @ k[b, :, h, :].T) * scale
            m = s.max(axis=1, keepdims=True)
            e = np.exp(s - m)
            out[b, :, h, :] = (e @ v[b, :, h, :]) / e.sum(axis=1, keepdims=True)
    return out


def mssa_forward(q, k_win, v_win, k_sink, v_sink, k_hist, v_hist, scales, grid_h, grid_w,
                 mode=AVG, softmax_scale=None, heads=None, frames=1):
    """MSSA over one window: every query group attends to its Eq. 4 context.

    Output [B, N, H, D] in the same token order as q. ``heads`` optionally
    restricts the computation to a list of head indices (the other heads are
    left as NaN), which lets a caller time or check a sample.
    """
    q = np.asarray(q, dtype=np.float64)
    D = q.shape[3]
    scale = D ** -0.5 if not softmax_scale else softmax_scale
    out = np.full(q.shape, np.nan, dtype=np.float64)
    hsel = list(range(q.shape[2])) if heads is None else list(heads)
    for grp in schedule.query_groups(scales, grid_h, grid_w, frames):
        kc = group_context(k_win[:, :, hsel], k_sink[:, :, hsel], k_hist[:, :, :, hsel],
                           scales, grid_h, grid_w, grp.scale, mode, frames)
        vc = group_context(v_win[:, :, hsel], v_sink[:, :, hsel], v_hist[:, :, :, hsel],
                           scales, grid_h, grid_w, grp.scale, mode, frames)
        qg = q[:, grp.q_begin:grp.q_end][:, :, hsel]
        out[:, grp.q_begin:grp.q_end, hsel] = attention(qg, kc, vc, scale)
    return out


def pyramid_segment(kv_win, kv_hist, scales, grid_h, grid_w, g, mode=AVG, frames=1):
    """Only the resampled part of group g's context: history@g followed by the
    window states finer than g, each pooled to scale g. [B, n, H, D] float64."""
    offs = schedule.token_offsets(scales, grid_h, grid_w, frames)
    cnt = schedule.token_counts(scales, grid_h, grid_w, frames)
    parts = []
    for f in range(kv_hist.shape[1]):
        parts.append(resample_frames(kv_hist[:, f], frames, grid_h, grid_w, g, mode))
    for l, s in enumerate(scales):
        if s < g:
            st = np.asarray(kv_win[:, offs[l]:offs[l] + cnt[l]], dtype=np.float64)
            parts.append(resample_frames(st, frames, grid_h // s, grid_w // s, g // s, mode))
    if not parts:
        return np.zeros((kv_win.shape[0], 0) + tuple(kv_win.shape[2:]))
    return np.concatenate(parts, axis=1)


def mssa_lse(q, k_win, k_sink, k_hist, scales, grid_h, grid_w, mode=AVG, softmax_scale=None,
             heads=None, frames=1):
    """Per query row, ln sum_j exp(scale q . k_j) over its Eq. 4 context (the
    softmax normaliser the backward pass rebuilds P from). [B, H, N] float64;
    heads outside ``heads`` are NaN."""
    q = np.asarray(q, dtype=np.float64)
    B, N, H, D = q.shape
    scale = D ** -0.5 if not softmax_scale else softmax_scale
    out = np.full((B, H, N), np.nan, dtype=np.float64)
    hsel = list(range(H)) if heads is None else list(heads)
    for grp in schedule.query_groups(scales, grid_h, grid_w, frames):
        kc = group_context(k_win[:, :, hsel], k_sink[:, :, hsel], k_hist[:, :, :, hsel],
                           scales, grid_h, grid_w, grp.scale, mode, frames)
        for b in range(B):
            for hi, h in enumerate(hsel):
                s = scale * (q[b, grp.q_begin:grp.q_end, h] @ kc[b, :, hi].T)
                m = s.max(axis=1)
                out[b, h, grp.q_begin:grp.q_end] = m + np.log(np.exp(s - m[:, None]).sum(axis=1))
    return out
