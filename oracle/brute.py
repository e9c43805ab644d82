"""A second enumeration of Eq. 4, query by query, for tiny grids.

Test infrastructure. Shares no helper with mssa.py: for each query token it
decides which window position it belongs to by scanning the states, lists
the visible key/value rows straight from the set definition
C_a = [C_sink || Concat_{b in V(a)} Subsample(C_b, max(1, p_a/p_b))] with
the subsampled rows built by explicit loops over each block, and evaluates
softmax attention with scalar Python loops. Pure Python; only for inputs
with a few hundred tokens. With chunked states (``frames`` = F latent frames
per state, Sec. 5.1) every state and history frame is F grids in a row, and
each grid is subsampled on its own.
"""
from __future__ import annotations

import math


def _state_of(token, scales, gh, gw, frames=1):
    start = 0
    for l, s in enumerate(scales):
        n = frames * (gh // s) * (gw // s)
        if token < start + n:
            return l, start
        start += n
    raise IndexError(token)


def _block(frame, fgh, fgw, stride, i, j, b, h, mode):
    """One subsampled row: frame is indexed frame[b][token][h] -> list of D floats."""
    D = len(frame[b][0][h])
    if mode == 1:
        return list(frame[b][(stride * i) * fgw + stride * j][h])
    acc = [0.0] * D
    for dy in range(stride):
        for dx in range(stride):
            row = frame[b][(stride * i + dy) * fgw + (stride * j + dx)][h]
            for d in range(D):
                acc[d] += float(row[d])
    return [a / (stride * stride) for a in acc]


def mssa_brute(q, k_win, v_win, k_sink, v_sink, k_hist, v_hist, scales, grid_h, grid_w,
               mode=0, softmax_scale=None, frames=1):
    """Nested lists / arrays in, nested lists out ([B][N][H][D])."""
    B, N, H, D = len(q), len(q[0]), len(q[0][0]), len(q[0][0][0])
    scale = softmax_scale or 1.0 / math.sqrt(D)
    # per-state views of the window tensors
    views = []
    start = 0
    for s in scales:
        n = frames * (grid_h // s) * (grid_w // s)
        views.append((start, n, s))
        start += n
    G = grid_h * grid_w
    out = [[[None] * H for _ in range(N)] for _ in range(B)]
    for b in range(B):
        for t in range(N):
            la, _ = _state_of(t, scales, grid_h, grid_w, frames)
            pa = scales[la]
            for h in range(H):
                keys, vals = [], []
                for n in range(len(k_sink[b])):
                    keys.append([float(x) for x in k_sink[b][n][h]])
                    vals.append([float(x) for x in v_sink[b][n][h]])
                # history frames: fine (p_b = p), stride max(1, p_a / p),
                # every latent frame of a chunk on its own
                for f in range(len(k_hist[b])):
                    st = max(1, pa)
                    for lf in range(frames):
                        for i in range(grid_h // st):
                            for j in range(grid_w // st):
                                keys.append(_hist_block(k_hist, b, f, lf * G, grid_w, st, i, j,
                                                        h, mode))
                                vals.append(_hist_block(v_hist, b, f, lf * G, grid_w, st, i, j,
                                                        h, mode))
                # window positions, the query's own included
                for (s0, n, pb) in views:
                    st = max(1, pa // pb)
                    fgh, fgw = grid_h // pb, grid_w // pb
                    for lf in range(frames):
                        base = s0 + lf * fgh * fgw
                        kf = [[k_win[b][base + r] for r in range(fgh * fgw)]]
                        vf = [[v_win[b][base + r] for r in range(fgh * fgw)]]
                        for i in range(fgh // st):
                            for j in range(fgw // st):
                                keys.append(_block(kf, fgh, fgw, st, i, j, 0, h, mode))
                                vals.append(_block(vf, fgh, fgw, st, i, j, 0, h, mode))
                qv = [float(x) for x in q[b][t][h]]
                logits = [scale * sum(qv[d] * kk[d] for d in range(D)) for kk in keys]
                m = max(logits)
                w = [math.exp(x - m) for x in logits]
                z = sum(w)
                out[b][t][h] = [sum(w[j] * vals[j][d] for j in range(len(w))) / z for d in range(D)]
    return out


def _hist_block(hist, b, f, base, fgw, st, i, j, h, mode):
    frame = [hist[b][f][base:]]
    return _block(frame, None, fgw, st, i, j, 0, h, mode)
