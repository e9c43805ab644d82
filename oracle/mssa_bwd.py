"""Gradient of Multi-Scale Self-Attention (Eq. 4) in fp64. Test infrastructure.

For a loss L with dL/dO = dO, written out as the definition: per query group
g the context K_g, V_g is built explicitly (mssa.group_context), then for each
(stream, head)

    S = c Q K_g^T,  P = softmax_rows(S),  O = P V_g          (c = 1/sqrt(D))
    dV_g = P^T dO
    dP = dO V_g^T
    dS = P * (dP - rowsum(P * dP))                            (softmax Jacobian)
    dQ = c dS K_g,  dK_g = c dS^T Q

and the context gradients flow back through the context construction: sink
rows to the sink, each history frame's rows to that frame and each window
state's rows to that state, every pooled block through the adjoint of
Subsample (AVG: each of the s x s source tokens receives 1/s^2 of the pooled
row's gradient; STRIDED: the top-left token receives all of it). Gradients of
a token that appears in several groups' contexts add up.

All seven gradients are returned. In Algorithm 1 the cache (sink and history)
is detached (sg), so a training step uses dq, dk_win and dv_win; the others
are here so that invariants over the whole context can be checked.
"""
from __future__ import annotations

import numpy as np

from . import mssa, schedule


def resample_adjoint(dy: np.ndarray, gh: int, gw: int, sigma: int, mode: int = mssa.AVG):
    """Adjoint of mssa.resample: [B, (gh/s)*(gw/s), ...] -> [B, gh*gw, ...]."""
    dy = np.asarray(dy, dtype=np.float64)
    if sigma == 1:
        return dy.copy()
    B = dy.shape[0]
    rest = dy.shape[2:]
    oh, ow = gh // sigma, gw // sigma
    g = dy.reshape((B, oh, ow) + rest)
    out = np.zeros((B, gh, gw) + rest, dtype=np.float64)
    for i in range(oh):
        for j in range(ow):
            if mode == mssa.AVG:
                for a in range(sigma):
                    for b in range(sigma):
                        out[:, sigma * i + a, sigma * j + b] += g[:, i, j] / (sigma * sigma)
            else:
                out[:, sigma * i, sigma * j] += g[:, i, j]
    return out.reshape((B, gh * gw) + rest)


def resample_frames_adjoint(dy, frames, gh, gw, sigma, mode=mssa.AVG):
    """Adjoint of mssa.resample_frames (each latent frame of a chunk on its own)."""
    dy = np.asarray(dy, dtype=np.float64)
    n = (gh // sigma) * (gw // sigma)
    return np.concatenate([resample_adjoint(dy[:, f * n:(f + 1) * n], gh, gw, sigma, mode)
                           for f in range(frames)], axis=1)


def attention_backward(q, k, v, dout, scale):
    """(dq, dk, dv) of o = softmax(scale q k^T) v per (b, h); [B, n, H, D] each."""
    q, k, v, dout = (np.asarray(a, dtype=np.float64) for a in (q, k, v, dout))
    B, Nq, H, D = q.shape
    dq, dk, dv = np.zeros_like(q), np.zeros_like(k), np.zeros_like(v)
    for b in range(B):
        for h in range(H):
            s = scale * (q[b, :, h] @ k[b, :, h].T)
            p = np.exp(s - s.max(axis=1, keepdims=True))
            p /= p.sum(axis=1, keepdims=True)
            do = dout[b, :, h]
            dv[b, :, h] = p.T @ do
            dp = do @ v[b, :, h].T
            ds = p * (dp - (p * dp).sum(axis=1, keepdims=True))
            dq[b, :, h] = scale * (ds @ k[b, :, h])
            dk[b, :, h] = scale * (ds.T @ q[b, :, h])
    return dq, dk, dv


def mssa_backward(q, k_win, v_win, k_sink, v_sink, k_hist, v_hist, dout, scales, grid_h, grid_w,
                  mode=mssa.AVG, softmax_scale=None, frames=1):
    """All gradients of sum(O * dout) for O = mssa.mssa_forward(...): a dict
    with dq, dk_win, dv_win ([B, N, H, D]), dk_sink, dv_sink ([B, Ns, H, D]),
    dk_hist, dv_hist ([B, nh, G, H, D])."""
    f64 = lambda a: np.asarray(a, dtype=np.float64)
    q, k_win, v_win, k_sink, v_sink, k_hist, v_hist, dout = map(
        f64, (q, k_win, v_win, k_sink, v_sink, k_hist, v_hist, dout))
    D = q.shape[3]
    scale = D ** -0.5 if not softmax_scale else softmax_scale
    offs = schedule.token_offsets(scales, grid_h, grid_w, frames)
    cnt = schedule.token_counts(scales, grid_h, grid_w, frames)
    g_ = {n: np.zeros_like(a) for n, a in (("dq", q), ("dk_win", k_win), ("dv_win", v_win),
                                           ("dk_sink", k_sink), ("dv_sink", v_sink),
                                           ("dk_hist", k_hist), ("dv_hist", v_hist))}
    ns, nh = k_sink.shape[1], k_hist.shape[1]
    for grp in schedule.query_groups(scales, grid_h, grid_w, frames):
        g = grp.scale
        kc = mssa.group_context(k_win, k_sink, k_hist, scales, grid_h, grid_w, g, mode, frames)
        vc = mssa.group_context(v_win, v_sink, v_hist, scales, grid_h, grid_w, g, mode, frames)
        qs = slice(grp.q_begin, grp.q_end)
        dq, dkc, dvc = attention_backward(q[:, qs], kc, vc, dout[:, qs], scale)
        g_["dq"][:, qs] += dq
        # context rows back to their sources, in Eq. 4 order
        for key, dc in (("k", dkc), ("v", dvc)):
            r = 0
            g_["d" + key + "_sink"] += dc[:, r:r + ns]
            r += ns
            for f in range(nh):
                n = frames * (grid_h // g) * (grid_w // g)
                g_["d" + key + "_hist"][:, f] += resample_frames_adjoint(
                    dc[:, r:r + n], frames, grid_h, grid_w, g, mode)
                r += n
            for l, s in enumerate(scales):
                st = max(1, g // s)
                n = cnt[l] // (st * st)
                g_["d" + key + "_win"][:, offs[l]:offs[l] + cnt[l]] += resample_frames_adjoint(
                    dc[:, r:r + n], frames, grid_h // s, grid_w // s, st, mode)
                r += n
            assert r == dc.shape[1]
    return g_
