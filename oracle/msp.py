"""Multi-Scale Patchification (Sec. 4.1, Eq. 3) in fp64. Test infrastructure.

A latent state [C, Hl, Wl] at window position l is cut into non-overlapping
P_l x P_l patches, P_l = patch * s_l. Token (i, j) (row-major over the
(Hl/P_l) x (Wl/P_l) grid) has feature f = c*P_l^2 + dy*P_l + dx holding
latent[c, P_l*i + dy, P_l*j + dx]; this is the flattening of a Conv2d
patch-embedding weight [E, C, P_l, P_l]. The tier's patch embedding is then a
projection by W_tier [C*P_l^2, E]; de-embedding of an emitted state is a
projection by W_out [E, C*P_l^2] followed by the inverse rearrangement.

A chunked state (Sec. 5.1: F latent frames per state, [C, F, Hl, Wl]) is
patchified frame by frame with the same spatial patch (a Conv3d patch
embedding with temporal extent 1); its tokens are the frames' token grids
in frame order.
"""
from __future__ import annotations

import numpy as np


def patchify(latent: np.ndarray, P: int) -> np.ndarray:
    """[B, C, Hl, Wl] -> [B, (Hl/P)*(Wl/P), C*P*P], written as explicit loops
    over the patch offset so the feature order can be read off directly."""
    x = np.asarray(latent, dtype=np.float64)
    B, C, Hl, Wl = x.shape
    gh, gw = Hl // P, Wl // P
    out = np.empty((B, gh, gw, C * P * P), dtype=np.float64)
    for c in range(C):
        for dy in range(P):
            for dx in range(P):
                out[:, :, :, c * P * P + dy * P + dx] = x[:, c, dy::P, dx::P][:, :gh, :gw]
    return out.reshape(B, gh * gw, C * P * P)


def unpatchify(tokens: np.ndarray, P: int, C: int, Hl: int, Wl: int) -> np.ndarray:
    """Inverse of ``patchify``: [B, (Hl/P)*(Wl/P), C*P*P] -> [B, C, Hl, Wl]."""
    t = np.asarray(tokens, dtype=np.float64)
    B = t.shape[0]
    gh, gw = Hl // P, Wl // P
    t = t.reshape(B, gh, gw, C * P * P)
    out = np.empty((B, C, Hl, Wl), dtype=np.float64)
    for c in range(C):
        for dy in range(P):
            for dx in range(P):
                out[:, c, dy::P, dx::P] = t[:, :, :, c * P * P + dy * P + dx]
    return out


def patchify_chunk(latent: np.ndarray, P: int) -> np.ndarray:
    """[B, C, F, Hl, Wl] -> [B, F*(Hl/P)*(Wl/P), C*P*P]: each latent frame
    patchified on its own, frames one after the other."""
    x = np.asarray(latent, dtype=np.float64)
    return np.concatenate([patchify(x[:, :, f], P) for f in range(x.shape[2])], axis=1)


def unpatchify_chunk(tokens: np.ndarray, P: int, C: int, F: int, Hl: int, Wl: int) -> np.ndarray:
    """Inverse of ``patchify_chunk``: -> [B, C, F, Hl, Wl]."""
    t = np.asarray(tokens, dtype=np.float64)
    n = (Hl // P) * (Wl // P)
    return np.stack([unpatchify(t[:, f * n:(f + 1) * n], P, C, Hl, Wl) for f in range(F)],
                    axis=2)


def patchify_window(latent: np.ndarray, scales, patch: int, w_tier=None):
    """MSP of a whole window: latent [B, T, C, Hl, Wl] (or [B, T, C, F, Hl, Wl]
    for chunked states) -> per-state token blocks.

    Without projections, returns a list of T arrays [B, N_l, C*P_l^2] (raw
    tokens; widths differ between tiers). With ``w_tier`` (dict scale ->
    [C*P_l^2, E]) returns [B, N_MSP, E] with states in position order.
    """
    x = np.asarray(latent, dtype=np.float64)
    cut = patchify_chunk if x.ndim == 6 else patchify
    blocks = [cut(x[:, l], patch * s) for l, s in enumerate(scales)]
    if w_tier is None:
        return blocks
    embs = [blk @ np.asarray(w_tier[s], dtype=np.float64) for blk, s in zip(blocks, scales)]
    return np.concatenate(embs, axis=1)


def unpatchify_state(tokens: np.ndarray, P: int, C: int, Hl: int, Wl: int, w_out=None,
                     frames: int = 0):
    """De-embed (optional) and rearrange one state's tokens back to a latent:
    [B, C, Hl, Wl], or [B, C, F, Hl, Wl] for a chunk of ``frames`` = F >= 1."""
    t = np.asarray(tokens, dtype=np.float64)
    if w_out is not None:
        t = t @ np.asarray(w_out, dtype=np.float64)
    if frames:
        return unpatchify_chunk(t, P, C, frames, Hl, Wl)
    return unpatchify(t, P, C, Hl, Wl)
