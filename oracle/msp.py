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


# ------------------------------------------------------------ tier modules --
#
# Sec. 4.1 gives every coarse tier its own module: patch embedding and
# de-embedding, LoRA adapters and a latent residual branch; the native tier
# keeps the pretrained path and has none of the extras. The paper does not
# fix where the adapters sit or what the residual branch computes; the
# reading taken here (row vectors, x @ W):
#   embedding      t = x W + g (x A) B          W [K, E], A [K, r], B [r, E]
#   de-embedding   y = h Wo + g (h Ao) Bo + x R  Wo [E, K], Ao [E, r], Bo [r, K]
# where x is the state's raw patch vector (K = C*P^2 features, the input
# latent of the same state), h its token after the backbone, g the LoRA
# scale and R [K, K] the latent residual branch: a learned linear map of the
# input patch added to the de-embedded output before the patches are put back.
# Every term is an fp64 matrix product in the order written.

def embed_tier(x, w, lora_a=None, lora_b=None, gamma=1.0):
    """Tier patch embedding of raw patch vectors x [..., K] -> [..., E]."""
    x = np.asarray(x, dtype=np.float64)
    t = x @ np.asarray(w, dtype=np.float64)
    if lora_a is not None:
        t = t + gamma * ((x @ np.asarray(lora_a, dtype=np.float64)) @ np.asarray(lora_b, dtype=np.float64))
    return t


def deembed_tier(h, w_out, lora_a=None, lora_b=None, gamma=1.0, x=None, residual=None):
    """Tier de-embedding of tokens h [..., E] -> patch vectors [..., K], with
    the latent residual x R of the state's input patch vectors x [..., K]."""
    h = np.asarray(h, dtype=np.float64)
    y = h @ np.asarray(w_out, dtype=np.float64)
    if lora_a is not None:
        y = y + gamma * ((h @ np.asarray(lora_a, dtype=np.float64)) @ np.asarray(lora_b, dtype=np.float64))
    if residual is not None:
        y = y + np.asarray(x, dtype=np.float64) @ np.asarray(residual, dtype=np.float64)
    return y


def patchify_window_tiers(latent, scales, patch, tiers):
    """MSP of a window with tier modules: latent [B, T, C, Hl, Wl] ->
    [B, N_MSP, E], states in position order. tiers: dict scale -> dict with
    'w' [K, E] and optionally 'lora_a' [K, r], 'lora_b' [r, E], 'gamma'."""
    x = np.asarray(latent, dtype=np.float64)
    out = []
    for l, s in enumerate(scales):
        t = tiers[s]
        xp = patchify(x[:, l], patch * s)
        out.append(embed_tier(xp, t["w"], t.get("lora_a"), t.get("lora_b"), t.get("gamma", 1.0)))
    return np.concatenate(out, axis=1)


def unpatchify_state_tier(tokens, latent_state, P, tier):
    """De-embedding of one state with its tier module: tokens [B, N_l, E] and
    the state's input latent [B, C, Hl, Wl] -> output latent [B, C, Hl, Wl].
    tier: dict with 'w_out' [E, K] and optionally 'out_a' [E, r], 'out_b'
    [r, K], 'gamma', 'residual' [K, K]."""
    lat = np.asarray(latent_state, dtype=np.float64)
    B, C, Hl, Wl = lat.shape
    x = patchify(lat, P)
    y = deembed_tier(tokens, tier["w_out"], tier.get("out_a"), tier.get("out_b"),
                     tier.get("gamma", 1.0), x, tier.get("residual"))
    return unpatchify(y, P, C, Hl, Wl)
