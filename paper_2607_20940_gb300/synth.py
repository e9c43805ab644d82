"""Seeded synthetic inputs for the MSSA/MSP window pass.

This module only draws random numbers and names workload shapes. It holds
none of the method's arithmetic (no token counting, no resampling, no
attention), so both the CUDA path and the fp64 oracle can consume what it
produces without sharing any of the computation.

Draw order for one window-pass layer (one torch CPU generator, fp32
``randn`` scaled by ``std``, then cast to the run dtype):
q, k_win, v_win, k_sink, v_sink, then for each history frame its k and v.
Patchify inputs (latent, tier projections, de-embedding) come from a
separate generator so that they never shift the attention draws.

The five workloads mirror the paper's 480p streaming setting (Sec. 5.1:
832x480 video, Wan latent 60x104 with 16 channels, patch 2 -> a 30x52 token
grid, a T=5 window with patch schedule (p,p,2p,2p,2p), Eq. 3). They stand in
for the paper's Wan2.1 activations, which need trained weights and data.
"""
from __future__ import annotations

import dataclasses
from typing import Optional, Sequence

import torch


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    T: int
    scales: tuple
    grid_h: int
    grid_w: int
    heads: int
    head_dim: int
    sink_tokens: int
    history_frames: int
    history_capacity: int
    batch: int
    seed: int
    std: float = 1.0
    layers: int = 1
    steps: int = 1
    latent_channels: int = 16
    patch: int = 2
    embed_dim: int = 0
    frames: int = 1   # latent frames per window state (a chunk)

    @property
    def fine_tokens(self) -> int:
        return self.frames * self.grid_h * self.grid_w

    def with_scales(self, scales: Sequence[int]) -> "Workload":
        return dataclasses.replace(self, scales=tuple(scales))


# Tiny case the oracle finishes instantly: T=3, 8x8 grid, scales (1,1,2).
TINY = Workload("tiny_t3_8x8_h2_d64", 3, (1, 1, 2), 8, 8, 2, 64, 64, 1, 1, 1, 0,
                patch=2, latent_channels=16)
# One 480p-shaped layer: T=5, 30x52 fine grid, scales (1,1,2,2,2), 12x128 heads.
LAYER_480P = Workload("mssa_480p_t5_30x52_h12_d128", 5, (1, 1, 2, 2, 2), 30, 52, 12, 128,
                      1560, 2, 2, 1, 1, patch=2, latent_channels=16, embed_dim=1536)
# Full window pass: 30 stacked layers at 480p shapes, std 0.5, seeds 100+l.
PASS_480P = dataclasses.replace(LAYER_480P, name="window_pass_480p_30_layers", seed=100,
                                std=0.5, layers=30)
# Three-scale 48x80 window: T=6, scales (1,1,2,2,4,4), 16 heads.
THREE_SCALE = Workload("mssa_3scale_t6_48x80_h16_d128", 6, (1, 1, 2, 2, 4, 4), 48, 80, 16,
                       128, 3840, 2, 2, 1, 3, patch=2, latent_channels=16)
# Streaming rollout: 480p layer, 4 streams, history 2 growing to capacity 4.
STREAM_480P = dataclasses.replace(LAYER_480P, name="stream_480p_b4_cap4_120_steps", batch=4,
                                  history_capacity=4, seed=4, steps=120)

# The paper's own window layout (Sec. 5.1): every state a chunk of 3 latent
# frames (4680 fine tokens at 480p), sink = one chunk, one history chunk.
CHUNKED_480P = dataclasses.replace(LAYER_480P, name="mssa_480p_chunk3_t5_30x52_h12_d128",
                                   frames=3, sink_tokens=3 * 1560, history_frames=1,
                                   history_capacity=1, seed=5)
# Small chunked case for element-wise parity: 2 frames per state, 8x12 grid.
CHUNKED_SMALL = Workload("chunk2_t3_8x12_h2_d128", 3, (1, 2, 4), 8, 12, 2, 128, 70, 1, 2, 1, 6,
                         patch=2, latent_channels=16, embed_dim=256, frames=2)

WORKLOADS = {w.name: w for w in (TINY, LAYER_480P, PASS_480P, THREE_SCALE, STREAM_480P,
                                 CHUNKED_480P, CHUNKED_SMALL)}


def _randn(gen: torch.Generator, shape, std: float, dtype: torch.dtype) -> torch.Tensor:
    x = torch.randn(*shape, generator=gen, dtype=torch.float32)
    if std != 1.0:
        x = x * std
    return x.to(dtype)


def window_tokens(w: Workload) -> int:
    """Sum of per-state grid sizes; plain shape bookkeeping for allocation."""
    return sum(w.frames * (w.grid_h // s) * (w.grid_w // s) for s in w.scales)


def attention_inputs(w: Workload, dtype: torch.dtype = torch.bfloat16, seed: Optional[int] = None,
                     history_frames: Optional[int] = None) -> dict:
    """q/k/v for one window-pass layer, as CPU tensors in ``dtype``.

    Layouts: q, k_win, v_win ``[B, N, H, D]``; k_sink, v_sink ``[B, Ns, H, D]``;
    k_hist, v_hist ``[B, nh, Gh*Gw, H, D]`` (history frames at the fine grid).
    """
    seed = w.seed if seed is None else seed
    nh = w.history_frames if history_frames is None else history_frames
    gen = torch.Generator().manual_seed(seed)
    B, H, D = w.batch, w.heads, w.head_dim
    N = window_tokens(w)
    out = {}
    out["q"] = _randn(gen, (B, N, H, D), w.std, dtype)
    out["k_win"] = _randn(gen, (B, N, H, D), w.std, dtype)
    out["v_win"] = _randn(gen, (B, N, H, D), w.std, dtype)
    out["k_sink"] = _randn(gen, (B, w.sink_tokens, H, D), w.std, dtype)
    out["v_sink"] = _randn(gen, (B, w.sink_tokens, H, D), w.std, dtype)
    G = w.fine_tokens
    kh = torch.empty((B, nh, G, H, D), dtype=dtype)
    vh = torch.empty((B, nh, G, H, D), dtype=dtype)
    for f in range(nh):
        kh[:, f] = _randn(gen, (B, G, H, D), w.std, dtype)
        vh[:, f] = _randn(gen, (B, G, H, D), w.std, dtype)
    out["k_hist"] = kh
    out["v_hist"] = vh
    return out


def step_kv(w: Workload, seed: int, dtype: torch.dtype = torch.bfloat16) -> dict:
    """Fresh q/k/v for one streaming step (no sink or history draws)."""
    gen = torch.Generator().manual_seed(seed)
    B, H, D = w.batch, w.heads, w.head_dim
    N = window_tokens(w)
    return {k: _randn(gen, (B, N, H, D), w.std, dtype) for k in ("q", "k_win", "v_win")}


def msp_inputs(w: Workload, dtype: torch.dtype = torch.bfloat16, seed: Optional[int] = None,
               embed_dim: Optional[int] = None) -> dict:
    """Latent window and seeded random tier projections for patchify/unpatchify.

    latent ``[B, T, C, Hl, Wl]`` (``[B, T, C, F, Hl, Wl]`` for chunks of F > 1
    latent frames) ~ N(0,1); for each distinct scale s a tier
    projection ``[C*(patch*s)^2, E]`` ~ N(0, 1/(C*(patch*s)^2)); the fine
    de-embedding ``[E, C*patch^2]`` ~ N(0, 1/E). With ``embed_dim`` 0 only
    the latent is drawn.
    """
    seed = (w.seed if seed is None else seed) + 7919
    E = w.embed_dim if embed_dim is None else embed_dim
    gen = torch.Generator().manual_seed(seed)
    C, P = w.latent_channels, w.patch
    Hl, Wl = w.grid_h * P, w.grid_w * P
    lat = (w.batch, w.T, C, Hl, Wl) if w.frames == 1 else (w.batch, w.T, C, w.frames, Hl, Wl)
    out = {"latent": _randn(gen, lat, 1.0, dtype)}
    if E:
        tiers = {}
        for s in sorted(set(w.scales)):
            F = C * (P * s) ** 2
            tiers[s] = _randn(gen, (F, E), F ** -0.5, dtype)
        out["w_tier"] = tiers
        F1 = C * (P * w.scales[0]) ** 2
        out["w_out"] = _randn(gen, (E, F1), E ** -0.5, dtype)
    return out


def tier_inputs(w: Workload, rank: int, dtype: torch.dtype = torch.bfloat16,
                seed: Optional[int] = None, gamma: float = 0.5) -> dict:
    """Seeded weights of the coarse tiers' modules (every scale s > 1 of the
    window), in the row-vector orientation x @ W, for each scale s with
    K = C*(patch*s)^2: LoRA of the embedding ``lora_a`` [K, r] ~ N(0, 1/K),
    ``lora_b`` [r, E] ~ N(0, 1/r); a de-embedding ``w_out`` [E, K] ~ N(0, 1/E)
    with LoRA ``out_a`` [E, r] ~ N(0, 1/E), ``out_b`` [r, K] ~ N(0, 1/r); the
    latent residual ``residual`` [K, K] ~ N(0, 1/K); and the LoRA scale
    ``gamma``. The tier's embedding ``w`` is msp_inputs' w_tier[s]. Drawn
    from their own generator, after nothing else."""
    seed = (w.seed if seed is None else seed) + 104729
    gen = torch.Generator().manual_seed(seed)
    C, E, r = w.latent_channels, w.embed_dim, rank
    out = {}
    for s in sorted(set(w.scales)):
        if s == 1:
            continue
        K = C * (w.patch * s) ** 2
        out[s] = {
            "lora_a": _randn(gen, (K, r), K ** -0.5, dtype),
            "lora_b": _randn(gen, (r, E), r ** -0.5, dtype),
            "w_out": _randn(gen, (E, K), E ** -0.5, dtype),
            "out_a": _randn(gen, (E, r), E ** -0.5, dtype),
            "out_b": _randn(gen, (r, K), r ** -0.5, dtype),
            "residual": _randn(gen, (K, K), K ** -0.5, dtype),
            "gamma": gamma,
        }
    return out


def to_f64(t: torch.Tensor):
    """Exact widening of the stored values to a float64 numpy array."""
    return t.to(torch.float64).numpy()
