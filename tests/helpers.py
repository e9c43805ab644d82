"""Shared test plumbing: plans from workloads, device copies, oracle calls."""
from __future__ import annotations

import numpy as np
import torch

from oracle import msp as omsp
from oracle import mssa as omssa
from paper_2607_20940_gb300 import synth

BF16 = torch.bfloat16
F32 = torch.float32


def msf():
    from paper_2607_20940_gb300 import msf as m
    return m


def make_plan(w: synth.Workload, dtype=BF16, resample=0, history_capacity=None, embed=False):
    m = msf()
    desc = m.make_desc(w.scales, w.grid_h, w.grid_w, w.heads, w.head_dim, w.sink_tokens,
                       w.history_frames,
                       history_capacity=w.history_capacity if history_capacity is None else history_capacity,
                       batch=w.batch, dtype=m.MSF_DTYPE_BF16 if dtype == BF16 else m.MSF_DTYPE_F32,
                       resample=resample, latent_channels=w.latent_channels, patch=w.patch,
                       embed_dim=w.embed_dim if embed else 0, frames_per_state=w.frames)
    return m.Plan(desc)


def device_inputs(x: dict, cap: int, device="cuda"):
    """Copy attention inputs to the device; the history ring gets `cap` slots
    with the live frames first (the rest zero)."""
    d = {k: v.to(device) for k, v in x.items() if k not in ("k_hist", "v_hist")}
    B, nh, G, H, D = x["k_hist"].shape
    for k in ("k_hist", "v_hist"):
        ring = torch.zeros((B, max(cap, 1), G, H, D), dtype=x[k].dtype, device=device)
        ring[:, :nh] = x[k].to(device)
        d[k] = ring
    return d


def bind(plan, dx):
    ws = plan.workspace()
    plan.bind(ws, dx["k_sink"], dx["v_sink"], dx["k_hist"], dx["v_hist"])
    return ws


def oracle_mssa(x: dict, w: synth.Workload, mode=0, heads=None):
    f = synth.to_f64
    return omssa.mssa_forward(f(x["q"]), f(x["k_win"]), f(x["v_win"]), f(x["k_sink"]),
                              f(x["v_sink"]), f(x["k_hist"]), f(x["v_hist"]), w.scales,
                              w.grid_h, w.grid_w, mode=mode, heads=heads, frames=w.frames)


def err_stats(got: torch.Tensor, ref: np.ndarray, heads=None):
    g = got.detach().to(torch.float64).cpu().numpy()
    if heads is not None:
        g = g[:, :, heads]
        ref = ref[:, :, heads]
    e = np.abs(g - ref)
    return float(e.max()), float(e.mean())


def bf16_round(x: np.ndarray) -> np.ndarray:
    """Round-to-nearest-even of fp64 values to bf16, returned as fp64."""
    return torch.from_numpy(np.ascontiguousarray(x)).to(torch.float32).to(BF16).to(torch.float64).numpy()
