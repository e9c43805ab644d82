"""Tier modules of MSP (Sec. 4.1) on the GPU against the fp64 oracle.

Every coarse tier gets rank-r LoRA adapters on its patch embedding and
de-embedding and a latent residual branch (the reading stated in
include/msf.h and oracle/msp.py); the native tier keeps the plain path. The
embedding of the whole window and the de-embedding of coarse and fine
positions are compared element by element with oracle.msp on the same bf16
values: tolerance 2^-7 of the output's range (bf16 output rounding, plus the
one rounding of the rank-r codes to bf16).
"""
import dataclasses

import numpy as np
import pytest
import torch

from oracle import msp as omsp
from paper_2607_20940_gb300 import synth

from helpers import BF16, make_plan, msf

pytestmark = pytest.mark.gpu

SMALL = synth.Workload("tier_t4_8x12_e256", 4, (1, 1, 2, 2), 8, 12, 2, 128, 96, 1, 1, 2, 9,
                       patch=2, latent_channels=16, embed_dim=256)


def _setup(w, rank, lora=True, residual=True, gamma=0.5):
    m = msf()
    plan = make_plan(w, BF16, embed=True)
    sink = torch.zeros((w.batch, w.sink_tokens, w.heads, w.head_dim), dtype=BF16, device="cuda")
    ring = torch.zeros((w.batch, max(w.history_capacity, 1), w.fine_tokens, w.heads, w.head_dim),
                       dtype=BF16, device="cuda")
    plan.bind(plan.workspace(), sink, sink, ring, ring)
    mi = synth.msp_inputs(w, BF16)
    ti = synth.tier_inputs(w, rank, BF16, gamma=gamma)
    dev = {}  # keeps the device tensors alive
    mods, otier = {}, {}
    for s in sorted(set(w.scales)):
        wt = mi["w_tier"][s]                       # [K, E] (x @ W)
        d = {"w_embed": wt.t().contiguous().cuda()}
        o = {"w": synth.to_f64(wt)}
        if s == 1:
            w_out = mi["w_out"]                    # [E, K]
            d["w_out"] = w_out.t().contiguous().cuda()
            o["w_out"] = synth.to_f64(w_out)
            mod = m.tier_module(d["w_embed"], d["w_out"])
        else:
            t = ti[s]
            d["w_out"] = t["w_out"].t().contiguous().cuda()
            o["w_out"] = synth.to_f64(t["w_out"])
            kw = {}
            if lora:
                d["embed_down"] = t["lora_a"].t().contiguous().cuda()   # [r, K]
                d["embed_up"] = t["lora_b"].t().contiguous().cuda()     # [E, r]
                d["out_down"] = t["out_a"].t().contiguous().cuda()      # [r, E]
                d["out_up"] = t["out_b"].t().contiguous().cuda()        # [K, r]
                kw.update(embed_down=d["embed_down"], embed_up=d["embed_up"], out_down=d["out_down"],
                          out_up=d["out_up"], lora_rank=rank, lora_scale=t["gamma"])
                o.update(lora_a=synth.to_f64(t["lora_a"]), lora_b=synth.to_f64(t["lora_b"]),
                         out_a=synth.to_f64(t["out_a"]), out_b=synth.to_f64(t["out_b"]),
                         gamma=t["gamma"])
            if residual:
                d["residual"] = t["residual"].t().contiguous().cuda()   # [K_out, K_in]
                kw["residual"] = d["residual"]
                o["residual"] = synth.to_f64(t["residual"])
            mod = m.tier_module(d["w_embed"], d["w_out"], **kw)
        dev[s], mods[s], otier[s] = d, mod, o
    return plan, mi, dev, mods, otier


def _tol(ref):
    return 2.0 ** -7 * np.abs(ref).max() + 1e-3


def _check_window(w, rank, lora=True, residual=True):
    plan, mi, dev, mods, otier = _setup(w, rank, lora, residual)
    N, E = plan.info.n_tokens, w.embed_dim
    lat = mi["latent"].cuda()
    tok = torch.full((w.batch, N, E), float("nan"), dtype=BF16, device="cuda")
    plan.patchify_tiers(lat, [mods[s] for s in w.scales], tok)
    torch.cuda.synchronize()
    assert plan.device_status() == msf().MSF_OK
    x = synth.to_f64(mi["latent"])
    if w.frames == 1:
        ref = omsp.patchify_window_tiers(x, w.scales, w.patch, otier)
    else:  # chunks: each latent frame is patchified on its own (spatial patches)
        ref = np.concatenate(
            [np.concatenate([omsp.embed_tier(omsp.patchify(x[:, l, :, f], w.patch * s), otier[s]["w"],
                                             otier[s].get("lora_a"), otier[s].get("lora_b"),
                                             otier[s].get("gamma", 1.0)) for f in range(w.frames)], 1)
             for l, s in enumerate(w.scales)], 1)
    got = tok.double().cpu().numpy()
    assert np.isfinite(got).all()
    err = np.abs(got - ref).max()
    assert err <= _tol(ref), err
    # de-embedding of every position from the bf16 tokens just made
    info = plan.info
    Hl, Wl = w.grid_h * w.patch, w.grid_w * w.patch
    shape = (w.batch, w.latent_channels) + ((w.frames,) if w.frames > 1 else ()) + (Hl, Wl)
    for pos, s in enumerate(w.scales):
        out = torch.full(shape, float("nan"), dtype=BF16, device="cuda")
        plan.unpatchify_tier(pos, tok, lat, mods[s], out.view(w.batch, w.latent_channels, -1, Wl))
        torch.cuda.synchronize()
        assert plan.device_status() == msf().MSF_OK
        o0, n = info.state_offset[pos], info.state_tokens[pos]
        P = w.patch * s
        t_h = tok[:, o0:o0 + n].double().cpu().numpy()
        if w.frames == 1:
            ref_l = omsp.unpatchify_state_tier(t_h, x[:, pos], P, otier[s])
        else:
            per = n // w.frames
            ref_l = np.stack([omsp.unpatchify_state_tier(t_h[:, f * per:(f + 1) * per], x[:, pos, :, f], P,
                                                         otier[s]) for f in range(w.frames)], axis=2)
        g = out.double().cpu().numpy()
        assert np.isfinite(g).all(), pos
        e = np.abs(g - ref_l).max()
        assert e <= _tol(ref_l), (pos, e)


@pytest.mark.parametrize("rank", [8, 32, 64])
def test_tier_modules_small_window(rank):
    _check_window(SMALL, rank)


def test_tier_modules_without_adapters_or_residual():
    _check_window(SMALL, 16, lora=False, residual=True)
    _check_window(SMALL, 16, lora=True, residual=False)


def test_tier_modules_480p_window():
    _check_window(synth.LAYER_480P, 32)


def test_tier_modules_480p_two_streams():
    _check_window(dataclasses.replace(synth.LAYER_480P, batch=2, heads=2), 16)


def test_tier_modules_chunked_states():
    _check_window(synth.CHUNKED_SMALL, 16)


def test_tier_module_rejects_bad_rank():
    plan, mi, dev, mods, otier = _setup(SMALL, 16)
    bad = msf().tier_module(dev[2]["w_embed"], dev[2]["w_out"], embed_down=dev[2]["embed_down"],
                            embed_up=dev[2]["embed_up"], lora_rank=12, lora_scale=0.5)
    N, E = plan.info.n_tokens, SMALL.embed_dim
    tok = torch.empty((SMALL.batch, N, E), dtype=BF16, device="cuda")
    with pytest.raises(Exception):
        plan.patchify_tiers(mi["latent"].cuda(), [mods[1], mods[1], bad, bad], tok)
