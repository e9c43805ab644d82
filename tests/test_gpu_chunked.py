"""GPU parity for chunked window states (Sec. 5.1: each state is a chunk of
F latent frames; patches and Subsample are spatial, frame by frame) against
the fp64 oracle's per-frame definition. Same tolerances as the one-frame
cases: bf16 attention max|err| <= 2e-2, mean <= 2e-3; fp32 <= 1e-4;
permutations bit-exact; AVG pooling within one bf16 ulp of the exact mean.
"""
import dataclasses

import numpy as np
import pytest
import torch

from oracle import msp as omsp
from oracle import mssa as omssa
from oracle import stream as ostream
from paper_2607_20940_gb300 import synth

from helpers import BF16, F32, bf16_round, bind, device_inputs, err_stats, make_plan, msf, oracle_mssa

pytestmark = pytest.mark.gpu

BF16_MAX, BF16_MEAN, F32_MAX = 2e-2, 2e-3, 1e-4

SMALL = synth.CHUNKED_SMALL
# two scales only, 3 frames, D = 64, ragged tails everywhere
SMALL3 = dataclasses.replace(SMALL, name="chunk3_d64", frames=3, head_dim=64, scales=(1, 1, 2),
                             sink_tokens=45, history_frames=2, history_capacity=2, seed=7)


def _run(w, dtype, mode=0):
    x = synth.attention_inputs(w, dtype)
    plan = make_plan(w, dtype, resample=mode)
    dx = device_inputs(x, w.history_capacity)
    ws = bind(plan, dx)
    out = torch.empty_like(dx["q"])
    plan.kv_resample(dx["k_win"], dx["v_win"])
    plan.mssa_forward(dx["q"], dx["k_win"], dx["v_win"], out)
    torch.cuda.synchronize()
    assert plan.device_status() == msf().MSF_OK
    return x, out, plan, ws


@pytest.mark.parametrize("w", [SMALL, SMALL3], ids=lambda w: w.name)
@pytest.mark.parametrize("mode", [0, 1], ids=["avg", "strided"])
def test_chunked_attention_bf16(w, mode):
    x, out, _, _ = _run(w, BF16, mode)
    mx, mean = err_stats(out, oracle_mssa(x, w, mode))
    assert mx <= BF16_MAX and mean <= BF16_MEAN, (mx, mean)


def test_chunked_attention_fp32():
    x, out, _, _ = _run(SMALL, F32, 0)
    mx, _ = err_stats(out, oracle_mssa(x, SMALL, 0))
    assert mx <= F32_MAX, mx


@pytest.mark.parametrize("mode", [0, 1], ids=["avg", "strided"])
def test_chunked_pyramid(mode):
    w = SMALL
    x, _, plan, ws = _run(w, BF16, mode)
    info = plan.info
    B, H, D = w.batch, w.heads, w.head_dim
    for which, off in (("k", info.pyramid_k_offset), ("v", info.pyramid_v_offset)):
        nb = B * info.pyramid_tokens * H * D * 2
        pyr = ws[off:off + nb].view(BF16).view(B, info.pyramid_tokens, H, D)
        for gi in range(info.n_groups):
            g = info.groups[gi]
            if g.scale == 1:
                continue
            got = pyr[:, g.pyr_offset:g.pyr_offset + g.n_pyramid].double().cpu().numpy()
            ref = omssa.pyramid_segment(synth.to_f64(x[which + "_win"]),
                                        synth.to_f64(x[which + "_hist"]), w.scales, w.grid_h,
                                        w.grid_w, g.scale, mode, frames=w.frames)
            if mode == 1:
                assert np.array_equal(got, ref)
            else:
                exact = bf16_round(ref)
                assert np.all(np.abs(got - exact) <= np.abs(exact) * 2.0 ** -7 + 1e-30)


def test_chunked_480p_sampled_heads():
    """The paper's layout at full size (12870 window tokens, one sink chunk,
    one history chunk; 1530.7 GFLOP), in the benchmark's launch
    configuration; the oracle computes every query of two heads."""
    w = synth.CHUNKED_480P
    heads = [0, 7]
    x, out, plan, _ = _run(w, BF16, 0)
    assert plan.info.n_tokens == 12870
    ref = oracle_mssa(x, w, 0, heads=heads)
    mx, mean = err_stats(out, ref, heads=heads)
    assert mx <= BF16_MAX and mean <= BF16_MEAN, (mx, mean)
    assert torch.isfinite(out).all()


def test_chunked_patchify_unpatchify_raw_bit_exact():
    w = SMALL3
    plan = make_plan(w, BF16)
    bind(plan, device_inputs(synth.attention_inputs(w, BF16), w.history_capacity))
    m = synth.msp_inputs(w, BF16, embed_dim=0)
    C, F, P = w.latent_channels, w.frames, w.patch
    Hl, Wl = w.grid_h * P, w.grid_w * P
    raw = torch.empty((w.batch, w.T, C * F * Hl * Wl), dtype=BF16, device="cuda")
    plan.patchify(m["latent"].cuda(), None, raw)
    back = torch.empty((w.batch, C, F, Hl, Wl), dtype=BF16, device="cuda")
    torch.cuda.synchronize()
    lat64 = synth.to_f64(m["latent"])
    for l, s in enumerate(w.scales):
        ref = omsp.patchify_chunk(lat64[:, l], P * s).reshape(w.batch, -1)
        assert np.array_equal(raw[:, l].double().cpu().numpy(), ref)
        plan.unpatchify(l, raw, None, back)
        torch.cuda.synchronize()
        assert torch.equal(back.cpu(), m["latent"][:, l])


def test_chunked_embed_and_deembed_480p():
    """Tier embedding of the five chunked states (12870 tokens, E = 1536) and
    de-embedding + unpatchify of the head chunk back to [C, 3, 60, 104]."""
    w = dataclasses.replace(synth.CHUNKED_480P, heads=2)
    plan = make_plan(w, BF16, embed=True)
    bind(plan, device_inputs(synth.attention_inputs(w, BF16), w.history_capacity))
    m = synth.msp_inputs(w, BF16)
    E, N, F, P = w.embed_dim, plan.info.n_tokens, w.frames, w.patch
    tiers = {s: m["w_tier"][s].t().contiguous().cuda() for s in set(w.scales)}
    tok = torch.empty((w.batch, N, E), dtype=BF16, device="cuda")
    plan.patchify(m["latent"].cuda(), [tiers[s] for s in w.scales], tok)
    w_out = m["w_out"].t().contiguous().cuda()
    lat = torch.empty((w.batch, w.latent_channels, F, w.grid_h * P, w.grid_w * P), dtype=BF16,
                      device="cuda")
    plan.unpatchify(0, tok, w_out, lat)
    torch.cuda.synchronize()
    assert plan.device_status() == msf().MSF_OK
    ref = omsp.patchify_window(synth.to_f64(m["latent"]), w.scales, P,
                               {s: synth.to_f64(m["w_tier"][s]) for s in set(w.scales)})
    e = np.abs(tok.double().cpu().numpy() - ref)
    assert e.max() <= 2.0 ** -7 * np.abs(ref).max() + 1e-3, e.max()
    n0 = plan.info.state_tokens[0]
    ref_lat = omsp.unpatchify_state(synth.to_f64(tok[:, :n0].cpu()), P, w.latent_channels,
                                    w.grid_h * P, w.grid_w * P, synth.to_f64(m["w_out"]), frames=F)
    e2 = np.abs(lat.double().cpu().numpy() - ref_lat)
    assert e2.max() <= 2.0 ** -7 * np.abs(ref_lat).max() + 1e-3, e2.max()


def test_chunked_streaming_ring():
    """Rolling steps with chunked states: the head chunk (F frames, fine)
    enters a ring of capacity 2 and its pyramid levels are pooled per frame;
    ring bit-exact against the oracle's cache, attention against a fresh
    oracle pass each step."""
    w = dataclasses.replace(SMALL, history_frames=1, history_capacity=2, batch=2)
    x = synth.attention_inputs(w, BF16)
    plan = make_plan(w, BF16)
    dx = device_inputs(x, w.history_capacity)
    bind(plan, dx)
    hist = ostream.History(synth.to_f64(x["k_hist"]), synth.to_f64(x["v_hist"]), w.history_capacity)
    G = w.fine_tokens
    for step in range(4):
        kv = synth.step_kv(w, 6000 + step, BF16)
        dkv = {k: v.cuda() for k, v in kv.items()}
        plan.kv_resample(dkv["k_win"], dkv["v_win"],
                         msf().MSF_RESAMPLE_FULL if step == 0 else msf().MSF_RESAMPLE_WINDOW_ONLY)
        out = torch.empty_like(dkv["q"])
        plan.mssa_forward(dkv["q"], dkv["k_win"], dkv["v_win"], out)
        hk, hv = hist.frames()
        ref = omssa.mssa_forward(synth.to_f64(kv["q"]), synth.to_f64(kv["k_win"]),
                                 synth.to_f64(kv["v_win"]), synth.to_f64(x["k_sink"]),
                                 synth.to_f64(x["v_sink"]), hk, hv, w.scales, w.grid_h, w.grid_w,
                                 frames=w.frames)
        mx, mean = err_stats(out, ref)
        assert mx <= BF16_MAX and mean <= BF16_MEAN, (step, mx, mean)
        plan.history_append(dkv["k_win"], dkv["v_win"])
        hist.append(synth.to_f64(kv["k_win"][:, :G]), synth.to_f64(kv["v_win"][:, :G]))
        torch.cuda.synchronize()
        n = hist.count
        assert np.array_equal(dx["k_hist"][:, :n].double().cpu().numpy(), hist.k[:, :n])
        assert np.array_equal(dx["v_hist"][:, :n].double().cpu().numpy(), hist.v[:, :n])
    assert plan.device_status() == msf().MSF_OK
