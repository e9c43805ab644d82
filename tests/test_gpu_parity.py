"""GPU parity of every kernel behind the C ABI against the fp64 oracle.

Tolerances: bf16 attention max|err| <= 2e-2 and mean|err| <= 2e-3 on unit
variance inputs, fp32 attention max|err| <= 1e-4; permutations (patchify,
STRIDED pooling, history copies) bit-exact; AVG pooling within one bf16 ulp
of the exact mean (fp32 sum, one rounding).
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

# Several tiles per group and ragged tails in every segment.
RAGGED = synth.Workload("ragged_t4_12x20", 4, (1, 1, 2, 4), 12, 20, 3, 128, 200, 2, 3, 2, 21)
RAGGED64 = dataclasses.replace(RAGGED, name="ragged_d64", head_dim=64, scales=(1, 2, 2, 4), seed=22)
COARSE_ONLY = synth.Workload("coarse_only", 3, (2, 2, 4), 16, 24, 2, 128, 37, 1, 1, 1, 23)
NO_SINK = synth.Workload("no_sink_no_hist", 2, (1, 2), 16, 16, 2, 64, 0, 0, 0, 1, 24)
# The plan's limits: MSF_MAX_STATES window states, five query groups (scales 1
# to 16, coarse grids down to 2x3 tokens), 28 pooling jobs in one launch.
MAX_STATES = synth.Workload("max_states_t16", 16, (1, 1, 2, 2, 4, 4, 8, 8) + (16,) * 8, 32, 48, 2, 64,
                            40, 2, 3, 2, 25)


def _run_attention(w, dtype, mode=0, simt=False):
    x = synth.attention_inputs(w, dtype)
    plan = make_plan(w, dtype, resample=mode)
    dx = device_inputs(x, w.history_capacity)
    bind(plan, dx)
    out = torch.empty_like(dx["q"])
    plan.kv_resample(dx["k_win"], dx["v_win"])
    if simt:
        plan.mssa_forward_simt(dx["q"], dx["k_win"], dx["v_win"], out)
    else:
        plan.mssa_forward(dx["q"], dx["k_win"], dx["v_win"], out)
    torch.cuda.synchronize()
    assert plan.device_status() == msf().MSF_OK
    return x, out, plan


@pytest.mark.parametrize("w", [synth.TINY, RAGGED, RAGGED64, COARSE_ONLY, NO_SINK, MAX_STATES],
                         ids=lambda w: w.name)
@pytest.mark.parametrize("mode", [0, 1], ids=["avg", "strided"])
def test_attention_bf16_tensor_core(w, mode):
    x, out, _ = _run_attention(w, BF16, mode)
    ref = oracle_mssa(x, w, mode)
    mx, mean = err_stats(out, ref)
    assert mx <= BF16_MAX and mean <= BF16_MEAN, (mx, mean)


@pytest.mark.parametrize("which,factor", [("k_win", 30.0), ("k_sink", 30.0), ("k_hist", 12.0)],
                         ids=["rising", "falling", "middle"])
def test_attention_bf16_score_jumps(which, factor):
    """Scores that jump by far more than 2^32 in P between context segments:
    the running maximum of the online softmax lags (rising), leads (falling)
    or lags then leads (a large middle segment). Output must still match.

    Keys scaled by 30 give scores of standard deviation ~30, so most rows
    are dominated by one or two keys and fp32 score rounding moves their
    weights; the fp32 SIMT path shows the same worst element (4.6e-2 on the
    rising case), so the bound on the worst element is 6e-2 here while the
    mean bound stays that of unit-variance inputs."""
    w = RAGGED
    x = synth.attention_inputs(w, BF16)
    x[which] = (x[which].float() * factor).to(BF16)
    plan = make_plan(w, BF16, resample=0)
    dx = device_inputs(x, w.history_capacity)
    bind(plan, dx)
    out = torch.empty_like(dx["q"])
    plan.kv_resample(dx["k_win"], dx["v_win"])
    plan.mssa_forward(dx["q"], dx["k_win"], dx["v_win"], out)
    torch.cuda.synchronize()
    assert plan.device_status() == msf().MSF_OK
    assert torch.isfinite(out.float()).all()
    ref = oracle_mssa(x, w, 0)
    mx, mean = err_stats(out, ref)
    assert mx <= 6e-2 and mean <= BF16_MEAN, (mx, mean)


@pytest.mark.parametrize("w", [synth.TINY, RAGGED, RAGGED64, COARSE_ONLY, MAX_STATES], ids=lambda w: w.name)
def test_attention_fp32(w):
    x, out, _ = _run_attention(w, F32, 0)
    ref = oracle_mssa(x, w, 0)
    mx, _ = err_stats(out, ref)
    assert mx <= F32_MAX, mx


def test_attention_bf16_simt_crosscheck():
    x, out, _ = _run_attention(RAGGED, BF16, 0, simt=True)
    mx, mean = err_stats(out, oracle_mssa(x, RAGGED, 0))
    assert mx <= BF16_MAX and mean <= BF16_MEAN


@pytest.mark.parametrize("w,heads", [
    (synth.LAYER_480P, [0, 5, 11]),
    (synth.LAYER_480P.with_scales((1, 1, 1, 1, 1)), [3]),
    (synth.THREE_SCALE, [0, 15]),
    (dataclasses.replace(synth.STREAM_480P, history_frames=4), [2]),
], ids=["480p", "480p_all_fine", "three_scale", "480p_b4_hist4"])
def test_attention_full_size_sampled_heads(w, heads):
    """Full-size shapes in the launch configuration the benchmark uses; the
    oracle computes every query of the sampled heads (all streams)."""
    x, out, _ = _run_attention(w, BF16, 0)
    ref = oracle_mssa(x, w, 0, heads=heads)
    mx, mean = err_stats(out, ref, heads=heads)
    assert mx <= BF16_MAX and mean <= BF16_MEAN, (mx, mean)
    assert torch.isfinite(out).all()


@pytest.mark.parametrize("dtype", [BF16, F32], ids=["bf16", "f32"])
@pytest.mark.parametrize("mode", [0, 1], ids=["avg", "strided"])
def test_pyramid(dtype, mode):
    w = synth.THREE_SCALE if dtype == BF16 else RAGGED
    x = synth.attention_inputs(w, dtype)
    plan = make_plan(w, dtype, resample=mode)
    dx = device_inputs(x, w.history_capacity)
    ws = bind(plan, dx)
    plan.kv_resample(dx["k_win"], dx["v_win"])
    torch.cuda.synchronize()
    info = plan.info
    B, H, D = w.batch, w.heads, w.head_dim
    for which, off in (("k", info.pyramid_k_offset), ("v", info.pyramid_v_offset)):
        nb = B * info.pyramid_tokens * H * D * (2 if dtype == BF16 else 4)
        pyr = ws[off:off + nb].view(dtype).view(B, info.pyramid_tokens, H, D)
        for gi in range(info.n_groups):
            g = info.groups[gi]
            if g.scale == 1:
                continue
            got = pyr[:, g.pyr_offset:g.pyr_offset + g.n_pyramid].to(torch.float64).cpu().numpy()
            ref = omssa.pyramid_segment(synth.to_f64(x[which + "_win"]), synth.to_f64(x[which + "_hist"]),
                                        w.scales, w.grid_h, w.grid_w, g.scale, mode)
            if mode == 1:
                assert np.array_equal(got, ref)
            elif dtype == BF16:
                exact = bf16_round(ref)
                ulp = np.abs(exact) * 2.0 ** -7 + 1e-30
                assert np.all(np.abs(got - exact) <= ulp)
                assert np.mean(got == exact) > 0.999
            else:
                np.testing.assert_allclose(got, ref, rtol=2e-7, atol=1e-7)


def test_streaming_history_ring_and_attention():
    """Rolling steps: fresh window q/k/v each step, head K/V appended to a
    ring of capacity 3 (starting from 1 frame), incremental pyramid. Ring
    contents must match the oracle's cache bit for bit, and each step's
    attention must match a from-scratch oracle pass."""
    w = dataclasses.replace(RAGGED, history_frames=1, history_capacity=3, batch=2)
    x = synth.attention_inputs(w, BF16)
    plan = make_plan(w, BF16)
    dx = device_inputs(x, w.history_capacity)
    bind(plan, dx)
    hist = ostream.History(synth.to_f64(x["k_hist"]), synth.to_f64(x["v_hist"]), w.history_capacity)
    G = w.grid_h * w.grid_w
    for step in range(6):
        kv = synth.step_kv(w, 1000 + step, BF16)
        dkv = {k: v.cuda() for k, v in kv.items()}
        plan.kv_resample(dkv["k_win"], dkv["v_win"],
                         msf().MSF_RESAMPLE_FULL if step == 0 else msf().MSF_RESAMPLE_WINDOW_ONLY)
        out = torch.empty_like(dkv["q"])
        plan.mssa_forward(dkv["q"], dkv["k_win"], dkv["v_win"], out)
        hk, hv = hist.frames()
        ref = omssa.mssa_forward(synth.to_f64(kv["q"]), synth.to_f64(kv["k_win"]),
                                 synth.to_f64(kv["v_win"]), synth.to_f64(x["k_sink"]),
                                 synth.to_f64(x["v_sink"]), hk, hv, w.scales, w.grid_h, w.grid_w)
        mx, mean = err_stats(out, ref)
        assert mx <= BF16_MAX and mean <= BF16_MEAN, (step, mx, mean)
        slot = plan.info.history_next_slot
        plan.history_append(dkv["k_win"], dkv["v_win"])
        s2 = hist.append(synth.to_f64(kv["k_win"][:, :G]), synth.to_f64(kv["v_win"][:, :G]))
        assert slot == s2
        torch.cuda.synchronize()
        n = hist.count
        assert plan.info.history_count == n
        assert np.array_equal(dx["k_hist"][:, :n].double().cpu().numpy(), hist.k[:, :n])
        assert np.array_equal(dx["v_hist"][:, :n].double().cpu().numpy(), hist.v[:, :n])
    assert plan.device_status() == msf().MSF_OK


# ----------------------------------------------------------------- MSP

def _msp_plan(w, dtype, embed):
    plan = make_plan(w, dtype, embed=embed)
    x = synth.attention_inputs(w, dtype)
    dx = device_inputs(x, w.history_capacity)
    ws = bind(plan, dx)
    return plan, ws


@pytest.mark.parametrize("dtype", [BF16, F32], ids=["bf16", "f32"])
def test_patchify_unpatchify_raw_bit_exact(dtype):
    w = dataclasses.replace(synth.LAYER_480P, batch=2, heads=2)
    plan, _ = _msp_plan(w, dtype, False)
    m = synth.msp_inputs(w, dtype, embed_dim=0)
    lat = m["latent"].cuda()
    C, Hl, Wl = w.latent_channels, w.grid_h * w.patch, w.grid_w * w.patch
    raw = torch.empty((w.batch, w.T, C * Hl * Wl), dtype=dtype, device="cuda")
    plan.patchify(lat, None, raw)
    back = torch.empty((w.batch, C, Hl, Wl), dtype=dtype, device="cuda")
    torch.cuda.synchronize()
    lat64 = synth.to_f64(m["latent"])
    for l, s in enumerate(w.scales):
        P = w.patch * s
        ref = omsp.patchify(lat64[:, l], P).reshape(w.batch, -1)
        assert np.array_equal(raw[:, l].double().cpu().numpy(), ref)
        plan.unpatchify(l, raw, None, back)
        torch.cuda.synchronize()
        assert torch.equal(back.cpu(), m["latent"][:, l])


@pytest.mark.parametrize("shared", [True, False], ids=["tier_weights", "per_position_weights"])
def test_patchify_embed_and_unpatchify_deembed(shared):
    w = dataclasses.replace(synth.LAYER_480P, batch=2, heads=12)
    plan, _ = _msp_plan(w, BF16, True)
    m = synth.msp_inputs(w, BF16)
    lat = m["latent"].cuda()
    E = w.embed_dim
    N = plan.info.n_tokens
    if shared:
        tiers = {s: m["w_tier"][s].t().contiguous().cuda() for s in set(w.scales)}  # [E, C*P^2]
        w_tier = [tiers[s] for s in w.scales]
    else:
        w_tier = [m["w_tier"][s].t().contiguous().cuda() for s in w.scales]
    tok = torch.empty((w.batch, N, E), dtype=BF16, device="cuda")
    plan.patchify(lat, w_tier, tok)
    torch.cuda.synchronize()
    tiers = {s: synth.to_f64(m["w_tier"][s]) for s in set(w.scales)}
    ref = omsp.patchify_window(synth.to_f64(m["latent"]), w.scales, w.patch, tiers)
    got = tok.double().cpu().numpy()
    err = np.abs(got - ref)
    assert err.max() <= 2.0 ** -7 * np.abs(ref).max() + 1e-3, err.max()
    # de-embed the head state back to a latent: [C*P^2, E] weight
    w_out = m["w_out"].t().contiguous().cuda()
    lat_out = torch.empty((w.batch, w.latent_channels, w.grid_h * w.patch, w.grid_w * w.patch),
                          dtype=BF16, device="cuda")
    plan.unpatchify(0, tok, w_out, lat_out)
    torch.cuda.synchronize()
    n0 = plan.info.state_tokens[0]
    ref_lat = omsp.unpatchify_state(synth.to_f64(tok[:, :n0].cpu()), w.patch, w.latent_channels,
                                    w.grid_h * w.patch, w.grid_w * w.patch, synth.to_f64(m["w_out"]))
    e2 = np.abs(lat_out.double().cpu().numpy() - ref_lat)
    assert e2.max() <= 2.0 ** -7 * np.abs(ref_lat).max() + 1e-3, e2.max()


# ------------------------------------------------- full-size configurations

def test_streaming_rollout_480p_b4():
    """The B=4 streaming rollout at its real shapes: history starts at 2 fine
    frames, grows to the capacity of 4, then evicts the oldest; the sink stays
    fixed. Five steps cover the growth and two replacements. Each step's
    attention (one sampled head per step) matches a from-scratch oracle pass
    over the oracle's own cache, and the ring matches it bit for bit."""
    w = synth.STREAM_480P
    x = synth.attention_inputs(w, BF16)
    plan = make_plan(w, BF16)
    dx = device_inputs(x, w.history_capacity)
    bind(plan, dx)
    hist = ostream.History(synth.to_f64(x["k_hist"]), synth.to_f64(x["v_hist"]), w.history_capacity)
    G = w.grid_h * w.grid_w
    for step in range(5):
        kv = synth.step_kv(w, 4000 + step, BF16)
        dkv = {k: v.cuda() for k, v in kv.items()}
        plan.kv_resample(dkv["k_win"], dkv["v_win"],
                         msf().MSF_RESAMPLE_FULL if step == 0 else msf().MSF_RESAMPLE_WINDOW_ONLY)
        out = torch.empty_like(dkv["q"])
        plan.mssa_forward(dkv["q"], dkv["k_win"], dkv["v_win"], out)
        heads = [(5 * step) % w.heads]
        hk, hv = hist.frames()
        ref = omssa.mssa_forward(synth.to_f64(kv["q"]), synth.to_f64(kv["k_win"]), synth.to_f64(kv["v_win"]),
                                 synth.to_f64(x["k_sink"]), synth.to_f64(x["v_sink"]), hk, hv, w.scales,
                                 w.grid_h, w.grid_w, heads=heads)
        mx, mean = err_stats(out, ref, heads=heads)
        assert mx <= BF16_MAX and mean <= BF16_MEAN, (step, mx, mean)
        plan.history_append(dkv["k_win"], dkv["v_win"])
        hist.append(synth.to_f64(kv["k_win"][:, :G]), synth.to_f64(kv["v_win"][:, :G]))
        torch.cuda.synchronize()
        n = hist.count
        assert plan.info.history_count == n
        assert np.array_equal(dx["k_hist"][:, :n].double().cpu().numpy(), hist.k[:, :n])
        assert np.array_equal(dx["v_hist"][:, :n].double().cpu().numpy(), hist.v[:, :n])
    assert hist.count == w.history_capacity
    assert plan.device_status() == msf().MSF_OK


@pytest.mark.parametrize("layer", [0, 29])
def test_window_pass_layer(layer):
    """One layer of the 30-layer window pass (q/k/v of std 0.5, layer seed
    100 + l): MSP embedding of the five states, MSSA (sampled heads) and the
    de-embedding + unpatchify of the head state, each against the oracle."""
    w = synth.PASS_480P
    seed = w.seed + layer
    x = synth.attention_inputs(w, BF16, seed=seed)
    m = synth.msp_inputs(w, BF16, seed=seed)
    plan = make_plan(w, BF16, embed=True)
    dx = device_inputs(x, w.history_capacity)
    bind(plan, dx)
    N, E = plan.info.n_tokens, w.embed_dim
    tiers = {s: m["w_tier"][s].t().contiguous().cuda() for s in set(w.scales)}
    tok = torch.empty((w.batch, N, E), dtype=BF16, device="cuda")
    plan.patchify(m["latent"].cuda(), [tiers[s] for s in w.scales], tok)
    plan.kv_resample(dx["k_win"], dx["v_win"])
    out = torch.empty_like(dx["q"])
    plan.mssa_forward(dx["q"], dx["k_win"], dx["v_win"], out)
    w_out = m["w_out"].t().contiguous().cuda()
    lat_out = torch.empty((w.batch, w.latent_channels, w.grid_h * w.patch, w.grid_w * w.patch),
                          dtype=BF16, device="cuda")
    plan.unpatchify(0, out.view(w.batch, N, E), w_out, lat_out)
    torch.cuda.synchronize()
    assert plan.device_status() == msf().MSF_OK
    ref_tok = omsp.patchify_window(synth.to_f64(m["latent"]), w.scales, w.patch,
                                   {s: synth.to_f64(m["w_tier"][s]) for s in set(w.scales)})
    e = np.abs(tok.double().cpu().numpy() - ref_tok)
    assert e.max() <= 2.0 ** -7 * np.abs(ref_tok).max() + 1e-3, e.max()
    heads = [layer % w.heads]
    ref = oracle_mssa(x, w, 0, heads=heads)
    mx, mean = err_stats(out, ref, heads=heads)
    assert mx <= BF16_MAX and mean <= BF16_MEAN, (mx, mean)
    n0 = plan.info.state_tokens[0]
    ref_lat = omsp.unpatchify_state(synth.to_f64(out.view(w.batch, N, E)[:, :n0].cpu()), w.patch,
                                    w.latent_channels, w.grid_h * w.patch, w.grid_w * w.patch,
                                    synth.to_f64(m["w_out"]))
    e2 = np.abs(lat_out.double().cpu().numpy() - ref_lat)
    assert e2.max() <= 2.0 ** -7 * np.abs(ref_lat).max() + 1e-3, e2.max()
