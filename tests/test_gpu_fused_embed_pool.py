"""The MSP embedding and the K/V pyramid in one launch (msf_patchify_resample)
against the two separate calls (msf_patchify with tier weights, then
msf_kv_resample): the tokens, both pyramids, the staged history head and the
attention that reads them must be bit for bit the same, because the pooling
CTAs run the same per-thread arithmetic as the pool kernel and the two parts
touch disjoint buffers."""
import dataclasses

import pytest
import torch

from paper_2607_20940_gb300 import synth

from helpers import BF16, msf

pytestmark = pytest.mark.gpu


def _run(w, fused_append, flags, fused_call, seed=3):
    m = msf()
    plan = m.Plan(m.make_desc(w.scales, w.grid_h, w.grid_w, w.heads, w.head_dim, w.sink_tokens,
                              w.history_frames, w.history_capacity, batch=w.batch,
                              latent_channels=w.latent_channels, patch=w.patch, embed_dim=w.embed_dim,
                              frames_per_state=w.frames, fused_append=fused_append))
    x = synth.attention_inputs(w, BF16, seed=seed)
    mi = synth.msp_inputs(w, BF16)
    d = {k: v.cuda() for k, v in x.items() if k not in ("k_hist", "v_hist")}
    slots = w.history_capacity + (1 if fused_append else 0)
    for k in ("k_hist", "v_hist"):
        ring = torch.zeros((w.batch, max(slots, 1)) + tuple(x[k].shape[2:]), dtype=BF16, device="cuda")
        ring[:, :w.history_frames] = x[k].cuda()
        d[k] = ring
    ws = plan.workspace()
    plan.bind(ws, d["k_sink"], d["v_sink"], d["k_hist"], d["v_hist"])
    if flags == m.MSF_RESAMPLE_WINDOW_ONLY:  # the history part is kept by the appends
        plan.kv_resample(d["k_win"], d["v_win"], m.MSF_RESAMPLE_FULL)
    lat = mi["latent"].cuda()
    tiers = {s: mi["w_tier"][s].t().contiguous().cuda() for s in set(w.scales)}
    w_tier = [tiers[s] for s in w.scales]
    tok = torch.full((w.batch, plan.info.n_tokens, w.embed_dim), float("nan"), dtype=BF16, device="cuda")
    if fused_call:
        plan.patchify_resample(lat, w_tier, tok, d["k_win"], d["v_win"], flags)
    else:
        plan.patchify(lat, w_tier, tok)
        plan.kv_resample(d["k_win"], d["v_win"], flags)
    out = torch.empty_like(d["q"])
    plan.mssa_forward(d["q"], d["k_win"], d["v_win"], out)
    torch.cuda.synchronize()
    assert plan.device_status() == m.MSF_OK
    info = plan.info
    pyr = int(info.pyramid_v_offset - info.pyramid_k_offset)
    res = {"tok": tok.cpu(), "out": out.cpu(), "ring_k": d["k_hist"].cpu(), "ring_v": d["v_hist"].cpu(),
           "pyr": ws[int(info.pyramid_k_offset):int(info.pyramid_k_offset) + 2 * pyr].cpu()}
    plan.close()
    return res


@pytest.mark.parametrize("name,w,fused_append,window_only", [
    ("480p_fused_append", synth.LAYER_480P, 1, True),
    ("480p_full", synth.LAYER_480P, 0, False),
    ("480p_b4_stream", synth.STREAM_480P, 1, True),
    ("chunked_small", synth.CHUNKED_SMALL, 0, False),
    ("three_scale_embed", dataclasses.replace(synth.THREE_SCALE, heads=4, embed_dim=512), 0, False),
])
def test_fused_embed_pool_matches_separate_calls(name, w, fused_append, window_only):
    m = msf()
    flags = m.MSF_RESAMPLE_WINDOW_ONLY if window_only else m.MSF_RESAMPLE_FULL
    a = _run(w, fused_append, flags, fused_call=False)
    b = _run(w, fused_append, flags, fused_call=True)
    for k in ("tok", "pyr", "ring_k", "ring_v", "out"):
        assert torch.equal(a[k], b[k]), (name, k)
    assert torch.isfinite(b["tok"].float()).all()


def test_fused_embed_pool_with_more_runs_than_one_launch_holds():
    """Six positions with six distinct tier-weight tensors make six runs:
    the embedding goes out in two launches (at most four runs each) and the
    pyramid jobs ride with the first; the result must still equal the two
    separate calls bit for bit."""
    m = msf()
    w = dataclasses.replace(synth.THREE_SCALE, heads=2, embed_dim=256)
    plan = m.Plan(m.make_desc(w.scales, w.grid_h, w.grid_w, w.heads, w.head_dim, w.sink_tokens,
                              w.history_frames, w.history_capacity, batch=w.batch,
                              latent_channels=w.latent_channels, patch=w.patch, embed_dim=w.embed_dim))
    x = synth.attention_inputs(w, BF16, seed=5)
    mi = synth.msp_inputs(w, BF16)
    d = {k: v.cuda() for k, v in x.items()}
    ws = plan.workspace()
    plan.bind(ws, d["k_sink"], d["v_sink"], d["k_hist"], d["v_hist"])
    lat = mi["latent"].cuda()
    # one distinct copy of the tier weight per position
    w_tier = [mi["w_tier"][s].t().contiguous().cuda().clone() for s in w.scales]
    info = plan.info
    pyr = int(info.pyramid_v_offset - info.pyramid_k_offset)
    outs = []
    for fused_call in (False, True):
        tok = torch.full((w.batch, info.n_tokens, w.embed_dim), float("nan"), dtype=BF16, device="cuda")
        ws[int(info.pyramid_k_offset):int(info.pyramid_k_offset) + 2 * pyr].zero_()
        if fused_call:
            plan.patchify_resample(lat, w_tier, tok, d["k_win"], d["v_win"], m.MSF_RESAMPLE_FULL)
        else:
            plan.patchify(lat, w_tier, tok)
            plan.kv_resample(d["k_win"], d["v_win"], m.MSF_RESAMPLE_FULL)
        torch.cuda.synchronize()
        assert plan.device_status() == m.MSF_OK
        outs.append((tok.cpu(), ws[int(info.pyramid_k_offset):int(info.pyramid_k_offset) + 2 * pyr].cpu()))
    assert torch.equal(outs[0][0], outs[1][0])
    assert torch.equal(outs[0][1], outs[1][1])
    assert torch.isfinite(outs[1][0].float()).all()
