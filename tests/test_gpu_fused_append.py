"""GPU parity of the fused history update (Algorithm 1's KV update folded
into the K/V resample): the head state is staged in the ring's spare slot by
the same launch that pools it, attention reads it from there, and a host-only
commit makes it a history frame. Every step's attention must match a fresh
oracle pass over the oracle's own FIFO cache, and the live ring slots must
hold exactly the oracle's live frames, bit for bit.
"""
import dataclasses

import numpy as np
import pytest
import torch

from oracle import mssa as omssa
from oracle import stream as ostream
from paper_2607_20940_gb300 import synth

from helpers import BF16, F32, err_stats, msf

pytestmark = pytest.mark.gpu

BF16_MAX, BF16_MEAN, F32_MAX = 2e-2, 2e-3, 1e-4

BASE = synth.Workload("fused_t4_12x20", 4, (1, 1, 2, 4), 12, 20, 3, 128, 200, 1, 3, 2, 31)


def _plan(w, dtype, mode):
    m = msf()
    return m.Plan(m.make_desc(w.scales, w.grid_h, w.grid_w, w.heads, w.head_dim, w.sink_tokens,
                              w.history_frames, history_capacity=w.history_capacity,
                              batch=w.batch,
                              dtype=m.MSF_DTYPE_BF16 if dtype == BF16 else m.MSF_DTYPE_F32,
                              resample=mode, frames_per_state=w.frames, fused_append=1))


def _rollout(w, dtype, mode, steps, heads=None, seed0=7000):
    x = synth.attention_inputs(w, dtype)
    plan = _plan(w, dtype, mode)
    B, G, H, D = w.batch, w.fine_tokens, w.heads, w.head_dim
    ring = {}
    for k in ("k_hist", "v_hist"):
        r = torch.zeros((B, w.history_capacity + 1, G, H, D), dtype=dtype, device="cuda")
        r[:, :w.history_frames] = x[k].cuda()
        ring[k] = r
    sink = {k: x[k].cuda() for k in ("k_sink", "v_sink")}
    ws = plan.workspace()
    plan.bind(ws, sink["k_sink"], sink["v_sink"], ring["k_hist"], ring["v_hist"])
    hist = ostream.History(synth.to_f64(x["k_hist"]), synth.to_f64(x["v_hist"]), w.history_capacity)
    tol = (BF16_MAX, BF16_MEAN) if dtype == BF16 else (F32_MAX, F32_MAX)
    for step in range(steps):
        kv = synth.step_kv(w, seed0 + step, dtype)
        dkv = {k: v.cuda() for k, v in kv.items()}
        plan.kv_resample(dkv["k_win"], dkv["v_win"],
                         msf().MSF_RESAMPLE_FULL if step == 0 else msf().MSF_RESAMPLE_WINDOW_ONLY)
        out = torch.empty_like(dkv["q"])
        plan.mssa_forward(dkv["q"], dkv["k_win"], dkv["v_win"], out)
        hk, hv = hist.frames()
        hs = None if heads is None else [heads[step % len(heads)]]
        ref = omssa.mssa_forward(synth.to_f64(kv["q"]), synth.to_f64(kv["k_win"]),
                                 synth.to_f64(kv["v_win"]), synth.to_f64(x["k_sink"]),
                                 synth.to_f64(x["v_sink"]), hk, hv, w.scales, w.grid_h, w.grid_w,
                                 mode=mode, heads=hs, frames=w.frames)
        mx, mean = err_stats(out, ref, heads=hs)
        assert mx <= tol[0] and mean <= tol[1], (step, mx, mean)
        spare = plan.info.history_next_slot
        plan.history_commit()
        hist.append(synth.to_f64(kv["k_win"][:, :G]), synth.to_f64(kv["v_win"][:, :G]))
        torch.cuda.synchronize()
        # the staged head sits in the slot that was spare, bit for bit
        assert torch.equal(ring["k_hist"][:, spare].cpu(), kv["k_win"][:, :G])
        assert torch.equal(ring["v_hist"][:, spare].cpu(), kv["v_win"][:, :G])
        # live slots (all used slots but the new spare) hold the oracle's live frames
        n = hist.count
        assert plan.info.history_count == n
        used = list(range(min(n + 1, w.history_capacity + 1)))
        live = [s for s in used if s != plan.info.history_next_slot]
        assert len(live) == n
        got = ring["k_hist"][:, live].double().cpu().numpy()
        for f in range(n):
            hits = [i for i in range(n) if np.array_equal(got[:, i], hist.k[:, f])]
            assert len(hits) == 1, (step, f, hits)
    assert plan.device_status() == msf().MSF_OK


@pytest.mark.parametrize("mode", [0, 1], ids=["avg", "strided"])
def test_fused_append_rollout(mode):
    """Three levels (g = 1, 2, 4), history 1 growing to capacity 3, then
    evictions: seven steps."""
    _rollout(BASE, BF16, mode, steps=7)


def test_fused_append_rollout_fp32():
    _rollout(dataclasses.replace(BASE, seed=32), F32, 0, steps=5)


def test_fused_append_no_coarse_level():
    """All states fine: the head is staged by a plain copy job."""
    w = dataclasses.replace(BASE, name="fused_all_fine", scales=(1, 1, 1), history_frames=0,
                            history_capacity=2, seed=33)
    _rollout(w, BF16, 0, steps=4)


def test_fused_append_stride_8_head_copy():
    """Scale 8 is pooled by the generic path, so the head copy goes out as
    its own job in the same launch."""
    w = synth.Workload("fused_s8", 2, (1, 8), 16, 16, 2, 64, 17, 1, 2, 1, 34)
    _rollout(w, BF16, 0, steps=4)


def test_fused_append_chunked():
    w = dataclasses.replace(synth.CHUNKED_SMALL, history_frames=1, history_capacity=2, batch=2)
    _rollout(w, BF16, 0, steps=4)


def test_fused_append_streaming_480p_b4():
    """The streaming rollout's shapes (B = 4, history 2 -> capacity 4,
    sink fixed) with the fused update; one sampled head per step."""
    _rollout(synth.STREAM_480P, BF16, 0, steps=5, heads=[0, 5, 10, 3, 8])
