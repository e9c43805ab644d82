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


@pytest.mark.parametrize("fused", [False, True], ids=["append", "fused"])
def test_checkpoint_resume_rollout(fused):
    """A rollout checkpointed after three steps (ring tensors + the ring's
    host state) and resumed in a fresh plan gives the same outputs, bit for
    bit, as the uninterrupted rollout (the restored plan rebuilds its pyramid
    with a full resample)."""
    m = msf()
    w = dataclasses.replace(BASE, history_frames=1, history_capacity=2, batch=2, seed=51)
    x = synth.attention_inputs(w, BF16)
    B, G, H, D = w.batch, w.fine_tokens, w.heads, w.head_dim
    slots = w.history_capacity + (1 if fused else 0)

    def new_plan():
        return m.Plan(m.make_desc(w.scales, w.grid_h, w.grid_w, w.heads, w.head_dim, w.sink_tokens,
                                  w.history_frames, history_capacity=w.history_capacity,
                                  batch=w.batch, fused_append=int(fused)))

    def ring_from(src):
        r = torch.zeros((B, slots, G, H, D), dtype=BF16, device="cuda")
        r[:, :src.shape[1]] = src
        return r

    sink = {k: x[k].cuda() for k in ("k_sink", "v_sink")}
    ring = {k: ring_from(x[k].cuda()) for k in ("k_hist", "v_hist")}
    a = new_plan()
    a.bind(a.workspace(), sink["k_sink"], sink["v_sink"], ring["k_hist"], ring["v_hist"])

    def step(plan, kv, first):
        plan.kv_resample(kv["k_win"], kv["v_win"], m.MSF_RESAMPLE_FULL if first else m.MSF_RESAMPLE_WINDOW_ONLY)
        out = torch.empty_like(kv["q"])
        plan.mssa_forward(kv["q"], kv["k_win"], kv["v_win"], out)
        if fused:
            plan.history_commit()
        else:
            plan.history_append(kv["k_win"], kv["v_win"])
        return out

    kvs = [{k: v.cuda() for k, v in synth.step_kv(w, 8000 + i, BF16).items()} for i in range(6)]
    for i in range(3):
        step(a, kvs[i], i == 0)
    torch.cuda.synchronize()
    # checkpoint: the ring buffers and the ring's host state
    saved = {k: v.clone() for k, v in ring.items()}
    st = a.history_state()
    b = new_plan()
    b.bind(b.workspace(), sink["k_sink"], sink["v_sink"], saved["k_hist"], saved["v_hist"])
    b.set_history_state(st)
    assert b.info.history_count == a.info.history_count
    for i in range(3, 6):
        oa = step(a, kvs[i], False)
        ob = step(b, kvs[i], i == 3)
        torch.cuda.synchronize()
        assert torch.equal(oa, ob), i
    assert torch.equal(ring["k_hist"], saved["k_hist"]) and torch.equal(ring["v_hist"], saved["v_hist"])
    assert a.device_status() == m.MSF_OK and b.device_status() == m.MSF_OK
