"""GPU parity of the one-launch resample + attention (msf_mssa_forward_resample,
Eq. 4 with its Subsample built in the attention kernel's prologue): the
output, the pyramid and the staged head must equal, bit for bit, those of
msf_kv_resample followed by msf_mssa_forward, whose own parity against the
oracle the other GPU tests check; launches in a row and CUDA graph replays
check that the launch's pyramid counts reset themselves. One case is also
checked against the oracle directly.
"""
import dataclasses

import pytest
import torch

from paper_2607_20940_gb300 import synth

from helpers import BF16, F32, bind, device_inputs, err_stats, make_plan, msf, oracle_mssa

pytestmark = pytest.mark.gpu

SMALL3 = synth.Workload("fr_t4_12x20", 4, (1, 1, 2, 4), 12, 20, 3, 128, 200, 2, 3, 2, 41)
RAGGED = synth.Workload("fr_ragged_t3_10x14_d64", 3, (1, 2, 2), 10, 14, 2, 64, 37, 1, 1, 1, 43)
CASES = [
    ("tiny", synth.TINY),
    ("small3", SMALL3),
    ("ragged_d64", RAGGED),
    ("layer_480p", synth.LAYER_480P),
    ("stream_b4", dataclasses.replace(synth.STREAM_480P, history_frames=3)),
    ("three_scale", synth.THREE_SCALE),
    ("chunked", synth.CHUNKED_480P),
    ("max_states", synth.Workload("fr_max_states_t16", 16, (1, 1, 2, 2, 4, 4, 8, 8) + (16,) * 8, 32, 48, 2,
                                  64, 40, 2, 3, 2, 45)),
]
STRIDED_CASES = [("small3", SMALL3), ("layer_480p", synth.LAYER_480P), ("three_scale", synth.THREE_SCALE)]


def _pyramid(plan, ws, w):
    info = plan.info
    n = w.batch * info.pyramid_tokens * w.heads * w.head_dim * 2
    k0, v0 = info.pyramid_k_offset, info.pyramid_v_offset
    return ws[k0:k0 + n].clone(), ws[v0:v0 + n].clone()


def _two_calls(plan, dx, flags):
    out = torch.empty_like(dx["q"])
    plan.kv_resample(dx["k_win"], dx["v_win"], flags)
    plan.mssa_forward(dx["q"], dx["k_win"], dx["v_win"], out)
    return out


def _one_launch(plan, dx, flags):
    out = torch.empty_like(dx["q"])
    plan.mssa_forward_resample(dx["q"], dx["k_win"], dx["v_win"], out, flags)
    return out


@pytest.mark.parametrize("name,w", CASES, ids=[c[0] for c in CASES])
@pytest.mark.parametrize("flags", ["full", "window"])
def test_one_launch_equals_resample_then_forward(name, w, flags):
    m = msf()
    fl = m.MSF_RESAMPLE_FULL if flags == "full" else m.MSF_RESAMPLE_WINDOW_ONLY
    x = synth.attention_inputs(w)
    dx = device_inputs(x, w.history_capacity)
    plan = make_plan(w)
    ws = bind(plan, dx)
    # the history part of the pyramid must exist before a window-only pass
    plan.kv_resample(dx["k_win"], dx["v_win"], m.MSF_RESAMPLE_FULL)
    ref = _two_calls(plan, dx, fl)
    pk_ref, pv_ref = _pyramid(plan, ws, w)
    # a pyramid built from other window K/V (the history part stays right):
    # the one launch has to rebuild every window part it reads
    plan.kv_resample(dx["v_win"], dx["k_win"], m.MSF_RESAMPLE_FULL)
    torch.cuda.synchronize()
    stale_k, _ = _pyramid(plan, ws, w)
    assert not torch.equal(stale_k, pk_ref)
    got = _one_launch(plan, dx, fl)
    torch.cuda.synchronize()
    assert plan.device_status() == m.MSF_OK
    pk, pv = _pyramid(plan, ws, w)
    assert torch.equal(pk, pk_ref) and torch.equal(pv, pv_ref)
    assert torch.equal(got, ref)
    plan.close()


@pytest.mark.parametrize("name,w", STRIDED_CASES, ids=[c[0] for c in STRIDED_CASES])
def test_one_launch_strided_subsample(name, w):
    """The literal stride-2 reading of Subsample (top-left token of each
    block) through the one launch, against the two calls."""
    m = msf()
    x = synth.attention_inputs(w)
    dx = device_inputs(x, w.history_capacity)
    plan = make_plan(w, resample=m.MSF_RESAMPLE_STRIDED)
    ws = bind(plan, dx)
    ref = _two_calls(plan, dx, m.MSF_RESAMPLE_FULL)
    pk_ref, pv_ref = _pyramid(plan, ws, w)
    plan.kv_resample(dx["v_win"], dx["k_win"], m.MSF_RESAMPLE_FULL)
    got = _one_launch(plan, dx, m.MSF_RESAMPLE_FULL)
    torch.cuda.synchronize()
    assert plan.device_status() == m.MSF_OK
    pk, pv = _pyramid(plan, ws, w)
    assert torch.equal(pk, pk_ref) and torch.equal(pv, pv_ref)
    assert torch.equal(got, ref)
    plan.close()


def test_one_launch_matches_oracle_tiny():
    m = msf()
    w = synth.TINY
    x = synth.attention_inputs(w)
    dx = device_inputs(x, w.history_capacity)
    plan = make_plan(w)
    bind(plan, dx)
    got = _one_launch(plan, dx, m.MSF_RESAMPLE_FULL)
    torch.cuda.synchronize()
    assert plan.device_status() == m.MSF_OK
    mx, mean = err_stats(got, oracle_mssa(x, w))
    assert mx <= 2e-2 and mean <= 2e-3, (mx, mean)
    plan.close()


def test_launches_in_a_row_and_graph_replays():
    """Each launch's counts reset at its end: five launches in a row with
    new window K/V, then a captured launch replayed on two more steps, each
    equal to the two-call path on the same inputs."""
    m = msf()
    w = synth.LAYER_480P
    x = synth.attention_inputs(w)
    dx = device_inputs(x, w.history_capacity)
    plan = make_plan(w)
    bind(plan, dx)
    plan.kv_resample(dx["k_win"], dx["v_win"], m.MSF_RESAMPLE_FULL)
    wo = m.MSF_RESAMPLE_WINDOW_ONLY
    for step in range(5):
        kv = {k: v.cuda() for k, v in synth.step_kv(w, 900 + step).items()}
        for k in ("q", "k_win", "v_win"):
            dx[k].copy_(kv[k])
        ref = _two_calls(plan, dx, wo)
        got = _one_launch(plan, dx, wo)
        torch.cuda.synchronize()
        assert plan.device_status() == m.MSF_OK
        assert torch.equal(got, ref), step
    out = torch.empty_like(dx["q"])
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.stream(s):
        plan.mssa_forward_resample(dx["q"], dx["k_win"], dx["v_win"], out, wo, stream=s)  # warm
        s.synchronize()
        with torch.cuda.graph(g, stream=s):
            plan.mssa_forward_resample(dx["q"], dx["k_win"], dx["v_win"], out, wo, stream=s)
    torch.cuda.current_stream().wait_stream(s)
    for step in range(2):
        kv = {k: v.cuda() for k, v in synth.step_kv(w, 950 + step).items()}
        for k in ("q", "k_win", "v_win"):
            dx[k].copy_(kv[k])
        torch.cuda.synchronize()
        g.replay()
        torch.cuda.synchronize()
        got = out.clone()
        ref = _two_calls(plan, dx, wo)
        torch.cuda.synchronize()
        assert plan.device_status() == m.MSF_OK
        assert torch.equal(got, ref), step
    plan.close()


FUSED = [
    ("small3", dataclasses.replace(SMALL3, history_frames=1)),
    ("layer_480p", synth.LAYER_480P),
    ("stream_b4", synth.STREAM_480P),
]


@pytest.mark.parametrize("name,w", FUSED, ids=[c[0] for c in FUSED])
def test_fused_append_rollout_stages_the_head(name, w):
    """fused_append: the one launch stages the head in the spare ring slot
    like msf_kv_resample does, and the fine group reads it from there after
    the launch's pooling count, over a rollout with commits that wraps the
    ring."""
    m = msf()
    x = synth.attention_inputs(w)

    def run(one):
        desc = m.make_desc(w.scales, w.grid_h, w.grid_w, w.heads, w.head_dim, w.sink_tokens,
                           w.history_frames, history_capacity=w.history_capacity, batch=w.batch,
                           fused_append=1)
        plan = m.Plan(desc)
        B, G, H, D = w.batch, w.fine_tokens, w.heads, w.head_dim
        ring = {}
        for k in ("k_hist", "v_hist"):
            r = torch.zeros((B, w.history_capacity + 1, G, H, D), dtype=BF16, device="cuda")
            r[:, :w.history_frames] = x[k].cuda()
            ring[k] = r
        sink = {k: x[k].cuda() for k in ("k_sink", "v_sink")}
        ws = plan.workspace()
        plan.bind(ws, sink["k_sink"], sink["v_sink"], ring["k_hist"], ring["v_hist"])
        outs = []
        for step in range(w.history_capacity + 2):
            kv = {k: v.cuda() for k, v in synth.step_kv(w, 700 + step).items()}
            fl = m.MSF_RESAMPLE_FULL if step == 0 else m.MSF_RESAMPLE_WINDOW_ONLY
            out = torch.empty_like(kv["q"])
            if one:
                plan.mssa_forward_resample(kv["q"], kv["k_win"], kv["v_win"], out, fl)
            else:
                plan.kv_resample(kv["k_win"], kv["v_win"], fl)
                plan.mssa_forward(kv["q"], kv["k_win"], kv["v_win"], out)
            plan.history_commit()
            outs.append(out)
        torch.cuda.synchronize()
        assert plan.device_status() == m.MSF_OK
        res = [o.cpu() for o in outs], ring["k_hist"].cpu(), ring["v_hist"].cpu()
        plan.close()
        return res

    o1, k1, v1 = run(True)
    o2, k2, v2 = run(False)
    for a, b in zip(o1, o2):
        assert torch.equal(a, b)
    assert torch.equal(k1, k2) and torch.equal(v1, v2)


def test_fp32_plan_runs_the_two_calls():
    m = msf()
    w = synth.TINY
    x = synth.attention_inputs(w, F32)
    dx = device_inputs(x, w.history_capacity)
    plan = make_plan(w, F32)
    bind(plan, dx)
    got = _one_launch(plan, dx, m.MSF_RESAMPLE_FULL)
    ref = _two_calls(plan, dx, m.MSF_RESAMPLE_FULL)
    torch.cuda.synchronize()
    assert plan.device_status() == m.MSF_OK
    assert torch.equal(got, ref)
    plan.close()
