"""GPU parity of the MSSA gradient (msf_mssa_forward_lse + msf_mssa_backward)
against the fp64 oracle (oracle/mssa_bwd.py), on the same seeded q/k/v and a
seeded dout.

Bounds. bf16 plans: the gradients are rounded once to bf16 (relative
2^-9) after fp32 accumulation, and the backward rebuilds P from the forward's
bf16 output through delta = rowsum(dout * out); max |err| <= 1e-2 * max|ref|
and mean |err| <= 1e-3 * max|ref| per tensor. fp32 plans: 1e-4 * max|ref|.
The row log-sum-exp is checked to 2e-3 (bf16) / 1e-5 (fp32) absolute.
"""
import dataclasses

import numpy as np
import pytest
import torch

from oracle import mssa as omssa
from oracle import mssa_bwd as obwd
from paper_2607_20940_gb300 import synth

from helpers import BF16, F32, bind, device_inputs, make_plan, msf

pytestmark = pytest.mark.gpu

RAGGED = synth.Workload("ragged_t4_12x20", 4, (1, 1, 2, 4), 12, 20, 3, 128, 200, 2, 3, 2, 21)
RAGGED64 = dataclasses.replace(RAGGED, name="ragged_d64", head_dim=64, scales=(1, 2, 2, 4), seed=22)
COARSE_ONLY = synth.Workload("coarse_only", 3, (2, 2, 4), 16, 24, 2, 128, 37, 1, 1, 1, 23)
# 16 window states in five query groups: a fine token's gradient gathers
# entries from up to five groups (odd and even counts in the gather)
MAX_STATES = synth.Workload("max_states_t16", 16, (1, 1, 2, 2, 4, 4, 8, 8) + (16,) * 8, 32, 48, 2, 64,
                            40, 2, 3, 1, 26)


def _dout(w, dtype, shape):
    g = torch.Generator().manual_seed(w.seed + 555)
    return torch.randn(*shape, generator=g, dtype=torch.float32).to(dtype)


def _run(w, dtype, mode=0, fused=False):
    x = synth.attention_inputs(w, dtype)
    m = msf()
    if fused:
        plan = m.Plan(m.make_desc(w.scales, w.grid_h, w.grid_w, w.heads, w.head_dim, w.sink_tokens,
                                  w.history_frames, history_capacity=w.history_capacity,
                                  batch=w.batch,
                                  dtype=m.MSF_DTYPE_BF16 if dtype == BF16 else m.MSF_DTYPE_F32,
                                  resample=mode, frames_per_state=w.frames, fused_append=1))
        dx = device_inputs(x, w.history_capacity + 1)
    else:
        plan = make_plan(w, dtype, resample=mode)
        dx = device_inputs(x, w.history_capacity)
    bind(plan, dx)
    dout = _dout(w, dtype, x["q"].shape)
    dd = dout.cuda()
    out = torch.empty_like(dx["q"])
    B, N, H = dx["q"].shape[0], dx["q"].shape[1], w.heads
    lse = torch.full((B, H, N), float("nan"), dtype=torch.float32, device="cuda")
    plan.kv_resample(dx["k_win"], dx["v_win"])
    plan.mssa_forward_lse(dx["q"], dx["k_win"], dx["v_win"], out, lse)
    g = {k: torch.full_like(dx["q"], float("nan")) for k in ("dq", "dk", "dv")}
    ws = plan.backward_workspace()
    plan.mssa_backward(dx["q"], dx["k_win"], dx["v_win"], out, dd, lse, g["dq"], g["dk"], g["dv"], ws)
    torch.cuda.synchronize()
    assert plan.device_status() == m.MSF_OK
    return x, dout, out, lse, g, plan


def _check(x, dout, lse, g, w, dtype, mode, heads=None):
    f = synth.to_f64
    hsel = list(range(w.heads)) if heads is None else heads
    sl = lambda a: a[..., hsel, :]
    ref = obwd.mssa_backward(sl(f(x["q"])), sl(f(x["k_win"])), sl(f(x["v_win"])),
                             sl(f(x["k_sink"])), sl(f(x["v_sink"])), sl(f(x["k_hist"])),
                             sl(f(x["v_hist"])), sl(f(dout)), w.scales, w.grid_h, w.grid_w,
                             mode, frames=w.frames)
    lref = omssa.mssa_lse(f(x["q"]), f(x["k_win"]), f(x["k_sink"]), f(x["k_hist"]), w.scales,
                          w.grid_h, w.grid_w, mode, heads=hsel, frames=w.frames)
    le = np.abs(lse.double().cpu().numpy()[:, hsel] - lref[:, hsel]).max()
    assert le <= (2e-3 if dtype == BF16 else 1e-5), le
    rel_max, rel_mean = (1e-2, 1e-3) if dtype == BF16 else (1e-4, 1e-5)
    for name, key in (("dq", "dq"), ("dk", "dk_win"), ("dv", "dv_win")):
        got = g[name].double().cpu().numpy()[:, :, hsel]
        r = ref[key]
        scale = np.abs(r).max()
        e = np.abs(got - r)
        assert np.isfinite(got).all(), name
        assert e.max() <= rel_max * scale and e.mean() <= rel_mean * scale, (name, e.max(), e.mean(), scale)


@pytest.mark.parametrize("w", [synth.TINY, RAGGED, RAGGED64, COARSE_ONLY, synth.CHUNKED_SMALL, MAX_STATES],
                         ids=lambda w: w.name)
@pytest.mark.parametrize("mode", [0, 1], ids=["avg", "strided"])
def test_backward_bf16(w, mode):
    x, dout, out, lse, g, _ = _run(w, BF16, mode)
    _check(x, dout, lse, g, w, BF16, mode)


@pytest.mark.parametrize("w", [synth.TINY, RAGGED], ids=lambda w: w.name)
def test_backward_fp32(w):
    x, dout, out, lse, g, _ = _run(w, F32, 0)
    _check(x, dout, lse, g, w, F32, 0)


def test_backward_fused_append_layout():
    """With the head staged in the ring's spare slot its gradient comes back
    from that slot (and its pooled level from the ring part of the pyramid)."""
    w = dataclasses.replace(RAGGED, history_frames=1, history_capacity=2, seed=41)
    x, dout, out, lse, g, _ = _run(w, BF16, 0, fused=True)
    _check(x, dout, lse, g, w, BF16, 0)


def test_backward_480p_sampled_heads():
    """Full 480p layer (all heads computed on the GPU; the oracle checks two)."""
    w = synth.LAYER_480P
    x, dout, out, lse, g, _ = _run(w, BF16, 0)
    _check(x, dout, lse, g, w, BF16, 0, heads=[0, 7])


@pytest.mark.parametrize("w", [RAGGED, RAGGED64], ids=lambda w: w.name)
def test_backward_tensor_core_matches_cuda_core(w):
    """bf16 plans: the tcgen05 backward against the fp32 CUDA-core backward on
    the same inputs (both checked against the oracle above)."""
    x, dout, out, lse, g, plan = _run(w, BF16, 0)
    dx = device_inputs(x, w.history_capacity)
    bind(plan, dx)
    plan.kv_resample(dx["k_win"], dx["v_win"])
    h = {k: torch.full_like(g["dq"], float("nan")) for k in ("dq", "dk", "dv")}
    plan.mssa_backward_simt(dx["q"], dx["k_win"], dx["v_win"], out, dout.cuda(), lse, h["dq"], h["dk"],
                            h["dv"], plan.backward_workspace())
    torch.cuda.synchronize()
    for k in ("dq", "dk", "dv"):
        a, b = g[k].float(), h[k].float()
        scale = b.abs().max().item()
        assert (a - b).abs().max().item() <= 1e-2 * scale, k


def test_backward_three_scale_sampled_head():
    """Three query groups (g = 1, 2, 4) at the 48x80 shapes: every pooled
    level's adjoint at full size; the oracle checks one head."""
    w = synth.THREE_SCALE
    x, dout, out, lse, g, _ = _run(w, BF16, 0)
    _check(x, dout, lse, g, w, BF16, 0, heads=[5])
