"""GPU failure paths and memory guards.

* A bounded device wait that nothing satisfies gives up, raises the TIMEOUT
  bit of the device status word, and leaves the context usable (no trap, no
  hang: the wait is bounded by a cycle count).
* Canaries: every output is written inside a larger buffer whose guard bands
  hold a pattern; the kernels must not touch the guards.
"""
import dataclasses

import numpy as np
import pytest
import torch

from paper_2607_20940_gb300 import synth

from helpers import BF16, bind, device_inputs, err_stats, make_plan, msf, oracle_mssa

pytestmark = pytest.mark.gpu

GUARD = 4096  # elements on each side
PATTERN = 0x7F7B  # a bf16 NaN pattern no kernel writes


def guarded(shape, dtype=BF16):
    n = int(np.prod(shape))
    buf = torch.empty(n + 2 * GUARD, dtype=dtype, device="cuda")
    buf.view(torch.int16).fill_(PATTERN)
    return buf, buf[GUARD:GUARD + n].view(shape)


def guards_intact(buf):
    g = buf.view(torch.int16)
    return bool((g[:GUARD] == PATTERN).all()) and bool((g[-GUARD:] == PATTERN).all())


def test_bounded_wait_timeout_is_reported_and_context_stays_usable():
    w = synth.TINY
    x = synth.attention_inputs(w, BF16)
    plan = make_plan(w, BF16)
    dx = device_inputs(x, w.history_capacity)
    bind(plan, dx)
    assert plan.device_status() == msf().MSF_OK
    plan.selftest_wait_timeout(200_000)  # ~0.1 ms of SM clock
    assert plan.device_status() == msf().MSF_ERR_TIMEOUT
    assert plan.device_status() == msf().MSF_OK  # read clears the word
    out = torch.empty_like(dx["q"])
    plan.kv_resample(dx["k_win"], dx["v_win"])
    plan.mssa_forward(dx["q"], dx["k_win"], dx["v_win"], out)
    assert plan.device_status() == msf().MSF_OK
    mx, mean = err_stats(out, oracle_mssa(x, w, 0))
    assert mx <= 2e-2 and mean <= 2e-3


def test_selftest_rejects_bad_arguments():
    plan = make_plan(synth.TINY, BF16)
    with pytest.raises(Exception):
        plan.selftest_wait_timeout(0)
    with pytest.raises(Exception):
        plan.selftest_wait_timeout(200_000)  # not bound yet


def test_canaries_around_every_output():
    w = dataclasses.replace(synth.LAYER_480P, heads=4, batch=2)
    x = synth.attention_inputs(w, BF16)
    m = synth.msp_inputs(w, BF16)
    plan = make_plan(w, BF16, embed=True)
    dx = device_inputs(x, w.history_capacity)
    rings = {}
    for k in ("k_hist", "v_hist"):  # the history ring inside guards too
        rbuf, ring = guarded(tuple(dx[k].shape))
        ring.copy_(dx[k])
        rings[k] = rbuf
        dx[k] = ring
    # workspace inside guards
    nws = plan.info.workspace_bytes
    ws_buf = torch.empty(nws + 2 * GUARD * 2, dtype=torch.uint8, device="cuda")
    ws_buf.view(torch.int16).fill_(PATTERN)
    ws = ws_buf[2 * GUARD:2 * GUARD + nws]
    plan.bind(ws, dx["k_sink"], dx["v_sink"], dx["k_hist"], dx["v_hist"])
    # attention output
    out_buf, out = guarded(tuple(dx["q"].shape))
    plan.kv_resample(dx["k_win"], dx["v_win"])
    plan.mssa_forward(dx["q"], dx["k_win"], dx["v_win"], out)
    # embedding output
    N, E = plan.info.n_tokens, w.embed_dim
    tiers = {s: m["w_tier"][s].t().contiguous().cuda() for s in set(w.scales)}
    tok_buf, tok = guarded((w.batch, N, E))
    plan.patchify(m["latent"].cuda(), [tiers[s] for s in w.scales], tok)
    # de-embedding output (from the attention output viewed as tokens)
    lat_buf, lat = guarded((w.batch, w.latent_channels, w.grid_h * w.patch, w.grid_w * w.patch))
    w_out = m["w_out"].t().contiguous().cuda()
    E_att = w.heads * w.head_dim
    if E_att == E:
        plan.unpatchify(0, out.view(w.batch, N, E), w_out, lat)
    else:
        plan.unpatchify(0, tok, w_out, lat)
    # history append into the ring
    plan.history_append(dx["k_win"], dx["v_win"])
    torch.cuda.synchronize()
    assert plan.device_status() == msf().MSF_OK
    for name, buf in (("attention", out_buf), ("embedding", tok_buf), ("de-embedding", lat_buf),
                      ("workspace", ws_buf), ("k ring", rings["k_hist"]), ("v ring", rings["v_hist"])):
        assert guards_intact(buf), name
    assert torch.isfinite(out.float()).all() and torch.isfinite(tok.float()).all()
    assert torch.isfinite(lat.float()).all()


def test_timeout_clears_attention_merge_counters():
    """A launch that gives up can leave the per-block merge counters counted.
    The status read that reports the timeout must zero them, so that the next
    launch merges only finished pieces. The stale counters are planted from
    the host and the TIMEOUT bit comes from the self-test wait: no attention
    launch is made to fail."""
    m = msf()
    w = synth.TINY  # every block is split over several CTAs: merges use the counters
    x = synth.attention_inputs(w, BF16)
    plan = make_plan(w, BF16)
    dx = device_inputs(x, w.history_capacity)
    ws = bind(plan, dx)
    off, nb = int(plan.info.attention_counter_offset), int(plan.info.attention_counter_bytes)
    assert nb > 0 and off % 256 == 0 and off + nb <= ws.numel()
    cnt = ws[off:off + nb].view(torch.int32)
    out = torch.empty_like(dx["q"])
    plan.kv_resample(dx["k_win"], dx["v_win"])
    plan.mssa_forward(dx["q"], dx["k_win"], dx["v_win"], out)
    assert plan.device_status() == m.MSF_OK
    assert bool((cnt == 0).all())  # every merge resets the counter it used
    cnt.fill_(0x00010001)  # one piece finished and one written, left behind
    plan.selftest_wait_timeout(200_000)
    assert plan.device_status() == m.MSF_ERR_TIMEOUT
    assert bool((cnt == 0).all())
    out.fill_(float("nan"))
    plan.mssa_forward(dx["q"], dx["k_win"], dx["v_win"], out)
    assert plan.device_status() == m.MSF_OK
    mx, mean = err_stats(out, oracle_mssa(x, w, 0))
    assert mx <= 2e-2 and mean <= 2e-3
