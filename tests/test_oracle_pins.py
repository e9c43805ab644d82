"""Pins of the fp64 oracle to things the paper and the mathematics fix.

Each test checks the oracle against something other than itself: a number
the paper prints (tests/golden/paper_ratios.json), a closed form, a library
routine on a special case, or a second enumeration written independently.
"""
import json
import math
import os
from fractions import Fraction

import numpy as np
import pytest
import torch

from oracle import brute, msp, mssa, schedule, stream

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "paper_ratios.json")


def _golden():
    with open(GOLDEN) as f:
        return json.load(f)


# ---------------------------------------------------------------- Eq. 3 --

def test_eq3_rho_tok_matches_paper():
    g = _golden()["rho_tok"]
    scales = g["scales"]
    # closed form of Eq. 3
    assert float(schedule.rho_tok(scales)) == pytest.approx(g["value"], abs=1e-12)
    # the same ratio from the enumerated token counts on the 480p grid
    cnt = schedule.token_counts(scales, 30, 52)
    assert cnt == [1560, 1560, 390, 390, 390]
    assert Fraction(sum(cnt), 5 * 30 * 52) == Fraction(55, 100)
    assert 1 - sum(cnt) / (5 * 1560) == pytest.approx(g["token_reduction"], abs=1e-12)


@pytest.mark.parametrize("scales,gh,gw,expect", [
    ((1, 1, 2), 8, 8, [64, 64, 16]),
    ((1, 1, 2, 2, 4, 4), 48, 80, [3840, 3840, 960, 960, 240, 240]),
    ((1, 1, 1, 1, 1), 30, 52, [1560] * 5),
])
def test_eq3_counts_and_bijective_token_index(scales, gh, gw, expect):
    cnt = schedule.token_counts(scales, gh, gw)
    assert cnt == expect
    seen = set()
    for l, s in enumerate(scales):
        for i in range(gh // s):
            for j in range(gw // s):
                seen.add(schedule.token_of(scales, gh, gw, l, i, j))
    assert seen == set(range(sum(expect)))


def test_schedule_validation():
    with pytest.raises(ValueError):
        schedule.validate((1, 2, 1), 8, 8)        # not monotone
    with pytest.raises(ValueError):
        schedule.validate((1, 3), 6, 6)           # not a power of two
    with pytest.raises(ValueError):
        schedule.validate((1, 1, 2, 2, 4), 30, 52)  # 30 not divisible by 4
    schedule.validate((1, 1, 2, 2, 2), 30, 52)


# ---------------------------------------------------------------- Eq. 5 --

def test_eq5_pair_reduction_matches_paper():
    g = _golden()["r_mssa"]
    scales, gh, gw = g["scales"], 30, 52
    G = gh * gw
    # one sink frame at full resolution = G sink tokens; one history frame
    pairs = schedule.attention_pairs(scales, gh, gw, G * g["sink_frames"], g["history_frames"])
    dense = schedule.msp_only_pairs(scales, gh, gw, G * g["sink_frames"], g["history_frames"])
    r_enum = 1 - Fraction(pairs, dense)
    r_eq5 = schedule.r_mssa_eq5(scales, g["sink_frames"], g["history_frames"])
    # enumeration of Eq. 4 contexts and the closed form of Eq. 5 agree exactly
    assert r_enum == r_eq5
    # and round to the paper's printed 12.9%
    assert round(float(r_enum), g["printed_digits"]) == pytest.approx(g["value"], abs=1e-12)


def test_eq5_other_layouts_enum_vs_closed_form():
    for scales, gh, gw, nh in [((1, 1, 2, 2, 4, 4), 48, 80, 2), ((1, 2), 4, 4, 3),
                               ((2, 2, 4), 8, 8, 1), ((1, 1, 1), 4, 6, 2)]:
        G = gh * gw
        pairs = schedule.attention_pairs(scales, gh, gw, G, nh)
        dense = schedule.msp_only_pairs(scales, gh, gw, G, nh)
        assert 1 - Fraction(pairs, dense) == schedule.r_mssa_eq5(scales, 1, nh)
    # an all-fine schedule removes nothing
    assert schedule.r_mssa_eq5((1, 1, 1, 1, 1), 1, 1) == 0


def test_cfg1_flops():
    # 480p layer: 3120 x 8970 + 1170 x 4290 pairs per head, 12 heads, D = 128
    pairs = schedule.attention_pairs((1, 1, 2, 2, 2), 30, 52, 1560, 2)
    assert pairs == 3120 * 8970 + 1170 * 4290
    fl = schedule.attention_flops((1, 1, 2, 2, 2), 30, 52, 1560, 2, 12, 128)
    assert fl == 4 * 128 * 12 * pairs
    assert fl / 1e9 == pytest.approx(202.79, abs=0.01)


# ------------------------------------------------------------- resample --

@pytest.mark.parametrize("mode", [mssa.AVG, mssa.STRIDED])
@pytest.mark.parametrize("sigma", [1, 2, 4])
def test_resample_constant_field_is_identity(mode, sigma):
    x = np.full((2, 8 * 12, 3, 5), 0.375)
    y = mssa.resample(x, 8, 12, sigma, mode)
    assert y.shape == (2, (8 // sigma) * (12 // sigma), 3, 5)
    assert np.all(y == 0.375)


@pytest.mark.parametrize("sigma", [2, 4])
def test_resample_linear_ramp(sigma):
    gh, gw = 8, 16
    a, b, c = 0.7, -1.3, 2.0
    i, j = np.meshgrid(np.arange(gh), np.arange(gw), indexing="ij")
    x = (a * i + b * j + c).reshape(1, gh * gw, 1, 1)
    oi, oj = np.meshgrid(np.arange(gh // sigma), np.arange(gw // sigma), indexing="ij")
    centre = a * (sigma * oi + (sigma - 1) / 2) + b * (sigma * oj + (sigma - 1) / 2) + c
    corner = a * (sigma * oi) + b * (sigma * oj) + c
    avg = mssa.resample(x, gh, gw, sigma, mssa.AVG).reshape(gh // sigma, gw // sigma)
    st = mssa.resample(x, gh, gw, sigma, mssa.STRIDED).reshape(gh // sigma, gw // sigma)
    np.testing.assert_allclose(avg, centre, rtol=0, atol=1e-12)
    np.testing.assert_allclose(st, corner, rtol=0, atol=0)


def test_resample_mean_is_block_mean_by_library_reshape():
    rng = np.random.default_rng(3)
    x = rng.standard_normal((2, 8 * 12, 2, 4))
    y = mssa.resample(x, 8, 12, 4, mssa.AVG)
    ref = x.reshape(2, 2, 4, 3, 4, 2, 4).mean(axis=(2, 4)).reshape(2, 6, 2, 4)
    np.testing.assert_allclose(y, ref, rtol=0, atol=1e-13)


# ------------------------------------------------------------ attention --

def _rand_inputs(rng, scales, gh, gw, ns, nh, H, D, B=1):
    N = sum(schedule.token_counts(scales, gh, gw))
    G = gh * gw
    return dict(
        q=rng.standard_normal((B, N, H, D)), k_win=rng.standard_normal((B, N, H, D)),
        v_win=rng.standard_normal((B, N, H, D)), k_sink=rng.standard_normal((B, ns, H, D)),
        v_sink=rng.standard_normal((B, ns, H, D)), k_hist=rng.standard_normal((B, nh, G, H, D)),
        v_hist=rng.standard_normal((B, nh, G, H, D)))


def test_all_fine_reduces_to_plain_attention_sdpa():
    rng = np.random.default_rng(0)
    scales, gh, gw = (1, 1, 1), 4, 6
    x = _rand_inputs(rng, scales, gh, gw, ns=5, nh=2, H=3, D=16, B=2)
    out = mssa.mssa_forward(x["q"], x["k_win"], x["v_win"], x["k_sink"], x["v_sink"],
                            x["k_hist"], x["v_hist"], scales, gh, gw)
    B, N, H, D = x["q"].shape
    kh = x["k_hist"].reshape(B, -1, H, D)
    vh = x["v_hist"].reshape(B, -1, H, D)
    K = np.concatenate([x["k_sink"], kh, x["k_win"]], axis=1)
    V = np.concatenate([x["v_sink"], vh, x["v_win"]], axis=1)
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a.transpose(0, 2, 1, 3)))
    ref = torch.nn.functional.scaled_dot_product_attention(t(x["q"]), t(K), t(V))
    np.testing.assert_allclose(out, ref.numpy().transpose(0, 2, 1, 3), rtol=0, atol=1e-12)


@pytest.mark.parametrize("mode", [mssa.AVG, mssa.STRIDED])
@pytest.mark.parametrize("scales,gh,gw,ns,nh", [
    ((1, 2), 4, 4, 3, 1),
    ((1, 2, 4), 4, 8, 2, 2),
    ((1, 1, 2), 8, 8, 64, 1),     # the tiny workload's grid and schedule
    ((2, 2, 4), 4, 8, 1, 1),      # no fine state at all
])
def test_brute_force_eq4(mode, scales, gh, gw, ns, nh):
    rng = np.random.default_rng(11)
    x = _rand_inputs(rng, scales, gh, gw, ns, nh, H=2, D=6)
    out = mssa.mssa_forward(x["q"], x["k_win"], x["v_win"], x["k_sink"], x["v_sink"],
                            x["k_hist"], x["v_hist"], scales, gh, gw, mode=mode)
    ref = brute.mssa_brute(x["q"].tolist(), x["k_win"].tolist(), x["v_win"].tolist(),
                           x["k_sink"].tolist(), x["v_sink"].tolist(), x["k_hist"].tolist(),
                           x["v_hist"].tolist(), scales, gh, gw, mode=mode)
    np.testing.assert_allclose(out, np.array(ref), rtol=0, atol=1e-12)


def test_equal_keys_give_weighted_value_mean():
    """All keys equal -> uniform softmax -> o = mean of the context values.
    For AVG pooling a frame pooled by s contributes (1/s^2) * (sum of its fine
    values) over (G/s^2) rows; the closed form below never builds a context."""
    rng = np.random.default_rng(5)
    scales, gh, gw, ns, nh = (1, 2, 4), 8, 8, 7, 2
    x = _rand_inputs(rng, scales, gh, gw, ns, nh, H=2, D=3)
    for key in ("k_win", "k_sink", "k_hist"):
        x[key] = np.ones_like(x[key]) * 0.25
    out = mssa.mssa_forward(x["q"], x["k_win"], x["v_win"], x["k_sink"], x["v_sink"],
                            x["k_hist"], x["v_hist"], scales, gh, gw)
    G = gh * gw
    cnt = [G // (s * s) for s in scales]
    offs = np.cumsum([0] + cnt)
    for l, g in enumerate(scales):
        num = x["v_sink"][0].sum(axis=0)
        den = ns
        for f in range(nh):
            num = num + x["v_hist"][0, f].sum(axis=0) / (g * g)
            den += G // (g * g)
        for m, s in enumerate(scales):
            st = max(1, g // s)
            num = num + x["v_win"][0, offs[m]:offs[m + 1]].sum(axis=0) / (st * st)
            den += cnt[m] // (st * st)
        expect = num / den
        got = out[0, offs[l]:offs[l + 1]]
        np.testing.assert_allclose(got, np.broadcast_to(expect, got.shape), rtol=0, atol=1e-12)


def test_permutation_invariance_and_convexity():
    rng = np.random.default_rng(7)
    scales, gh, gw, ns, nh = (1, 1, 2), 8, 8, 9, 2
    x = _rand_inputs(rng, scales, gh, gw, ns, nh, H=2, D=8)
    args = lambda d: (d["q"], d["k_win"], d["v_win"], d["k_sink"], d["v_sink"], d["k_hist"],
                      d["v_hist"], scales, gh, gw)
    out = mssa.mssa_forward(*args(x))
    perm = rng.permutation(ns)
    y = dict(x)
    y["k_sink"] = x["k_sink"][:, perm]
    y["v_sink"] = x["v_sink"][:, perm]
    y["k_hist"] = x["k_hist"][:, ::-1]
    y["v_hist"] = x["v_hist"][:, ::-1]
    np.testing.assert_allclose(mssa.mssa_forward(*args(y)), out, rtol=0, atol=1e-12)
    allv = np.concatenate([x["v_sink"], x["v_hist"].reshape(1, -1, 2, 8), x["v_win"]], axis=1)
    lo, hi = allv.min(axis=1, keepdims=True), allv.max(axis=1, keepdims=True)
    assert np.all(out >= lo - 1e-12) and np.all(out <= hi + 1e-12)


def test_softmax_scale_default_is_inverse_sqrt_d():
    rng = np.random.default_rng(9)
    q = rng.standard_normal((1, 3, 1, 16))
    k = rng.standard_normal((1, 5, 1, 16))
    v = rng.standard_normal((1, 5, 1, 16))
    o = mssa.attention(q, k, v, 0.25)
    s = q[0, :, 0] @ k[0, :, 0].T / math.sqrt(16)
    p = np.exp(s) / np.exp(s).sum(axis=1, keepdims=True)
    np.testing.assert_allclose(o[0, :, 0], p @ v[0, :, 0], rtol=0, atol=1e-13)


# ------------------------------------------------------------------ MSP --

@pytest.mark.parametrize("P", [1, 2, 4, 8])
def test_patchify_roundtrip_and_library_reshape(P):
    rng = np.random.default_rng(P)
    B, C, Hl, Wl = 2, 3, 16, 24
    x = rng.standard_normal((B, C, Hl, Wl))
    t = msp.patchify(x, P)
    gh, gw = Hl // P, Wl // P
    ref = x.reshape(B, C, gh, P, gw, P).transpose(0, 2, 4, 1, 3, 5).reshape(B, gh * gw, C * P * P)
    assert np.array_equal(t, ref)
    assert np.array_equal(msp.unpatchify(t, P, C, Hl, Wl), x)


def test_patch_embedding_equals_strided_conv():
    """Tier embedding of (c, dy, dx)-ordered patches == Conv2d with kernel = stride = P."""
    rng = np.random.default_rng(1)
    B, C, Hl, Wl, P, E = 1, 4, 8, 12, 2, 5
    x = rng.standard_normal((B, C, Hl, Wl))
    W = rng.standard_normal((C * P * P, E))
    emb = msp.patchify(x, P) @ W
    conv = torch.nn.functional.conv2d(torch.from_numpy(x),
                                      torch.from_numpy(W.T.reshape(E, C, P, P).copy()), stride=P)
    ref = conv.numpy().reshape(B, E, -1).transpose(0, 2, 1)
    np.testing.assert_allclose(emb, ref, rtol=0, atol=1e-12)


# ------------------------------------------------------------ streaming --

def test_history_ring_keeps_newest_frames():
    B, G, H, D, cap = 1, 4, 1, 2, 4
    h0 = np.stack([np.full((B, G, H, D), f) for f in range(2)], axis=1)
    hist = stream.History(h0, h0 + 100, cap)
    for f in range(2, 9):
        hist.append(np.full((B, G, H, D), f), np.full((B, G, H, D), f + 100))
        k, v = hist.frames()
        assert k.shape[1] == min(cap, f + 1)
        live = sorted(int(k[0, s, 0, 0, 0]) for s in range(k.shape[1]))
        assert live == list(range(max(0, f + 1 - cap), f + 1))
        assert np.all(v == k + 100)


# --------------------------------------------- chunked states (Sec. 5.1) --
# The paper's window holds T = 5 chunks of 3 latent frames each; patches are
# spatial, so Eq. 3 applies per latent frame and Subsample acts on each
# latent frame's grid separately.

def test_chunked_counts_keep_the_printed_token_ratio():
    g = _golden()["rho_tok"]
    cnt = schedule.token_counts(g["scales"], 30, 52, frames=3)
    assert cnt == [4680, 4680, 1170, 1170, 1170]
    assert Fraction(sum(cnt), 5 * 3 * 30 * 52) == Fraction(55, 100)
    assert 1 - sum(cnt) / (5 * 3 * 1560) == pytest.approx(g["token_reduction"], abs=1e-12)


def test_chunked_contexts_keep_the_printed_pair_ratio():
    """Every per-frame count scales by F, every pair count by F^2, so Eq. 5's
    closed form (written per frame) must still equal the chunked enumeration."""
    g = _golden()["r_mssa"]
    scales, gh, gw, F = g["scales"], 30, 52, 3
    sink = F * gh * gw * g["sink_frames"]
    pairs = schedule.attention_pairs(scales, gh, gw, sink, g["history_frames"], frames=F)
    dense = schedule.msp_only_pairs(scales, gh, gw, sink, g["history_frames"], frames=F)
    r = 1 - Fraction(pairs, dense)
    assert r == schedule.r_mssa_eq5(scales, g["sink_frames"], g["history_frames"])
    assert round(float(r), g["printed_digits"]) == pytest.approx(g["value"], abs=1e-12)
    # and exactly F^2 times the one-frame pair count
    assert pairs == F * F * schedule.attention_pairs(scales, gh, gw, gh * gw, 1)


@pytest.mark.parametrize("mode", [mssa.AVG, mssa.STRIDED])
@pytest.mark.parametrize("sigma", [2, 4])
def test_chunked_resample_is_per_frame(mode, sigma):
    """Frame f of the chunk holds 100 f + row: pooled rows stay inside their
    frame (no temporal mixing) and land at the block centre (AVG) or the
    block's top row (STRIDED)."""
    F, gh, gw = 3, 8, 4
    f, i, _ = np.meshgrid(np.arange(F), np.arange(gh), np.arange(gw), indexing="ij")
    x = (100.0 * f + i).reshape(1, F * gh * gw, 1, 1)
    y = mssa.resample_frames(x, F, gh, gw, sigma, mode).reshape(F, gh // sigma, gw // sigma)
    of, oi, _ = np.meshgrid(np.arange(F), np.arange(gh // sigma), np.arange(gw // sigma),
                            indexing="ij")
    off = (sigma - 1) / 2 if mode == mssa.AVG else 0
    np.testing.assert_allclose(y, 100.0 * of + sigma * oi + off, rtol=0, atol=1e-12)


def test_chunked_index_rows_are_bijective():
    scales, gh, gw, F = (1, 2, 4), 8, 8, 3
    seen = set()
    for l, s in enumerate(scales):
        for f in range(F):
            for i in range(gh // s):
                for j in range(gw // s):
                    seen.add(schedule.token_of(scales, gh, gw, l, i, j, f=f, frames=F))
    assert seen == set(range(sum(schedule.token_counts(scales, gh, gw, F))))


def _rand_chunk_inputs(rng, scales, gh, gw, F, ns, nh, H, D, B=1):
    N = sum(schedule.token_counts(scales, gh, gw, F))
    G = F * gh * gw
    return dict(
        q=rng.standard_normal((B, N, H, D)), k_win=rng.standard_normal((B, N, H, D)),
        v_win=rng.standard_normal((B, N, H, D)), k_sink=rng.standard_normal((B, ns, H, D)),
        v_sink=rng.standard_normal((B, ns, H, D)), k_hist=rng.standard_normal((B, nh, G, H, D)),
        v_hist=rng.standard_normal((B, nh, G, H, D)))


@pytest.mark.parametrize("mode", [mssa.AVG, mssa.STRIDED])
@pytest.mark.parametrize("scales,gh,gw,F,ns,nh", [
    ((1, 2), 4, 4, 2, 3, 1),
    ((1, 1, 2), 4, 4, 3, 2, 2),
    ((2, 4), 4, 8, 2, 1, 1),
])
def test_chunked_brute_force_eq4(mode, scales, gh, gw, F, ns, nh):
    rng = np.random.default_rng(13)
    x = _rand_chunk_inputs(rng, scales, gh, gw, F, ns, nh, H=2, D=5)
    out = mssa.mssa_forward(x["q"], x["k_win"], x["v_win"], x["k_sink"], x["v_sink"],
                            x["k_hist"], x["v_hist"], scales, gh, gw, mode=mode, frames=F)
    ref = brute.mssa_brute(x["q"].tolist(), x["k_win"].tolist(), x["v_win"].tolist(),
                           x["k_sink"].tolist(), x["v_sink"].tolist(), x["k_hist"].tolist(),
                           x["v_hist"].tolist(), scales, gh, gw, mode=mode, frames=F)
    np.testing.assert_allclose(out, np.array(ref), rtol=0, atol=1e-12)


def test_chunked_patch_embedding_equals_conv3d():
    """A chunk's tier embedding == Conv3d with kernel = stride = (1, P, P),
    tokens in (frame, row, col) order; the rearrangement inverts exactly."""
    rng = np.random.default_rng(2)
    B, C, F, Hl, Wl, P, E = 2, 3, 3, 8, 12, 4, 5
    x = rng.standard_normal((B, C, F, Hl, Wl))
    W = rng.standard_normal((C * P * P, E))
    t = msp.patchify_chunk(x, P)
    conv = torch.nn.functional.conv3d(torch.from_numpy(x),
                                      torch.from_numpy(W.T.reshape(E, C, 1, P, P).copy()),
                                      stride=(1, P, P))
    ref = conv.numpy().reshape(B, E, -1).transpose(0, 2, 1)
    np.testing.assert_allclose(t @ W, ref, rtol=0, atol=1e-12)
    assert np.array_equal(msp.unpatchify_chunk(t, P, C, F, Hl, Wl), x)


# ------------------------------------------- pyramid part and tier projections --

def _pooled_row_by_loops(src, kind_grid, st, row, col, mode):
    """One Subsample row of Eq. 4 built by explicit loops from its source
    frame. src [B, F*gh*gw, H, D] holds F latent-frame grids of gh x gw (the
    source grid before pooling); (row, col) is on the pooled grid with the
    latent frame folded into the row (row = f * (gh/st) + i)."""
    gh, gw = kind_grid
    ph = gh // st
    f, i = divmod(row, ph)
    base = f * gh * gw
    if mode == mssa.STRIDED:
        return src[:, base + (st * i) * gw + st * col]
    acc = np.zeros(src.shape[:1] + src.shape[2:])
    for dy in range(st):
        for dx in range(st):
            acc = acc + src[:, base + (st * i + dy) * gw + (st * col + dx)]
    return acc / (st * st)


@pytest.mark.parametrize("mode", [mssa.AVG, mssa.STRIDED])
@pytest.mark.parametrize("scales,gh,gw,nh,F", [
    ((1, 1, 2, 2, 2), 4, 8, 2, 1),
    ((1, 2, 4, 4), 8, 8, 1, 1),
    ((1, 1, 2, 4), 8, 4, 2, 2),
])
def test_pyramid_segment_is_context_rows_pooled_by_loops(mode, scales, gh, gw, nh, F):
    """The resampled part of group g's context (the segment the GPU pyramid
    holds) is, row for row, the history and finer-window rows of Eq. 4's
    context in context order, each pooled from its source by explicit loops."""
    rng = np.random.default_rng(11)
    B, H, D = 2, 2, 3
    N = sum(schedule.token_counts(scales, gh, gw, F))
    kv_win = rng.standard_normal((B, N, H, D))
    kv_hist = rng.standard_normal((B, nh, F * gh * gw, H, D))
    offs = schedule.token_offsets(scales, gh, gw, F)
    cnt = schedule.token_counts(scales, gh, gw, F)
    for g in sorted(set(scales)):
        if g == 1:
            continue
        seg = mssa.pyramid_segment(kv_win, kv_hist, scales, gh, gw, g, mode, F)
        rows = [r for r in schedule.context_rows(scales, gh, gw, 0, nh, g, F)
                if r[0] == schedule.HIST or (r[0] == schedule.WIN and scales[r[1]] < g)]
        assert seg.shape == (B, len(rows), H, D)
        for n, (kind, frame, st, row, col) in enumerate(rows):
            if kind == schedule.HIST:
                src, grid = kv_hist[:, frame], (gh, gw)
            else:
                s = scales[frame]
                src, grid = kv_win[:, offs[frame]:offs[frame] + cnt[frame]], (gh // s, gw // s)
            want = _pooled_row_by_loops(src, grid, st, row, col, mode)
            np.testing.assert_allclose(seg[:, n], want, rtol=0, atol=1e-12)


@pytest.mark.parametrize("F", [1, 2])
def test_tier_embedding_is_a_strided_conv_per_state(F):
    """MSP of a window with tier projections: each state is embedded by the
    patch-embedding conv (kernel = stride = its patch P_l) of its own tier's
    weight, and the states' token blocks follow in position order. Weights of
    the patch-2 tier are square (C*P^2 = E) so that using one transposed
    cannot go unnoticed."""
    rng = np.random.default_rng(12)
    scales, patch, C, E, B = (1, 1, 2, 2), 2, 4, 16, 2
    Hl, Wl = 8, 16
    lat_shape = (B, len(scales), C, Hl, Wl) if F == 1 else (B, len(scales), C, F, Hl, Wl)
    latent = rng.standard_normal(lat_shape)
    w_tier = {s: rng.standard_normal((C * (patch * s) ** 2, E)) for s in set(scales)}
    got = msp.patchify_window(latent, scales, patch, w_tier)
    blocks = []
    for l, s in enumerate(scales):
        P = patch * s
        wt = torch.from_numpy(w_tier[s].T.reshape(E, C, P, P).copy())
        x = torch.from_numpy(latent[:, l].copy())
        if F == 1:
            y = torch.nn.functional.conv2d(x, wt, stride=P)              # [B, E, gh, gw]
            blocks.append(y.flatten(2).transpose(1, 2))
        else:
            y = torch.nn.functional.conv3d(x, wt.unsqueeze(2), stride=(1, P, P))  # [B, E, F, gh, gw]
            blocks.append(y.flatten(2).transpose(1, 2))
    want = torch.cat(blocks, dim=1).numpy()
    assert got.shape == want.shape
    np.testing.assert_allclose(got, want, rtol=0, atol=1e-10)


@pytest.mark.parametrize("P", [2, 4])
def test_deembedding_is_linear_then_fold(P):
    """De-embedding + unpatchify of one state: the nn.Linear map E -> C*P^2
    of every token, then torch's fold with kernel = stride = P (the inverse
    patch rearrangement, feature order (c, dy, dx)). E = C*P^2 makes the
    weight square, so a transposed use changes the values, not the shape."""
    rng = np.random.default_rng(13)
    B, C, gh, gw = 2, 3, 3, 5
    E = C * P * P
    tokens = rng.standard_normal((B, gh * gw, E))
    w_out = rng.standard_normal((E, C * P * P))  # [E, C*P^2]: tokens @ w_out
    got = msp.unpatchify_state(tokens, P, C, gh * P, gw * P, w_out=w_out)
    lin = torch.nn.functional.linear(torch.from_numpy(tokens), torch.from_numpy(w_out.T.copy()))
    want = torch.nn.functional.fold(lin.transpose(1, 2), output_size=(gh * P, gw * P),
                                    kernel_size=P, stride=P).numpy()
    np.testing.assert_allclose(got, want, rtol=0, atol=1e-10)


# ------------------------------------------------------- tier modules --

def _tier_weights(rng, K, E, r):
    return {"w": rng.standard_normal((K, E)), "lora_a": rng.standard_normal((K, r)),
            "lora_b": rng.standard_normal((r, E)), "gamma": 0.375}


def test_tier_lora_embedding_is_a_conv_with_the_merged_weight():
    """Embedding with LoRA = the patch-embedding conv whose kernel is the tier
    weight plus the scaled rank-r product (linearity of the conv in its
    weight); the native tier (no adapters) is the plain conv."""
    rng = np.random.default_rng(21)
    scales, patch, C, E, B, r = (1, 2, 2), 2, 4, 24, 2, 8
    latent = rng.standard_normal((B, len(scales), C, 8, 16))
    tiers = {1: {"w": rng.standard_normal((C * 4, E))},
             2: _tier_weights(rng, C * 16, E, r)}
    got = msp.patchify_window_tiers(latent, scales, patch, tiers)
    blocks = []
    for l, s in enumerate(scales):
        P, t = patch * s, tiers[s]
        merged = t["w"] + (t["gamma"] * (t["lora_a"] @ t["lora_b"]) if "lora_a" in t else 0.0)
        wt = torch.from_numpy(np.ascontiguousarray(merged.T).reshape(E, C, P, P))
        y = torch.nn.functional.conv2d(torch.from_numpy(latent[:, l].copy()), wt, stride=P)
        blocks.append(y.flatten(2).transpose(1, 2))
    np.testing.assert_allclose(got, torch.cat(blocks, 1).numpy(), rtol=0, atol=1e-9)


def test_tier_lora_update_has_rank_r_and_vanishes_with_a_zero_up_projection():
    rng = np.random.default_rng(22)
    K, E, r, n = 64, 48, 8, 200
    t = _tier_weights(rng, K, E, r)
    x = rng.standard_normal((n, K))
    delta = msp.embed_tier(x, t["w"], t["lora_a"], t["lora_b"], t["gamma"]) - msp.embed_tier(x, t["w"])
    sv = np.linalg.svd(delta, compute_uv=False)
    assert sv[r - 1] > 1e-3 * sv[0] and sv[r] < 1e-10 * sv[0]
    zero = msp.embed_tier(x, t["w"], t["lora_a"], np.zeros_like(t["lora_b"]), t["gamma"])
    assert np.array_equal(zero, msp.embed_tier(x, t["w"]))
    d2 = msp.deembed_tier(x[:, :E], t["w"].T, t["lora_b"].T, t["lora_a"].T, t["gamma"]) - \
        msp.deembed_tier(x[:, :E], t["w"].T)
    sv = np.linalg.svd(d2, compute_uv=False)
    assert sv[r] < 1e-10 * sv[0]


@pytest.mark.parametrize("P", [2, 4])
def test_latent_residual_identity_passes_the_input_latent_through(P):
    """With R = I, no de-embedding weight and no adapters the tier's output
    latent is its input latent, exactly; with a de-embedding it is that
    de-embedding plus the input latent."""
    rng = np.random.default_rng(23)
    B, C, gh, gw, E = 2, 3, 3, 4, 20
    K = C * P * P
    lat = rng.standard_normal((B, C, gh * P, gw * P))
    tok = rng.standard_normal((B, gh * gw, E))
    ident = {"w_out": np.zeros((E, K)), "residual": np.eye(K)}
    assert np.array_equal(msp.unpatchify_state_tier(tok, lat, P, ident), lat)
    w_out = rng.standard_normal((E, K))
    got = msp.unpatchify_state_tier(tok, lat, P, {"w_out": w_out, "residual": np.eye(K)})
    base = msp.unpatchify_state(tok, P, C, gh * P, gw * P, w_out=w_out)
    np.testing.assert_allclose(got, base + lat, rtol=0, atol=1e-12)


@pytest.mark.parametrize("P", [2, 4])
def test_latent_residual_is_a_patch_conv_then_fold(P):
    """The residual branch alone (zero de-embedding) is a strided conv of the
    input latent (kernel = stride = P, weight R as C*P^2 filters) followed by
    fold, torch's inverse patch rearrangement. R is square, so a transposed
    use changes the values."""
    rng = np.random.default_rng(24)
    B, C, gh, gw, E = 2, 2, 3, 5, 8
    K = C * P * P
    lat = rng.standard_normal((B, C, gh * P, gw * P))
    R = rng.standard_normal((K, K))
    got = msp.unpatchify_state_tier(np.zeros((B, gh * gw, E)), lat, P,
                                    {"w_out": np.zeros((E, K)), "residual": R})
    wt = torch.from_numpy(np.ascontiguousarray(R.T).reshape(K, C, P, P))
    y = torch.nn.functional.conv2d(torch.from_numpy(lat), wt, stride=P)  # [B, K, gh, gw]
    want = torch.nn.functional.fold(y.flatten(2), output_size=(gh * P, gw * P), kernel_size=P,
                                    stride=P).numpy()
    np.testing.assert_allclose(got, want, rtol=0, atol=1e-10)


def test_tier_deembedding_lora_is_linear_with_the_merged_weight_then_fold():
    rng = np.random.default_rng(25)
    B, C, P, gh, gw, E, r = 2, 2, 4, 2, 3, 40, 8
    K = C * P * P
    tok = rng.standard_normal((B, gh * gw, E))
    lat = rng.standard_normal((B, C, gh * P, gw * P))
    t = {"w_out": rng.standard_normal((E, K)), "out_a": rng.standard_normal((E, r)),
         "out_b": rng.standard_normal((r, K)), "gamma": 0.625}
    got = msp.unpatchify_state_tier(tok, lat, P, t)
    merged = t["w_out"] + t["gamma"] * (t["out_a"] @ t["out_b"])
    lin = torch.nn.functional.linear(torch.from_numpy(tok), torch.from_numpy(merged.T.copy()))
    want = torch.nn.functional.fold(lin.transpose(1, 2), output_size=(gh * P, gw * P),
                                    kernel_size=P, stride=P).numpy()
    np.testing.assert_allclose(got, want, rtol=0, atol=1e-9)
