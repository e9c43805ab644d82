"""Planted mistakes: each test swaps one plausible error into the fp64 oracle
(on the CPU, through monkeypatch, so the oracle itself is untouched) and
checks that at least one of its pins in test_oracle_pins.py then fails.
A pin that still passed with the mistake in place would not be pinning
that part of the oracle.
"""
import numpy as np
import pytest

import test_oracle_pins as pins
from oracle import msp, mssa, schedule


def _fails(fn, *args):
    with pytest.raises(AssertionError):
        fn(*args)


def test_pool_normalised_by_sigma_not_sigma_squared(monkeypatch):
    good = mssa.resample

    def bad(x, gh, gw, sigma, mode=mssa.AVG):
        y = good(x, gh, gw, sigma, mode)
        return y * sigma if mode == mssa.AVG else y
    monkeypatch.setattr(mssa, "resample", bad)
    _fails(pins.test_resample_constant_field_is_identity, mssa.AVG, 2)
    _fails(pins.test_equal_keys_give_weighted_value_mean)


def test_strided_pick_off_the_corner(monkeypatch):
    good = mssa.resample

    def bad(x, gh, gw, sigma, mode=mssa.AVG):
        if mode != mssa.STRIDED or sigma == 1:
            return good(x, gh, gw, sigma, mode)
        x = np.asarray(x, dtype=np.float64)
        grid = x.reshape((x.shape[0], gh, gw) + x.shape[2:])
        out = grid[:, 1::sigma, 1::sigma]      # bottom-right of a 2x2 block
        return out.reshape((x.shape[0], -1) + x.shape[2:])
    monkeypatch.setattr(mssa, "resample", bad)
    _fails(pins.test_resample_linear_ramp, 2)


def test_query_state_left_out_of_its_own_context(monkeypatch):
    good = schedule.context_rows

    def bad(scales, gh, gw, ns, nh, g, frames=1):
        return [r for r in good(scales, gh, gw, ns, nh, g, frames)
                if not (r[0] == schedule.WIN and scales[r[1]] == g)]
    monkeypatch.setattr(schedule, "context_rows", bad)
    _fails(pins.test_eq5_pair_reduction_matches_paper)


def test_history_not_pooled_for_coarse_queries(monkeypatch):
    good = mssa.group_context

    def bad(kv_win, kv_sink, kv_hist, scales, gh, gw, g, mode=mssa.AVG, frames=1):
        # the correct context, but with the history frames at full resolution
        ctx = good(kv_win, kv_sink, kv_hist[:, :0], scales, gh, gw, g, mode, frames)
        ns = np.asarray(kv_sink).shape[1]
        hist = [np.asarray(kv_hist[:, f], dtype=np.float64) for f in range(kv_hist.shape[1])]
        return np.concatenate([ctx[:, :ns]] + hist + [ctx[:, ns:]], axis=1)
    monkeypatch.setattr(mssa, "group_context", bad)
    _fails(pins.test_brute_force_eq4, mssa.AVG, (1, 2), 4, 4, 3, 1)


def test_softmax_scale_dropped(monkeypatch):
    good = mssa.attention
    monkeypatch.setattr(mssa, "attention", lambda q, k, v, scale: good(q, k, v, 1.0))
    _fails(pins.test_all_fine_reduces_to_plain_attention_sdpa)


def test_patch_offsets_swapped(monkeypatch):
    def bad(latent, P):
        x = np.asarray(latent, dtype=np.float64)
        B, C, Hl, Wl = x.shape
        gh, gw = Hl // P, Wl // P
        out = np.empty((B, gh, gw, C * P * P))
        for c in range(C):
            for dy in range(P):
                for dx in range(P):
                    out[:, :, :, c * P * P + dx * P + dy] = x[:, c, dy::P, dx::P]
        return out.reshape(B, gh * gw, C * P * P)
    monkeypatch.setattr(msp, "patchify", bad)
    _fails(pins.test_patch_embedding_equals_strided_conv)
    _fails(pins.test_chunked_patch_embedding_equals_conv3d)


def test_chunk_pooled_across_latent_frames(monkeypatch):
    good = mssa.resample_frames

    def bad(x, frames, gh, gw, sigma, mode=mssa.AVG):
        # per-frame pooling followed by a temporal mean over frame pairs
        y = good(x, frames, gh, gw, sigma, mode).copy()
        n = y.shape[1] // frames
        for f in range(0, frames - 1, 2):
            m = 0.5 * (y[:, f * n:(f + 1) * n] + y[:, (f + 1) * n:(f + 2) * n])
            y[:, f * n:(f + 2) * n] = np.concatenate([m, m], axis=1)
        return y
    monkeypatch.setattr(mssa, "resample_frames", bad)
    _fails(pins.test_chunked_resample_is_per_frame, mssa.AVG, 2)
    _fails(pins.test_chunked_brute_force_eq4, mssa.AVG, (1, 2), 4, 4, 2, 3, 1)


def test_chunk_tokens_frame_minor(monkeypatch):
    good = msp.patchify

    def bad(latent, P):
        x = np.asarray(latent, dtype=np.float64)
        per = [good(x[:, :, f], P) for f in range(x.shape[2])]
        return np.stack(per, axis=2).reshape(x.shape[0], -1, per[0].shape[2])
    monkeypatch.setattr(msp, "patchify_chunk", bad)
    _fails(pins.test_chunked_patch_embedding_equals_conv3d)


# ----------------------------------------------------------- gradient --

import test_oracle_bwd_pins as bpins  # noqa: E402
from oracle import mssa_bwd  # noqa: E402


def test_softmax_jacobian_without_row_term(monkeypatch):
    def bad(q, k, v, dout, scale):
        q, k, v, dout = (np.asarray(a, dtype=np.float64) for a in (q, k, v, dout))
        B, Nq, H, D = q.shape
        dq, dk, dv = np.zeros_like(q), np.zeros_like(k), np.zeros_like(v)
        for b in range(B):
            for h in range(H):
                s = scale * (q[b, :, h] @ k[b, :, h].T)
                p = np.exp(s - s.max(axis=1, keepdims=True))
                p /= p.sum(axis=1, keepdims=True)
                dv[b, :, h] = p.T @ dout[b, :, h]
                ds = p * (dout[b, :, h] @ v[b, :, h].T)       # row term dropped
                dq[b, :, h] = scale * (ds @ k[b, :, h])
                dk[b, :, h] = scale * (ds.T @ q[b, :, h])
        return dq, dk, dv
    monkeypatch.setattr(mssa_bwd, "attention_backward", bad)
    _fails(bpins.test_backward_equals_torch_autograd, mssa.AVG, (1, 2), 4, 4, 1, 3, 1)
    _fails(bpins.test_backward_invariants, mssa.AVG)


def test_pool_adjoint_without_normalisation(monkeypatch):
    good = mssa_bwd.resample_adjoint

    def bad(dy, gh, gw, sigma, mode=mssa.AVG):
        y = good(dy, gh, gw, sigma, mode)
        return y * (sigma * sigma) if mode == mssa.AVG else y
    monkeypatch.setattr(mssa_bwd, "resample_adjoint", bad)
    _fails(bpins.test_backward_equals_torch_autograd, mssa.AVG, (1, 2), 4, 4, 1, 3, 1)


def test_strided_adjoint_to_the_wrong_token(monkeypatch):
    good = mssa_bwd.resample_adjoint

    def bad(dy, gh, gw, sigma, mode=mssa.AVG):
        y = good(dy, gh, gw, sigma, mode)
        if mode != mssa.STRIDED or sigma == 1:
            return y
        B = y.shape[0]
        grid = y.reshape((B, gh, gw) + y.shape[2:])
        return np.roll(grid, 1, axis=2).reshape(y.shape)   # one column to the right
    monkeypatch.setattr(mssa_bwd, "resample_adjoint", bad)
    _fails(bpins.test_backward_equals_torch_autograd, mssa.STRIDED, (1, 2), 4, 4, 1, 3, 1)


# ------------------------------------------- pyramid part, tier projections --

def test_pyramid_states_before_history(monkeypatch):
    good = mssa.pyramid_segment

    def bad(kv_win, kv_hist, scales, gh, gw, g, mode=mssa.AVG, frames=1):
        seg = good(kv_win, kv_hist, scales, gh, gw, g, mode, frames)
        nh = np.asarray(kv_hist).shape[1] * frames * (gh // g) * (gw // g)
        return np.concatenate([seg[:, nh:], seg[:, :nh]], axis=1)
    monkeypatch.setattr(mssa, "pyramid_segment", bad)
    _fails(pins.test_pyramid_segment_is_context_rows_pooled_by_loops, mssa.AVG, (1, 1, 2, 2, 2),
           4, 8, 2, 1)


def test_pyramid_finer_states_pooled_by_g_not_g_over_s(monkeypatch):
    def bad(kv_win, kv_hist, scales, gh, gw, g, mode=mssa.AVG, frames=1):
        offs = schedule.token_offsets(scales, gh, gw, frames)
        cnt = schedule.token_counts(scales, gh, gw, frames)
        parts = [mssa.resample_frames(kv_hist[:, f], frames, gh, gw, g, mode)
                 for f in range(kv_hist.shape[1])]
        for l, s in enumerate(scales):
            if s < g:
                st = np.asarray(kv_win[:, offs[l]:offs[l] + cnt[l]], dtype=np.float64)
                # stride g on a state that is already s times coarser
                parts.append(mssa.resample_frames(st, frames, gh // s, gw // s, g, mode))
        return np.concatenate(parts, axis=1)
    monkeypatch.setattr(mssa, "pyramid_segment", bad)
    _fails(pins.test_pyramid_segment_is_context_rows_pooled_by_loops, mssa.AVG, (1, 2, 4, 4),
           8, 8, 1, 1)


def test_tier_weights_swapped_between_states(monkeypatch):
    good = msp.patchify_window

    def bad(latent, scales, patch, w_tier=None):
        if w_tier is None:
            return good(latent, scales, patch, w_tier)
        # the window's states embedded in reverse position order
        x = np.asarray(latent, dtype=np.float64)
        cut = msp.patchify_chunk if x.ndim == 6 else msp.patchify
        blocks = [cut(x[:, l], patch * s) @ np.asarray(w_tier[s]) for l, s in enumerate(scales)]
        return np.concatenate(blocks[::-1], axis=1)
    monkeypatch.setattr(msp, "patchify_window", bad)
    _fails(pins.test_tier_embedding_is_a_strided_conv_per_state, 1)


def test_tier_embedding_weight_transposed(monkeypatch):
    good = msp.patchify_window

    def bad(latent, scales, patch, w_tier=None):
        if w_tier is None:
            return good(latent, scales, patch, w_tier)
        sq = {s: (np.asarray(w).T if np.asarray(w).shape[0] == np.asarray(w).shape[1] else w)
              for s, w in w_tier.items()}
        return good(latent, scales, patch, sq)
    monkeypatch.setattr(msp, "patchify_window", bad)
    _fails(pins.test_tier_embedding_is_a_strided_conv_per_state, 1)


def test_deembedding_weight_transposed(monkeypatch):
    good = msp.unpatchify_state

    def bad(tokens, P, C, Hl, Wl, w_out=None, frames=0):
        return good(tokens, P, C, Hl, Wl, None if w_out is None else np.asarray(w_out).T, frames)
    monkeypatch.setattr(msp, "unpatchify_state", bad)
    _fails(pins.test_deembedding_is_linear_then_fold, 2)


# ------------------------------------------------------- tier modules --

def test_tier_lora_scale_dropped(monkeypatch):
    good = msp.embed_tier
    monkeypatch.setattr(msp, "embed_tier", lambda x, w, a=None, b=None, gamma=1.0: good(x, w, a, b, 1.0))
    _fails(pins.test_tier_lora_embedding_is_a_conv_with_the_merged_weight)
    good_d = msp.deembed_tier
    monkeypatch.setattr(msp, "deembed_tier",
                        lambda h, wo, a=None, b=None, gamma=1.0, x=None, r=None: good_d(h, wo, a, b, 1.0, x, r))
    _fails(pins.test_tier_deembedding_lora_is_linear_with_the_merged_weight_then_fold)


def test_latent_residual_transposed(monkeypatch):
    good = msp.deembed_tier

    def bad(h, w_out, a=None, b=None, gamma=1.0, x=None, residual=None):
        return good(h, w_out, a, b, gamma, x, None if residual is None else np.asarray(residual).T)
    monkeypatch.setattr(msp, "deembed_tier", bad)
    _fails(pins.test_latent_residual_is_a_patch_conv_then_fold, 2)


def test_latent_residual_of_the_output_not_the_input(monkeypatch):
    good = msp.deembed_tier

    def bad(h, w_out, a=None, b=None, gamma=1.0, x=None, residual=None):
        y = good(h, w_out, a, b, gamma)
        return y if residual is None else y + y @ np.asarray(residual)
    monkeypatch.setattr(msp, "deembed_tier", bad)
    _fails(pins.test_latent_residual_identity_passes_the_input_latent_through, 2)
