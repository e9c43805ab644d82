"""Pins of the fp64 MSSA gradient (oracle/mssa_bwd.py) to things other than
itself: torch autograd through an independent torch formulation of Eq. 4
(contexts from avg_pool2d / strided slicing, attention from
scaled_dot_product_attention), central finite differences of the pinned
forward oracle, and two invariants of softmax attention."""
import numpy as np
import pytest
import torch
import torch.nn.functional as Fn

from oracle import mssa, mssa_bwd, schedule


def _inputs(rng, scales, gh, gw, F, ns, nh, H, D, B=1):
    N = sum(schedule.token_counts(scales, gh, gw, F))
    G = F * gh * gw
    sh = dict(q=(B, N, H, D), k_win=(B, N, H, D), v_win=(B, N, H, D), k_sink=(B, ns, H, D),
              v_sink=(B, ns, H, D), k_hist=(B, nh, G, H, D), v_hist=(B, nh, G, H, D),
              dout=(B, N, H, D))
    return {k: rng.standard_normal(s) for k, s in sh.items()}


def _torch_pool(x, frames, gh, gw, s, mode):
    """[B, frames*gh*gw, H, D] -> pooled per latent frame, via the library's
    avg_pool2d (AVG) or a strided slice (STRIDED)."""
    if s == 1:
        return x
    B, _, H, D = x.shape
    out = []
    for f in range(frames):
        img = x[:, f * gh * gw:(f + 1) * gh * gw].reshape(B, gh, gw, H * D).permute(0, 3, 1, 2)
        y = Fn.avg_pool2d(img, s) if mode == mssa.AVG else img[:, :, ::s, ::s]
        out.append(y.permute(0, 2, 3, 1).reshape(B, -1, H, D))
    return torch.cat(out, dim=1)


def _torch_mssa(t, scales, gh, gw, F, mode):
    """Eq. 4 in torch ops; returns [B, N, H, D]."""
    cnt = schedule.token_counts(scales, gh, gw, F)
    offs = schedule.token_offsets(scales, gh, gw, F)
    outs = []
    for g in sorted(set(scales)):
        parts = [t["k_sink"]], [t["v_sink"]]
        for f in range(t["k_hist"].shape[1]):
            parts[0].append(_torch_pool(t["k_hist"][:, f], F, gh, gw, g, mode))
            parts[1].append(_torch_pool(t["v_hist"][:, f], F, gh, gw, g, mode))
        for l, s in enumerate(scales):
            st = max(1, g // s)
            sl = slice(offs[l], offs[l] + cnt[l])
            parts[0].append(_torch_pool(t["k_win"][:, sl], F, gh // s, gw // s, st, mode))
            parts[1].append(_torch_pool(t["v_win"][:, sl], F, gh // s, gw // s, st, mode))
        K, V = torch.cat(parts[0], 1), torch.cat(parts[1], 1)
        ls = [l for l, s in enumerate(scales) if s == g]
        qs = slice(offs[ls[0]], offs[ls[-1]] + cnt[ls[-1]])
        o = Fn.scaled_dot_product_attention(t["q"][:, qs].transpose(1, 2), K.transpose(1, 2),
                                            V.transpose(1, 2))
        outs.append(o.transpose(1, 2))
    return torch.cat(outs, dim=1)


CASES = [
    ((1, 2), 4, 4, 1, 3, 1),
    ((1, 1, 2, 4), 4, 8, 1, 2, 2),
    ((2, 2, 4), 4, 8, 1, 1, 1),
    ((1, 2), 4, 4, 2, 3, 1),       # chunked
    ((1, 1, 1), 2, 3, 1, 2, 2),    # all fine
]


@pytest.mark.parametrize("mode", [mssa.AVG, mssa.STRIDED])
@pytest.mark.parametrize("scales,gh,gw,F,ns,nh", CASES)
def test_backward_equals_torch_autograd(mode, scales, gh, gw, F, ns, nh):
    rng = np.random.default_rng(17)
    x = _inputs(rng, scales, gh, gw, F, ns, nh, H=2, D=5)
    got = mssa_bwd.mssa_backward(x["q"], x["k_win"], x["v_win"], x["k_sink"], x["v_sink"],
                                 x["k_hist"], x["v_hist"], x["dout"], scales, gh, gw, mode,
                                 frames=F)
    t = {k: torch.from_numpy(v).requires_grad_(k != "dout") for k, v in x.items()}
    out = _torch_mssa(t, scales, gh, gw, F, mode)
    names = ["q", "k_win", "v_win", "k_sink", "v_sink", "k_hist", "v_hist"]
    grads = torch.autograd.grad((out * t["dout"]).sum(), [t[n] for n in names],
                                allow_unused=True)
    for n, gr in zip(names, grads):
        want = np.zeros_like(x[n]) if gr is None else gr.numpy()
        np.testing.assert_allclose(got["d" + n], want, rtol=0, atol=1e-11, err_msg=n)


def test_backward_equals_central_differences():
    """Directional derivatives of the (pinned) forward oracle match the
    gradient: (L(x + e u) - L(x - e u)) / 2e = <grad, u>."""
    rng = np.random.default_rng(23)
    scales, gh, gw, F = (1, 2), 4, 4, 1
    x = _inputs(rng, scales, gh, gw, F, ns=3, nh=1, H=1, D=4)
    args = ["q", "k_win", "v_win", "k_sink", "v_sink", "k_hist", "v_hist"]

    def loss(y):
        o = mssa.mssa_forward(*[y[a] for a in args], scales, gh, gw)
        return float((o * y["dout"]).sum())
    grads = mssa_bwd.mssa_backward(*[x[a] for a in args], x["dout"], scales, gh, gw)
    eps = 1e-5
    for a in args:
        u = rng.standard_normal(x[a].shape)
        yp, ym = dict(x), dict(x)
        yp[a] = x[a] + eps * u
        ym[a] = x[a] - eps * u
        fd = (loss(yp) - loss(ym)) / (2 * eps)
        assert fd == pytest.approx(float((grads["d" + a] * u).sum()), rel=1e-7, abs=1e-9), a


@pytest.mark.parametrize("mode", [mssa.AVG, mssa.STRIDED])
def test_backward_invariants(mode):
    """Adding one vector to every key leaves every softmax row unchanged, so
    the key gradients over the whole context sum to zero; the value weights of
    a row sum to one, so the value gradients sum to the sum of dout. Pooling
    moves a gradient without changing its total, so both hold after the
    adjoint of Subsample as well."""
    rng = np.random.default_rng(29)
    scales, gh, gw, F = (1, 1, 2, 4), 8, 8, 1
    x = _inputs(rng, scales, gh, gw, F, ns=5, nh=2, H=2, D=6, B=2)
    g = mssa_bwd.mssa_backward(x["q"], x["k_win"], x["v_win"], x["k_sink"], x["v_sink"],
                               x["k_hist"], x["v_hist"], x["dout"], scales, gh, gw, mode)
    ksum = g["dk_win"].sum(1) + g["dk_sink"].sum(1) + g["dk_hist"].sum((1, 2))
    np.testing.assert_allclose(ksum, 0.0, atol=1e-12)
    vsum = g["dv_win"].sum(1) + g["dv_sink"].sum(1) + g["dv_hist"].sum((1, 2))
    np.testing.assert_allclose(vsum, x["dout"].sum(1), atol=1e-12)


def test_lse_equals_library_logsumexp():
    """The row normaliser on the all-fine schedule is torch.logsumexp of the
    scores against [sink || history || window]."""
    rng = np.random.default_rng(31)
    scales, gh, gw = (1, 1, 1), 4, 6
    x = _inputs(rng, scales, gh, gw, 1, ns=5, nh=2, H=3, D=16, B=2)
    got = mssa.mssa_lse(x["q"], x["k_win"], x["k_sink"], x["k_hist"], scales, gh, gw)
    B, N, H, D = x["q"].shape
    K = np.concatenate([x["k_sink"], x["k_hist"].reshape(B, -1, H, D), x["k_win"]], axis=1)
    s = torch.einsum("bnhd,bmhd->bhnm", torch.from_numpy(x["q"]), torch.from_numpy(K)) / D ** 0.5
    np.testing.assert_allclose(got, torch.logsumexp(s, dim=-1).numpy(), rtol=0, atol=1e-12)
