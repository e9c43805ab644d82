"""Static multi-scale schedule: token counts (Eq. 3), MSSA contexts (Eq. 4)
and the attention-pair reduction (Eq. 5). Test infrastructure; fp64/int only.

Notation follows Sec. 4.1: window positions l = 1..T carry patch sizes
p_l = s_l * p with s_l in {1, 2, 4, ...}, non-decreasing in l. A latent frame
tokenised at the native patch p gives a fine Gh x Gw grid; at p_l it gives a
(Gh/s_l) x (Gw/s_l) grid, so N_l = Gh*Gw / s_l^2 (Eq. 3).

Chunked states (Sec. 5.1: each window state is a chunk of F latent frames):
patchification is spatial, so a state holds F such grids, N_l = F*Gh*Gw/s_l^2,
its tokens ordered (latent frame, row, col). Every per-frame count above is
multiplied by F; ``frames`` defaults to 1 (one latent frame per state).
"""
from __future__ import annotations

from fractions import Fraction
from typing import List, NamedTuple, Sequence, Tuple

# Kinds of context rows, used by the index maps.
SINK, HIST, WIN = 0, 1, 2


def validate(scales: Sequence[int], grid_h: int, grid_w: int) -> None:
    """The schedule Sec. 4.1 allows: p_1 <= ... <= p_T, p_l in {p, 2p, 4p, ...}.
    A grid the coarsest stride does not divide has no defined coarse grid."""
    if len(scales) == 0:
        raise ValueError("empty schedule")
    for s in scales:
        if s < 1 or (s & (s - 1)) != 0:
            raise ValueError(f"scale {s} is not a power of two")
    for a, b in zip(scales, scales[1:]):
        if b < a:
            raise ValueError("scales must be non-decreasing along the window")
    smax = max(scales)
    if grid_h % smax or grid_w % smax:
        raise ValueError("grid not divisible by the coarsest scale")


def state_grid(grid_h: int, grid_w: int, s: int) -> Tuple[int, int]:
    return grid_h // s, grid_w // s


def token_counts(scales: Sequence[int], grid_h: int, grid_w: int, frames: int = 1) -> List[int]:
    """N_l^MSP = HW / p_l^2 (Eq. 3) per latent frame, in tokens of the fine
    grid Gh x Gw; a chunk of F frames has F times as many."""
    return [frames * ((grid_h // s) * (grid_w // s)) for s in scales]


def token_offsets(scales, grid_h, grid_w, frames: int = 1) -> List[int]:
    """Start of state l's tokens in the window sequence (states in position order)."""
    out, acc = [], 0
    for n in token_counts(scales, grid_h, grid_w, frames):
        out.append(acc)
        acc += n
    return out


def rho_tok(scales: Sequence[int]) -> Fraction:
    """rho_tok = (1/T) sum_l (p/p_l)^2 (Eq. 3), exact."""
    T = len(scales)
    return sum((Fraction(1, s * s) for s in scales), Fraction(0)) / T


def token_of(scales, grid_h, grid_w, l: int, i: int, j: int, f: int = 0, frames: int = 1) -> int:
    """Index of token (row i, col j) of latent frame f of state l (0-based) in
    the window sequence."""
    gh, gw = grid_h // scales[l], grid_w // scales[l]
    return token_offsets(scales, grid_h, grid_w, frames)[l] + (f * gh + i) * gw + j


class Group(NamedTuple):
    scale: int          # g: the query scale of this group
    states: Tuple[int, ...]  # 0-based window positions whose s_l == g
    q_begin: int        # first query token (window order)
    q_end: int          # one past the last


def query_groups(scales, grid_h, grid_w, frames: int = 1) -> List[Group]:
    """Queries that share one context: all tokens of states with equal s_l."""
    offs = token_offsets(scales, grid_h, grid_w, frames)
    cnt = token_counts(scales, grid_h, grid_w, frames)
    groups = []
    for g in sorted(set(scales)):
        st = tuple(l for l, s in enumerate(scales) if s == g)
        groups.append(Group(g, st, offs[st[0]], offs[st[-1]] + cnt[st[-1]]))
    return groups


def context_rows(scales, grid_h, grid_w, sink_tokens: int, n_hist: int, g: int, frames: int = 1):
    """The rows of C_a^MSSA (Eq. 4) for queries of scale g, in context order.

    Each row is (kind, frame, stride, row, col): kind SINK has frame 0,
    stride 1, row = sink token, col 0; kind HIST has frame = history slot and
    (row, col) on the (Gh/st) x (Gw/st) grid of that frame pooled by
    st = g (history is fine, p_b = p); kind WIN has frame = window position l
    and (row, col) on the grid of state l pooled by st = max(1, g / s_l).
    For chunked states each history frame and window state holds F latent
    frames, each subsampled on its own; latent frame f's grid rows are
    numbered f*gh .. f*gh + gh - 1 (gh the rows of one pooled frame).
    """
    rows = []
    for n in range(sink_tokens):
        rows.append((SINK, 0, 1, n, 0))
    for f in range(n_hist):
        st = max(1, g // 1)
        gh, gw = grid_h // st, grid_w // st
        for lf in range(frames):
            for i in range(gh):
                for j in range(gw):
                    rows.append((HIST, f, st, lf * gh + i, j))
    for l, s in enumerate(scales):
        st = max(1, g // s)
        gh, gw = grid_h // (s * st), grid_w // (s * st)
        for lf in range(frames):
            for i in range(gh):
                for j in range(gw):
                    rows.append((WIN, l, st, lf * gh + i, j))
    return rows


def context_length(scales, grid_h, grid_w, sink_tokens, n_hist, g, frames: int = 1) -> int:
    return len(context_rows(scales, grid_h, grid_w, sink_tokens, n_hist, g, frames))


def attention_pairs(scales, grid_h, grid_w, sink_tokens, n_hist, frames: int = 1) -> int:
    """Query-key pairs MSSA evaluates per (stream, head): sum_g Nq_g * Nkv_g."""
    tot = 0
    for grp in query_groups(scales, grid_h, grid_w, frames):
        nq = grp.q_end - grp.q_begin
        tot += nq * context_length(scales, grid_h, grid_w, sink_tokens, n_hist, grp.scale, frames)
    return tot


def msp_only_pairs(scales, grid_h, grid_w, sink_tokens, n_hist, frames: int = 1) -> int:
    """Pairs when every query sees the un-resampled context (MSP without MSSA):
    each of the N_MSP queries against sink + fine history + all window tokens."""
    n = sum(token_counts(scales, grid_h, grid_w, frames))
    return n * (sink_tokens + n_hist * frames * grid_h * grid_w + n)


def attention_flops(scales, grid_h, grid_w, sink_tokens, n_hist, heads, head_dim, batch=1,
                    frames: int = 1) -> int:
    """Algorithmic FLOPs: 2 for each multiply-add of Q K^T and of P V."""
    return 4 * head_dim * heads * batch * attention_pairs(scales, grid_h, grid_w, sink_tokens,
                                                          n_hist, frames)


def r_mssa_eq5(scales: Sequence[int], n_sink_frames: int, n_hist: int) -> Fraction:
    """Eq. 5 as printed: eta_l = (p/p_l)^2, s_ab = max(1, p_a/p_b), V(a) = all
    history frames (fine, eta = 1) and all window positions. The sink frames
    contribute the leading term (one per sink frame)."""
    eta = [Fraction(1, s * s) for s in scales]
    num = Fraction(0)
    den = Fraction(0)
    for a, sa in enumerate(scales):
        vis = [(Fraction(1), 1)] * n_hist + [(eta[b], sb) for b, sb in enumerate(scales)]
        inner_num = Fraction(n_sink_frames)
        inner_den = Fraction(n_sink_frames)
        for eb, sb in vis:
            sab = max(1, sa // sb)
            inner_num += eb / (sab * sab)
            inner_den += eb
        num += eta[a] * inner_num
        den += eta[a] * inner_den
    return 1 - num / den
