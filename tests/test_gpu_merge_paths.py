"""The three ways the tensor-core attention merges an item cut into pieces.

The persistent attention kernel splits the tile sequence of the query blocks
that do not fill whole rounds over its CTAs (stream-K); each split block's
pieces are combined by the piece that finishes last. By construction of the
schedule (152 persistent CTAs on a GB300, fewer when the sequence is short):

* tiny window (2 heads, 4 blocks): no whole rounds, each block cut into at
  most 8 pieces -> the merger keeps its own piece in TMEM and merges in place;
* one head over a 3072-row context (2 blocks of 24 K/V tiles, ~58 CTAs):
  blocks cut into more than 8 pieces -> the merger reads every piece's
  partial result from its slot;
* the 480p layer (156 fine-group blocks >= 152 CTAs), and a head_dim-64
  window with 160: one whole round, the rest split -> the merge runs on the
  helper warps beside the whole blocks.

Each case is checked against the fp64 oracle and for run-to-run
reproducibility: pieces are combined in a fixed order whichever CTA merges,
so two launches give the same bits.
"""
import pytest
import torch

from paper_2607_20940_gb300 import synth

from helpers import BF16, bind, device_inputs, err_stats, make_plan, oracle_mssa

pytestmark = pytest.mark.gpu

# One head, two fine states of 16x16 tokens, a 2048-token sink and two history
# frames: query blocks of 256 rows over a 3072-row context (24 K/V tiles).
LONG_CTX = synth.Workload("long_ctx_h1_t2_16x16_sink2048", 2, (1, 1), 16, 16, 1, 128, 2048, 2, 2, 1, 11)
# head_dim 64 with whole rounds: 16 heads x 10 fine-group blocks = 160 >= 152.
HELPER_D64 = synth.Workload("helper_d64_t3_32x40_h16", 3, (1, 1, 2), 32, 40, 16, 64, 1280, 1, 1, 1, 12)


@pytest.mark.parametrize("w,heads", [
    (synth.TINY, None),
    (LONG_CTX, None),
    (synth.LAYER_480P, [0, 7]),
    (HELPER_D64, [0, 15]),
], ids=["in_place", "from_slots", "helper_warps", "helper_warps_d64"])
def test_split_merge_paths(w, heads):
    x = synth.attention_inputs(w, BF16)
    plan = make_plan(w, BF16)
    dx = device_inputs(x, w.history_capacity)
    bind(plan, dx)
    plan.kv_resample(dx["k_win"], dx["v_win"])
    outs = []
    for _ in range(2):
        out = torch.full_like(dx["q"], float("nan"))
        plan.mssa_forward(dx["q"], dx["k_win"], dx["v_win"], out)
        torch.cuda.synchronize()
        outs.append(out)
    assert plan.device_status() == 0
    assert torch.equal(outs[0], outs[1])
    ref = oracle_mssa(x, w, heads=heads)
    mx, mean = err_stats(outs[0], ref, heads)
    assert mx <= 2e-2 and mean <= 2e-3, (mx, mean)


def test_output_16_byte_aligned():
    """An output that is 16-byte but not 32-byte aligned (the ABI asks for 16)
    takes the 16-byte store path of the whole-block epilogue (the 480p layer
    has whole blocks); the result is the same as with an aligned output, bit
    for bit, and nothing is written outside the output."""
    w = synth.LAYER_480P
    x = synth.attention_inputs(w, BF16)
    plan = make_plan(w, BF16)
    dx = device_inputs(x, w.history_capacity)
    bind(plan, dx)
    plan.kv_resample(dx["k_win"], dx["v_win"])
    aligned = torch.empty_like(dx["q"])
    plan.mssa_forward(dx["q"], dx["k_win"], dx["v_win"], aligned)
    n = dx["q"].numel()
    buf = torch.full((n + 16,), float("nan"), dtype=BF16, device="cuda")
    assert buf.data_ptr() % 32 == 0
    shifted = buf[8:8 + n].view(dx["q"].shape)  # 16 bytes past a 32-byte boundary
    plan.mssa_forward(dx["q"], dx["k_win"], dx["v_win"], shifted)
    torch.cuda.synchronize()
    assert plan.device_status() == 0
    assert torch.equal(aligned, shifted)
    assert torch.isnan(buf[:8]).all() and torch.isnan(buf[8 + n:]).all()
