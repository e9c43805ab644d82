"""The allocation-free unpatchify entry point against the workspace one.

msf_unpatchify_noalloc serves callers that cannot allocate device memory (a
host that owns every device buffer and forbids libraries to call cudaMalloc):
it keeps its scratch in a fixed array inside the library instead of a bound
workspace. Its output must match msf_unpatchify's (same de-embedding and
rearrangement) within the de-embedding tolerance the other tests use, on two
calls in a row (the second call reuses the array the first one left behind),
and the fp64 oracle's de-embedding of the same tokens. The cases cover the
fine tier (64 features, split-K), a coarse tier (256 features, the 128-column
split kernel), a batch large enough that the array leaves room for one split
only (direct GEMM output), the rejection of a problem beyond the array, and
the array's own device status word (a bounded wait that runs out is reported
by msf_noalloc_device_status, and the entry point still works afterwards).
This file is collected last so that a stop-at-first-failure run has already
run every other test.
"""
import dataclasses

import numpy as np
import pytest
import torch

from oracle import msp as omsp
from paper_2607_20940_gb300 import synth

from helpers import BF16, make_plan, msf

pytestmark = pytest.mark.gpu


def _check_noalloc(w, position, calls=2):
    """Workspace path, then `calls` no-alloc calls, each against the workspace
    output and the oracle's de-embedding of the same bf16 tokens."""
    m = msf()
    plan = make_plan(w, BF16, embed=True)
    info = plan.info
    N, E, C = info.n_tokens, w.embed_dim, w.latent_channels
    P = w.patch * w.scales[position]
    gen = torch.Generator().manual_seed(77 + position)
    tokens_h = torch.randn((w.batch, N, E), generator=gen).to(BF16)
    w_out_h = (torch.randn((E, C * P * P), generator=gen) * E ** -0.5).to(BF16)  # [E, C*P^2]
    tokens = tokens_h.cuda()
    w_out = w_out_h.t().contiguous().cuda()  # the C ABI takes [C*P^2, E]
    shape = (w.batch, C, w.grid_h * w.patch, w.grid_w * w.patch)
    # The workspace path needs a bound plan (its attention buffers stay unused).
    sink = torch.zeros((w.batch, w.sink_tokens, w.heads, w.head_dim), dtype=BF16, device="cuda")
    ring = torch.zeros((w.batch, max(w.history_capacity, 1), w.grid_h * w.grid_w, w.heads,
                        w.head_dim), dtype=BF16, device="cuda")
    plan.bind(plan.workspace(), sink, sink, ring, ring)
    ref = torch.empty(shape, dtype=BF16, device="cuda")
    plan.unpatchify(position, tokens, w_out, ref)
    torch.cuda.synchronize()
    assert plan.device_status() == m.MSF_OK
    ref64 = ref.double().cpu().numpy()
    o0, n = info.state_offset[position], info.state_tokens[position]
    ora = omsp.unpatchify_state(synth.to_f64(tokens_h[:, o0:o0 + n]), P, C, shape[2], shape[3],
                                w_out=synth.to_f64(w_out_h))
    tol = 2.0 ** -7 * np.abs(ora).max() + 1e-3
    assert np.abs(ref64 - ora).max() <= tol
    for call in range(calls):
        got = torch.full(shape, float("nan"), dtype=BF16, device="cuda")
        m.msf_unpatchify_noalloc(plan.handle, position, tokens, w_out, got)
        torch.cuda.synchronize()
        g = got.double().cpu().numpy()
        assert np.isfinite(g).all(), call
        assert np.abs(g - ref64).max() <= tol, (call, np.abs(g - ref64).max())
        assert np.abs(g - ora).max() <= tol, (call, np.abs(g - ora).max())
    assert m.msf_noalloc_device_status() == m.MSF_OK


def test_unpatchify_noalloc_matches_workspace_path_twice():
    _check_noalloc(dataclasses.replace(synth.LAYER_480P, batch=2, heads=2), 0)


def test_unpatchify_noalloc_coarse_tier():
    # position 2 has scale 2: 256 features per token, the 128-column GEMM tiles
    _check_noalloc(dataclasses.replace(synth.LAYER_480P, batch=2, heads=2), 2)


def test_unpatchify_noalloc_single_split():
    # 9 streams of 16x60x104: the raw tokens take 1.8 MB of the 8 MiB array and
    # leave room for one fp32 partial set only, so the GEMM writes bf16 directly.
    _check_noalloc(dataclasses.replace(synth.LAYER_480P, batch=9, heads=1), 0, calls=2)


def test_unpatchify_noalloc_rejects_problem_beyond_its_array():
    m = msf()
    w = dataclasses.replace(synth.LAYER_480P, batch=43, heads=1)  # 43 x 200 KB > 8 MiB
    plan = make_plan(w, BF16, embed=True)
    dummy = torch.zeros(64, dtype=BF16, device="cuda")
    st = m._lib.msf_unpatchify_noalloc(plan.handle, 0, dummy.data_ptr(), dummy.data_ptr(),
                                       dummy.data_ptr(), m._stream(None))
    assert st == m.MSF_ERR_UNSUPPORTED


def test_noalloc_status_word_reports_timeout():
    m = msf()
    assert m.msf_noalloc_device_status() == m.MSF_OK
    m.msf_noalloc_selftest_wait_timeout(200_000)  # ~0.1 ms of SM clock
    assert m.msf_noalloc_device_status() == m.MSF_ERR_TIMEOUT
    assert m.msf_noalloc_device_status() == m.MSF_OK  # the read clears it
    with pytest.raises(Exception):
        m.msf_noalloc_selftest_wait_timeout(0)
    _check_noalloc(dataclasses.replace(synth.LAYER_480P, batch=2, heads=2), 0, calls=1)
