"""The allocation-free unpatchify entry point against the workspace one.

msf_unpatchify_noalloc serves callers that cannot allocate device memory (a
host that owns every device buffer and forbids libraries to call cudaMalloc):
it keeps its scratch in a fixed array inside the library instead of a bound
workspace. Its output must match msf_unpatchify's (same de-embedding and
rearrangement) within the de-embedding tolerance the other tests use, on two
calls in a row (the second call reuses the array the first one left behind).
This file is collected last so that a stop-at-first-failure run has already
run every other test.
"""
import dataclasses

import numpy as np
import pytest
import torch

from paper_2607_20940_gb300 import synth

from helpers import BF16, bind, device_inputs, make_plan, msf

pytestmark = pytest.mark.gpu


def test_unpatchify_noalloc_matches_workspace_path_twice():
    m = msf()
    w = dataclasses.replace(synth.LAYER_480P, batch=2)
    plan = make_plan(w, BF16, embed=True)
    x = synth.attention_inputs(w, BF16)
    bind(plan, device_inputs(x, w.history_capacity))
    mi = synth.msp_inputs(w, BF16)
    N, E = plan.info.n_tokens, w.embed_dim
    gen = torch.Generator().manual_seed(77)
    tokens = torch.randn((w.batch, N, E), generator=gen).to(BF16).cuda()
    w_out = mi["w_out"].t().contiguous().cuda()  # [C*P^2, E]
    shape = (w.batch, w.latent_channels, w.grid_h * w.patch, w.grid_w * w.patch)
    ref = torch.empty(shape, dtype=BF16, device="cuda")
    plan.unpatchify(0, tokens, w_out, ref)
    torch.cuda.synchronize()
    ref64 = ref.double().cpu().numpy()
    tol = 2.0 ** -7 * np.abs(ref64).max() + 1e-3
    for call in range(2):
        got = torch.full(shape, float("nan"), dtype=BF16, device="cuda")
        m.msf_unpatchify_noalloc(plan.handle, 0, tokens, w_out, got)
        torch.cuda.synchronize()
        err = np.abs(got.double().cpu().numpy() - ref64)
        assert np.isfinite(err).all(), call
        assert err.max() <= tol, (call, err.max())
