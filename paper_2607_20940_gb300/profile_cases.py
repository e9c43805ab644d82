"""Profiling driver: runs one kernel family of the window pass on seeded
synthetic inputs so that `ncu -k <kernel>` can capture it in isolation.

    python -m paper_2607_20940_gb300.profile_cases pool     # K/V pyramid at three sizes
    python -m paper_2607_20940_gb300.profile_cases pool_fused  # pyramid + staged history head
    python -m paper_2607_20940_gb300.profile_cases embed    # MSP patchify + tier embedding
    python -m paper_2607_20940_gb300.profile_cases deembed  # de-embedding + unpatchify
    python -m paper_2607_20940_gb300.profile_cases embed_pool  # embedding + pyramid, one launch
    python -m paper_2607_20940_gb300.profile_cases tier     # coarse-tier modules (LoRA, residual)
    python -m paper_2607_20940_gb300.profile_cases backward # forward with lse + MSSA gradient
    python -m paper_2607_20940_gb300.profile_cases attention # MSSA forward, 480p layer

Each case runs twice after an L2 flush (a 256 MiB write) and checks the
device status word. Nothing here is timed; the numbers come from the
profiler.
"""
from __future__ import annotations

import sys

import torch

from paper_2607_20940_gb300 import msf, synth


def _setup(w, embed=False, fused=False):
    dev = torch.device("cuda", 0)
    x = synth.attention_inputs(w)
    plan = msf.Plan(msf.make_desc(w.scales, w.grid_h, w.grid_w, w.heads, w.head_dim, w.sink_tokens,
                                  w.history_frames, w.history_capacity, batch=w.batch,
                                  latent_channels=w.latent_channels, patch=w.patch,
                                  embed_dim=w.embed_dim if embed else 0, fused_append=int(fused)))
    d = {k: v.to(dev) for k, v in x.items()}
    for k in ("k_hist", "v_hist"):
        slots = w.history_capacity + 1 if fused else max(w.history_capacity, 1)
        ring = torch.zeros((w.batch, slots) + tuple(d[k].shape[2:]),
                           dtype=d[k].dtype, device=dev)
        ring[:, :w.history_frames] = d[k]
        d[k] = ring
    ws = plan.workspace(dev)
    plan.bind(ws, d["k_sink"], d["v_sink"], d["k_hist"], d["v_hist"])
    return plan, d, ws


def run(case: str) -> None:
    dev = torch.device("cuda", 0)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    if case == "pool":
        for w, mode in ((synth.LAYER_480P, msf.MSF_RESAMPLE_WINDOW_ONLY),
                        (synth.STREAM_480P, msf.MSF_RESAMPLE_WINDOW_ONLY),
                        (synth.THREE_SCALE, msf.MSF_RESAMPLE_FULL)):
            plan, d, _ = _setup(w)
            for _ in range(2):
                flush.fill_(1)
                plan.kv_resample(d["k_win"], d["v_win"], mode)
            torch.cuda.synchronize()
            assert plan.device_status() == msf.MSF_OK
            plan.close()
    elif case == "pool_fused":
        for w in (synth.LAYER_480P, synth.STREAM_480P):
            plan, d, _ = _setup(w, fused=True)
            for _ in range(2):
                flush.fill_(1)
                plan.kv_resample(d["k_win"], d["v_win"], msf.MSF_RESAMPLE_WINDOW_ONLY)
            torch.cuda.synchronize()
            assert plan.device_status() == msf.MSF_OK
            plan.close()
    elif case in ("embed", "deembed"):
        for w in (synth.LAYER_480P, synth.STREAM_480P):
            plan, d, _ = _setup(w, embed=True)
            mi = synth.msp_inputs(w)
            lat = mi["latent"].to(dev)
            tiers = {s: mi["w_tier"][s].t().contiguous().to(dev) for s in set(w.scales)}
            w_out = mi["w_out"].t().contiguous().to(dev)
            N, E = plan.info.n_tokens, w.embed_dim
            tok = torch.randn((w.batch, N, E), device=dev).to(torch.bfloat16)
            lat_out = torch.empty((w.batch, w.latent_channels, w.grid_h * w.patch, w.grid_w * w.patch),
                                  dtype=torch.bfloat16, device=dev)
            for _ in range(2):
                flush.fill_(1)
                if case == "embed":
                    plan.patchify(lat, [tiers[s] for s in w.scales], tok)
                else:
                    plan.unpatchify(0, tok, w_out, lat_out)
            torch.cuda.synchronize()
            assert plan.device_status() == msf.MSF_OK
            plan.close()
    elif case == "embed_pool":
        # the one-launch MSP embedding + window pyramid with the staged head
        for w in (synth.LAYER_480P, synth.STREAM_480P):
            plan, d, _ = _setup(w, embed=True, fused=True)
            mi = synth.msp_inputs(w)
            lat = mi["latent"].to(dev)
            tiers = {s: mi["w_tier"][s].t().contiguous().to(dev) for s in set(w.scales)}
            tok = torch.empty((w.batch, plan.info.n_tokens, w.embed_dim), dtype=torch.bfloat16, device=dev)
            for _ in range(2):
                flush.fill_(1)
                plan.patchify_resample(lat, [tiers[s] for s in w.scales], tok, d["k_win"], d["v_win"],
                                       msf.MSF_RESAMPLE_WINDOW_ONLY)
            torch.cuda.synchronize()
            assert plan.device_status() == msf.MSF_OK
            plan.close()
    elif case == "tier":
        # coarse-tier modules: rank-32 LoRA on embedding and de-embedding, latent residual
        w = synth.LAYER_480P
        plan, d, _ = _setup(w, embed=True)
        mi = synth.msp_inputs(w)
        ti = synth.tier_inputs(w, 32)
        lat = mi["latent"].to(dev)
        keep, mods = [], {}
        for s in sorted(set(w.scales)):
            w_emb = mi["w_tier"][s].t().contiguous().to(dev)
            if s == 1:
                w_o = mi["w_out"].t().contiguous().to(dev)
                mods[s] = msf.tier_module(w_emb, w_o)
                keep += [w_emb, w_o]
                continue
            t = {k: (v.t().contiguous().to(dev) if torch.is_tensor(v) else v) for k, v in ti[s].items()}
            mods[s] = msf.tier_module(w_emb, t["w_out"], embed_down=t["lora_a"], embed_up=t["lora_b"],
                                      out_down=t["out_a"], out_up=t["out_b"], residual=t["residual"],
                                      lora_rank=32, lora_scale=t["gamma"])
            keep += [w_emb] + [v for v in t.values() if torch.is_tensor(v)]
        tok = torch.empty((w.batch, plan.info.n_tokens, w.embed_dim), dtype=torch.bfloat16, device=dev)
        lat_out = torch.empty((w.batch, w.latent_channels, w.grid_h * w.patch, w.grid_w * w.patch),
                              dtype=torch.bfloat16, device=dev)
        for _ in range(2):
            flush.fill_(1)
            plan.patchify_tiers(lat, [mods[s] for s in w.scales], tok)
            plan.unpatchify_tier(2, tok, lat, mods[2], lat_out)
        torch.cuda.synchronize()
        assert plan.device_status() == msf.MSF_OK
        plan.close()
    elif case == "attention":
        w = synth.LAYER_480P
        plan, d, _ = _setup(w)
        out = torch.empty_like(d["q"])
        plan.kv_resample(d["k_win"], d["v_win"])
        for _ in range(2):
            flush.fill_(1)
            plan.mssa_forward(d["q"], d["k_win"], d["v_win"], out)
        torch.cuda.synchronize()
        assert plan.device_status() == msf.MSF_OK
        plan.close()
    elif case == "backward":
        w = synth.LAYER_480P
        plan, d, _ = _setup(w)
        B, N, H = w.batch, plan.info.n_tokens, w.heads
        lse = torch.empty((B, H, N), dtype=torch.float32, device=dev)
        out = torch.empty_like(d["q"])
        dout = torch.randn(d["q"].shape, device=dev).to(torch.bfloat16)
        grads = [torch.empty_like(d["q"]) for _ in range(3)]
        bws = plan.backward_workspace(dev)
        plan.kv_resample(d["k_win"], d["v_win"])
        for _ in range(2):
            flush.fill_(1)
            plan.mssa_forward_lse(d["q"], d["k_win"], d["v_win"], out, lse)
            plan.mssa_backward(d["q"], d["k_win"], d["v_win"], out, dout, lse, *grads, bws)
        torch.cuda.synchronize()
        assert plan.device_status() == msf.MSF_OK
        plan.close()
    else:
        raise SystemExit(f"unknown case {case!r}: pool, pool_fused, embed, embed_pool, deembed, tier, "
                         "backward or attention")


if __name__ == "__main__":
    run(sys.argv[1] if len(sys.argv) > 1 else "pool")
