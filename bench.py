"""Benchmark of the Ms. Forcing MSSA window pass on GB300.

A step is one rolling-window pass of the whole hot path at the 480p layer
shapes (T=5, 30x52 fine grid, scales (1,1,2,2,2), 12 heads of 128, sink 1560
tokens, history ring of 2 frames):
  MSP patchify + tier embedding of the 5 latent states (16x60x104 -> 4290x1536)
  -> window part of the K/V pyramid, with the head's K/V staged in the history
     ring's spare slot and pooled (the history update, folded into that launch)
  -> MSSA attention (Eq. 4) -> history commit (host) -> de-embed + unpatchify
     of the head state.
The MSP embedding and the K/V pyramid go out as one launch (the pooling CTAs
take the SM slots the embedding tiles leave free); attention follows it on the
same stream.
`value` is the MSSA FLOPs the schedule requires (4*D*H*sum_g Nq_g*Nkv_g =
202.79 GFLOP) divided by the device time of the whole step, in TFLOP/s.
Inputs are resident in HBM; the L2 is flushed (a 256 MiB write) between
timed steps, outside the timed events. The CPU-baseline leg (rank 0, one GPU) times
the oracle and also compares the attention kernel's output for the same
inputs with the oracle's, element by element (`parity`).

Usage: python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]
Under torchrun every rank runs its own stream of windows (weak scaling);
rank 0 prints one JSON line.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "MSSA TFLOP/s and µs per window-pass layer (bf16, 1 GB300); % of tensor peak"
UNIT = "TFLOP/s"
FLUSH_BYTES = 256 << 20


def _dist():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def _peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return d, "measured"
    except Exception:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}, "fallback"


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled during the timed region."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = os.path.join("/tmp", f"msf_clocks_{os.getpid()}.csv")

    def start(self):
        try:
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=self.f, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.f.close()
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    sm.append(float(parts[1]))
                    mx = float(parts[2])
                except ValueError:
                    continue
                for n, v in zip(names, parts[5:9]):
                    if v.lower() == "active":
                        reasons.add(n)
        try:
            os.remove(self.path)
        except OSError:
            pass
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": mx,
                "reasons": sorted(reasons), "samples": len(sm)}


def _host_info() -> dict:
    """The host the oracle runs on: CPU model, logical cores, and the thread
    count of the BLAS that numpy's fp64 matmuls use (read from the loaded
    OpenBLAS itself), with OMP_NUM_THREADS / OPENBLAS_NUM_THREADS as set."""
    import ctypes
    import re

    import numpy  # noqa: F401  (loads its BLAS)
    model = None
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.strip().lower().startswith("model name"):
                model = line.split(":", 1)[1].strip()
                break
    except (OSError, subprocess.SubprocessError):
        pass
    if model is None:
        try:
            with open("/proc/cpuinfo") as f:
                for line in f:
                    if line.lower().startswith("model name"):
                        model = line.split(":", 1)[1].strip()
                        break
        except OSError:
            pass
    blas, threads = None, None
    try:
        with open("/proc/self/maps") as f:
            libs = sorted(set(re.findall(r"/\S*openblas\S*\.so\S*", f.read())))
        for path in libs:
            lib = ctypes.CDLL(path)
            for sym in ("scipy_openblas_get_num_threads64_", "openblas_get_num_threads64_",
                        "scipy_openblas_get_num_threads", "openblas_get_num_threads"):
                fn = getattr(lib, sym, None)
                if fn is not None:
                    fn.restype = ctypes.c_int
                    blas, threads = os.path.basename(path), int(fn())
                    break
            if threads is not None:
                break
    except OSError:
        pass
    return {"cpu_model": model, "logical_cores": os.cpu_count(), "blas": blas,
            "blas_threads": threads, "OMP_NUM_THREADS": os.environ.get("OMP_NUM_THREADS"),
            "OPENBLAS_NUM_THREADS": os.environ.get("OPENBLAS_NUM_THREADS")}


def max_over_ranks(value: float, device) -> float:
    """The largest per-rank time (the job ends when the slowest rank ends)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return value
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def _oracle_step(w, x, m, heads=None):
    """The oracle's version of one step (patchify+embed, MSSA, de-embed+unpatchify
    of the head state, history append as a copy)."""
    import numpy as np

    from oracle import msp as omsp
    from oracle import mssa as omssa
    from paper_2607_20940_gb300 import synth
    f = synth.to_f64
    tiers = {s: f(m["w_tier"][s]) for s in set(w.scales)}
    omsp.patchify_window(f(m["latent"]), w.scales, w.patch, tiers)
    out = omssa.mssa_forward(f(x["q"]), f(x["k_win"]), f(x["v_win"]), f(x["k_sink"]),
                             f(x["v_sink"]), f(x["k_hist"]), f(x["v_hist"]), w.scales, w.grid_h,
                             w.grid_w, heads=heads)
    G = w.grid_h * w.grid_w
    if heads is None:
        head_tok = out[:, :G].reshape(w.batch, G, -1)
        omsp.unpatchify_state(head_tok, w.patch, w.latent_channels, w.grid_h * w.patch,
                              w.grid_w * w.patch, f(m["w_out"]))
    np.copy(f(x["k_win"])[:, :G])
    return out


def run_reference(args, w):
    """The oracle (fp64 numpy) on the host cores, same workload and metric.
    Each step computes 3 of the 12 heads of the layer (a bounded sample);
    FLOPs are counted for the heads computed."""
    import torch

    from oracle import schedule
    from paper_2607_20940_gb300 import synth
    x = synth.attention_inputs(w, torch.bfloat16)
    m = synth.msp_inputs(w, torch.bfloat16)
    heads = [0, 5, 11]
    fl = schedule.attention_flops(w.scales, w.grid_h, w.grid_w, w.sink_tokens, w.history_frames,
                                  len(heads), w.head_dim, w.batch)
    for _ in range(args.warmup):
        _oracle_step(w, x, m, heads)
    times = []
    for _ in range(args.steps):
        t0 = time.perf_counter()
        _oracle_step(w, x, m, heads)
        times.append(time.perf_counter() - t0)
    tot = sum(times)
    value = fl * args.steps / tot / 1e12
    host = _host_info()
    cores = host["blas_threads"] or os.cpu_count()
    sample = f"3 of 12 heads of the 480p layer per step (oracle fp64, numpy), {fl/1e9:.2f} GFLOP"
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * tot / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": {"workload": w.name, "kind": "oracle sample"},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                         "sample": sample, "host": host},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))


def oracle_other_configs():
    """The oracle (fp64 numpy, as it stands) on the host cores for the other
    workloads of the family: the tiny and the three-scale windows whole, the
    30-layer pass on layers 0, 15 and 29 (each: patchify + tier embedding of
    the window, MSSA on 2 of 12 heads, de-embedding + unpatchify of the head),
    and the B=4 rollout on steps 0, 1, 2, 60 and 119 of stream 0 (2 of 12
    heads; the history holds min(2 + step, 4) frames). Sampled heads, layers
    and steps are scaled up to the whole workload and marked "extrapolated"
    (the oracle's time is linear in heads, layers, streams and steps)."""
    import dataclasses

    import torch

    from oracle import msp as omsp
    from oracle import mssa as omssa
    from oracle import schedule
    from paper_2607_20940_gb300 import synth
    f = synth.to_f64

    def flops(w, n_hist, heads, batch=1):
        return schedule.attention_flops(w.scales, w.grid_h, w.grid_w, w.sink_tokens, n_hist, heads,
                                        w.head_dim, batch, w.frames)

    def attn(w, x, heads):
        t0 = time.perf_counter()
        omssa.mssa_forward(f(x["q"]), f(x["k_win"]), f(x["v_win"]), f(x["k_sink"]), f(x["v_sink"]),
                           f(x["k_hist"]), f(x["v_hist"]), w.scales, w.grid_h, w.grid_w, heads=heads,
                           frames=w.frames)
        return time.perf_counter() - t0

    res = {}
    # tiny window (T=3, 8x8, scales (1,1,2), 2 heads of 64): the whole call
    w = synth.TINY
    dt = attn(w, synth.attention_inputs(w, torch.float32), None)
    fl = flops(w, w.history_frames, w.heads)
    res["tiny"] = {"workload": w.name, "seconds": dt, "gflop": fl / 1e9, "tflops": fl / dt / 1e12,
                   "sample": "whole call (fp32 inputs)"}
    # three-scale 48x80 window: the whole call (all 16 heads)
    w = synth.THREE_SCALE
    dt = attn(w, synth.attention_inputs(w, torch.bfloat16), None)
    fl = flops(w, w.history_frames, w.heads)
    res["three_scale"] = {"workload": w.name, "seconds": dt, "gflop": fl / 1e9, "tflops": fl / dt / 1e12,
                          "sample": "whole call (all 16 heads)"}
    # 30-layer window pass: layers 0, 15, 29
    w = synth.PASS_480P
    hs = [0, 6]
    G = w.grid_h * w.grid_w
    per_layer = []
    for layer in (0, 15, 29):
        x = synth.attention_inputs(w, torch.bfloat16, seed=w.seed + layer)
        m = synth.msp_inputs(w, torch.bfloat16, seed=w.seed + layer)
        tiers = {s: f(m["w_tier"][s]) for s in set(w.scales)}
        lat, w_out = f(m["latent"]), f(m["w_out"])
        t0 = time.perf_counter()
        tok = omsp.patchify_window(lat, w.scales, w.patch, tiers)
        t_msp = time.perf_counter() - t0
        t_attn = attn(w, x, hs)
        t0 = time.perf_counter()
        omsp.unpatchify_state(tok[:, :G], w.patch, w.latent_channels, w.grid_h * w.patch,
                              w.grid_w * w.patch, w_out)
        t_msp += time.perf_counter() - t0
        per_layer.append(t_msp + t_attn * w.heads / len(hs))
    dt = statistics.mean(per_layer) * w.layers
    fl = flops(w, w.history_frames, w.heads) * w.layers
    res["window_pass_30"] = {"workload": w.name, "seconds": dt, "gflop": fl / 1e9,
                             "tflops": fl / dt / 1e12,
                             "sample": "layers 0, 15, 29 (2 of 12 heads each), extrapolated to 30 layers"}
    # B=4 streaming rollout: steps 0, 1, 2, 60, 119 of stream 0
    w = synth.STREAM_480P
    w1 = dataclasses.replace(w, batch=1)
    hs = [0, 6]
    n_hist = lambda s: min(w.history_frames + s, w.history_capacity)  # noqa: E731
    samples = {}
    for s in (0, 1, 2, 60, 119):
        x = synth.attention_inputs(w1, torch.bfloat16, seed=w.seed, history_frames=n_hist(s))
        samples[s] = attn(w1, x, hs) * w.heads / len(hs) * w.batch
    # steps 3..119 all run at capacity: the mean of the two sampled ones
    full = samples[0] + samples[1] + samples[2] + (w.steps - 3) * (samples[60] + samples[119]) / 2
    fl = sum(flops(w, n_hist(s), w.heads, w.batch) for s in range(w.steps))
    res["stream_b4"] = {"workload": w.name, "seconds": full, "gflop": fl / 1e9, "tflops": fl / full / 1e12,
                        "seconds_per_step_at_cap": samples[119],
                        "sample": "steps 0, 1, 2, 60, 119 of stream 0 (2 of 12 heads), extrapolated "
                                  "to 4 streams x 12 heads x 120 steps"}
    return res


def _parity_check(msf, w, x, ref):
    """The attention kernel's output for the step's inputs against the
    oracle's output that the CPU baseline computed for the same inputs: max and
    mean |err| over every element of the 480p layer. The plan here has no
    fused history update, so its history is the inputs' initial one."""
    import numpy as np
    import torch
    dev = torch.device("cuda", torch.cuda.current_device())
    plan = msf.Plan(msf.make_desc(w.scales, w.grid_h, w.grid_w, w.heads, w.head_dim, w.sink_tokens,
                                  w.history_frames, w.history_capacity, batch=w.batch))
    d = {k: v.to(dev) for k, v in x.items()}
    ws = plan.workspace(dev)
    plan.bind(ws, d["k_sink"], d["v_sink"], d["k_hist"], d["v_hist"])
    out = torch.empty_like(d["q"])
    plan.kv_resample(d["k_win"], d["v_win"])
    plan.mssa_forward(d["q"], d["k_win"], d["v_win"], out)
    torch.cuda.synchronize()
    status_ok = plan.device_status() == msf.MSF_OK
    plan.close()
    err = np.abs(out.double().cpu().numpy() - ref)
    mx, mean = float(err.max()), float(err.mean())
    return {"max_abs_err": mx, "mean_abs_err": mean, "elements": int(err.size),
            "tolerance": {"max": 2e-2, "mean": 2e-3},
            "pass": bool(status_ok and mx <= 2e-2 and mean <= 2e-3)}


def _traffic_from_profile(kernel_src: str):
    """dram bytes per launch of the attention kernel from the committed ncu
    summary, if it was taken on the current kernel source."""
    import hashlib
    path = os.path.join(ROOT, "profiles", "mssa_tc_480p_traffic.json")
    try:
        with open(path) as f:
            d = json.load(f)
        h = hashlib.sha256(open(kernel_src, "rb").read()).hexdigest()[:16]
        if d.get("kernel_sha") == h:
            return float(d["dram_bytes_per_launch"])
    except Exception:
        pass
    return None


def _timed(fn, flush, reps=5, warm=2, sleep=True):
    """Median device time (ms) of fn() between two events; the L2 is flushed
    and the GPU kept busy while the host enqueues, so launch latency counts
    but host gaps do not."""
    import torch
    ts = []
    for i in range(warm + reps):
        flush.fill_(1)
        if sleep:
            torch.cuda._sleep(1000000)
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record()
        fn()
        b.record()
        torch.cuda.synchronize()
        if i >= warm:
            ts.append(a.elapsed_time(b))
    return statistics.median(ts)


def other_configs(msf, synth, dev, flush, peaks, rank):
    """The remaining configurations of the workload family, measured after the
    timed region: the three-scale 48x80 window, the training direction (forward
    with the row log-sum-exp and the MSSA gradient), the paper's chunked layout
    (3 latent frames per state) beside its all-fine window, the STRIDED Subsample
    reading at the 480p layer, the B=4 streaming rollout
    (120 steps, history 2 -> capacity 4), the 30-layer window pass, the
    bandwidth of the pyramid and embedding kernels, and the coarse tiers'
    modules (LoRA adapters and latent residual) beside the plain projections."""
    import torch
    out = {}
    hbm = float(peaks["hbm_gbs"])
    bf16 = float(peaks["bf16_tflops"])
    gen = torch.Generator(device=dev)
    gen.manual_seed(1234 + rank)

    def rnd(shape):
        return torch.randn(shape, generator=gen, device=dev, dtype=torch.float32).to(torch.bfloat16)

    def setup(w, embed=False, fused=False):
        plan = msf.Plan(msf.make_desc(w.scales, w.grid_h, w.grid_w, w.heads, w.head_dim, w.sink_tokens,
                                      w.history_frames, w.history_capacity, batch=w.batch,
                                      latent_channels=w.latent_channels, patch=w.patch,
                                      embed_dim=w.embed_dim if embed else 0,
                                      frames_per_state=w.frames, fused_append=int(fused)))
        N, G, H, D, B = plan.info.n_tokens, w.fine_tokens, w.heads, w.head_dim, w.batch
        t = {k: rnd((B, N, H, D)) for k in ("q", "k_win", "v_win")}
        t["k_sink"], t["v_sink"] = rnd((B, w.sink_tokens, H, D)), rnd((B, w.sink_tokens, H, D))
        for k in ("k_hist", "v_hist"):
            slots = w.history_capacity + 1 if fused else max(w.history_capacity, 1)
            ring = torch.zeros((B, slots, G, H, D), dtype=torch.bfloat16, device=dev)
            ring[:, :w.history_frames] = rnd((B, w.history_frames, G, H, D))
            t[k] = ring
        ws = plan.workspace(dev)
        plan.bind(ws, t["k_sink"], t["v_sink"], t["k_hist"], t["v_hist"])
        t["out"] = torch.empty_like(t["q"])
        t["ws"] = ws
        return plan, t

    # ---- three-scale window (T=6, 48x80, scales (1,1,2,2,4,4), 16 heads)
    w3 = synth.THREE_SCALE
    plan, t = setup(w3)
    pyr_ms = _timed(lambda: plan.kv_resample(t["k_win"], t["v_win"], msf.MSF_RESAMPLE_FULL), flush)
    attn_ms = _timed(lambda: plan.mssa_forward(t["q"], t["k_win"], t["v_win"], t["out"]), flush)
    fl = plan.info.attention_flops
    out["three_scale"] = {"workload": w3.name, "attention_us": attn_ms * 1e3, "gflop": fl / 1e9,
                          "tflops": fl / (attn_ms * 1e-3) / 1e12, "frac": fl / (attn_ms * 1e-3) / 1e12 / bf16,
                          "pyramid_full_us": pyr_ms * 1e3}
    if plan.device_status() != msf.MSF_OK:
        raise RuntimeError("device status error (three-scale)")
    plan.close()
    del t

    # ---- the literal stride-2 reading of Subsample (STRIDED: top-left token
    #      of each block) at the 480p layer: pyramid and attention
    wl = synth.LAYER_480P
    plan = msf.Plan(msf.make_desc(wl.scales, wl.grid_h, wl.grid_w, wl.heads, wl.head_dim, wl.sink_tokens,
                                  wl.history_frames, wl.history_capacity, batch=wl.batch,
                                  resample=msf.MSF_RESAMPLE_STRIDED))
    N, G, H, D, B = plan.info.n_tokens, wl.fine_tokens, wl.heads, wl.head_dim, wl.batch
    ts_ = {k: rnd((B, N, H, D)) for k in ("q", "k_win", "v_win")}
    ts_["k_sink"], ts_["v_sink"] = rnd((B, wl.sink_tokens, H, D)), rnd((B, wl.sink_tokens, H, D))
    for k in ("k_hist", "v_hist"):
        ts_[k] = rnd((B, wl.history_capacity, G, H, D))
    ws_s = plan.workspace(dev)
    plan.bind(ws_s, ts_["k_sink"], ts_["v_sink"], ts_["k_hist"], ts_["v_hist"])
    out_s = torch.empty_like(ts_["q"])
    pyr_ms = _timed(lambda: plan.kv_resample(ts_["k_win"], ts_["v_win"], msf.MSF_RESAMPLE_WINDOW_ONLY), flush)
    attn_ms = _timed(lambda: plan.mssa_forward(ts_["q"], ts_["k_win"], ts_["v_win"], out_s), flush)
    fl = plan.info.attention_flops
    if plan.device_status() != msf.MSF_OK:
        raise RuntimeError("device status error (strided)")
    out["strided_480p"] = {"workload": wl.name, "resample": "STRIDED", "attention_us": attn_ms * 1e3,
                           "tflops": fl / (attn_ms * 1e-3) / 1e12, "pyramid_window_us": pyr_ms * 1e3}
    plan.close()
    del ts_, ws_s, out_s

    # ---- the window pyramid built in the attention launch's prologue
    #      (msf_mssa_forward_resample) beside the pool launch + attention, at
    #      the 480p layer with the fused history update (the step's plan)
    plan, t = setup(wl, fused=True)
    WO = msf.MSF_RESAMPLE_WINDOW_ONLY
    plan.kv_resample(t["k_win"], t["v_win"], msf.MSF_RESAMPLE_FULL)

    def two_launches():
        plan.kv_resample(t["k_win"], t["v_win"], WO)
        plan.mssa_forward(t["q"], t["k_win"], t["v_win"], t["out"])

    two_ms = _timed(two_launches, flush, reps=9)
    one_ms = _timed(lambda: plan.mssa_forward_resample(t["q"], t["k_win"], t["v_win"], t["out"], WO), flush,
                    reps=9)
    alone_ms = _timed(lambda: plan.mssa_forward(t["q"], t["k_win"], t["v_win"], t["out"]), flush, reps=9)
    if plan.device_status() != msf.MSF_OK:
        raise RuntimeError("device status error (resample in attention)")
    out["resample_in_attention_480p"] = {
        "workload": wl.name, "pool_launch_plus_attention_us": two_ms * 1e3,
        "one_launch_us": one_ms * 1e3, "attention_alone_us": alone_ms * 1e3,
        "note": "msf_mssa_forward_resample; the step uses the embedding + pyramid launch instead"}
    plan.close()
    del t

    # ---- training direction at the 480p layer: forward with the row
    #      log-sum-exp, then the MSSA gradient (dq, dk_win, dv_win)
    wl = synth.LAYER_480P
    plan, t = setup(wl)
    B, N, H = wl.batch, plan.info.n_tokens, wl.heads
    lse = torch.empty((B, H, N), dtype=torch.float32, device=dev)
    dout = rnd(t["q"].shape)
    grads = [torch.empty_like(t["q"]) for _ in range(3)]
    bws = plan.backward_workspace(dev)
    plan.kv_resample(t["k_win"], t["v_win"], msf.MSF_RESAMPLE_FULL)
    fwd_ms = _timed(lambda: plan.mssa_forward_lse(t["q"], t["k_win"], t["v_win"], t["out"], lse), flush)
    bwd_ms = _timed(lambda: plan.mssa_backward(t["q"], t["k_win"], t["v_win"], t["out"], dout, lse,
                                               *grads, bws), flush)
    simt_ms = _timed(lambda: plan.mssa_backward_simt(t["q"], t["k_win"], t["v_win"], t["out"], dout,
                                                     lse, *grads, bws), flush, reps=1, warm=1)
    bfl = plan.info.backward_flops
    if plan.device_status() != msf.MSF_OK:
        raise RuntimeError("device status error (backward)")
    out["backward_480p"] = {"workload": wl.name, "forward_lse_us": fwd_ms * 1e3,
                            "backward_us": bwd_ms * 1e3, "backward_gflop": bfl / 1e9,
                            "backward_tflops": bfl / (bwd_ms * 1e-3) / 1e12,
                            "backward_frac": bfl / (bwd_ms * 1e-3) / 1e12 / bf16,
                            "backward_cuda_core_us": simt_ms * 1e3}
    plan.close()
    del t, grads, bws

    # ---- the paper's chunked layout: 3 latent frames per state (12870 tokens),
    #      sink = one chunk, one history chunk; MSSA beside the all-fine window
    wc = synth.CHUNKED_480P
    plan, t = setup(wc)
    pyr_ms = _timed(lambda: plan.kv_resample(t["k_win"], t["v_win"], msf.MSF_RESAMPLE_FULL), flush)
    attn_ms = _timed(lambda: plan.mssa_forward(t["q"], t["k_win"], t["v_win"], t["out"]), flush)
    fl = plan.info.attention_flops
    if plan.device_status() != msf.MSF_OK:
        raise RuntimeError("device status error (chunked)")
    plan.close()
    del t
    wcf = wc.with_scales((1,) * wc.T)
    plan, t = setup(wcf)
    plan.kv_resample(t["k_win"], t["v_win"], msf.MSF_RESAMPLE_FULL)
    fine_ms = _timed(lambda: plan.mssa_forward(t["q"], t["k_win"], t["v_win"], t["out"]), flush,
                     warm=2, reps=5)
    fl_fine = plan.info.attention_flops
    if plan.device_status() != msf.MSF_OK:
        raise RuntimeError("device status error (chunked, all fine)")
    plan.close()
    del t
    out["chunked_480p"] = {"workload": wc.name, "frames_per_state": wc.frames,
                           "attention_us": attn_ms * 1e3, "gflop": fl / 1e9,
                           "tflops": fl / (attn_ms * 1e-3) / 1e12,
                           "frac": fl / (attn_ms * 1e-3) / 1e12 / bf16,
                           "pyramid_full_us": pyr_ms * 1e3,
                           "all_fine_us": fine_ms * 1e3, "all_fine_gflop": fl_fine / 1e9,
                           "all_fine_tflops": fl_fine / (fine_ms * 1e-3) / 1e12,
                           "speedup_vs_all_fine": fine_ms / attn_ms}

    # ---- streaming rollout: B=4, 120 steps, history 2 -> cap 4, sink fixed.
    #      Per step: K/V resample -> MSSA -> history update, on one stream;
    #      the update fused into the resample (spare ring slot + host commit),
    #      and, for comparison, as its own launch after the attention.
    ws4 = synth.STREAM_480P

    def rollout(fused):
        plan, t = setup(ws4, fused=fused)
        sets = [{k: rnd(t[k].shape) for k in ("q", "k_win", "v_win")} for _ in range(4)]
        plan.kv_resample(t["k_win"], t["v_win"], msf.MSF_RESAMPLE_FULL)
        step_ev, attn_ev, fl_steps = [], [], 0.0
        torch.cuda.synchronize()
        for i in range(ws4.steps):
            x = sets[i % len(sets)]
            e0, e1, e2, e3 = (torch.cuda.Event(enable_timing=True) for _ in range(4))
            e0.record()
            plan.kv_resample(x["k_win"], x["v_win"], msf.MSF_RESAMPLE_WINDOW_ONLY)
            e1.record()
            plan.mssa_forward(x["q"], x["k_win"], x["v_win"], t["out"])
            e2.record()
            fl_steps += plan.info.attention_flops
            if fused:
                plan.history_commit()
            else:
                plan.history_append(x["k_win"], x["v_win"])
            e3.record()
            step_ev.append((e0, e3))
            attn_ev.append((e1, e2))
        torch.cuda.synchronize()
        if plan.device_status() != msf.MSF_OK:
            raise RuntimeError("device status error (stream)")
        steps_us = sorted(a.elapsed_time(b) * 1e3 for a, b in step_ev)
        attn_s = sum(a.elapsed_time(b) for a, b in attn_ev) * 1e-3
        res = {"step_us_p50": steps_us[len(steps_us) // 2],
               "step_us_p99": steps_us[min(len(steps_us) - 1, int(0.99 * len(steps_us)))],
               "attention_frames_per_s": ws4.batch * ws4.steps / attn_s,
               "attention_tflops": fl_steps / attn_s / 1e12,
               "history_frames_end": plan.info.history_count}
        plan.close()
        del t, sets
        return res

    fused_r = rollout(True)
    sep_r = rollout(False)
    out["stream_b4"] = dict({"workload": ws4.name, "steps": ws4.steps, "streams": ws4.batch,
                             "history_update": "fused into the resample"}, **fused_r)
    out["stream_b4"]["separate_append"] = {"step_us_p50": sep_r["step_us_p50"],
                                           "step_us_p99": sep_r["step_us_p99"]}
    out["stream_b4"]["note"] = "steps back to back without an L2 flush (a sustained rollout)"

    # ---- 30-layer window pass at 480p shapes (MSP embed -> pyramid -> MSSA -> de-embed per layer)
    wp = synth.PASS_480P
    plan, t = setup(wp, embed=True)
    mi = synth.msp_inputs(wp, torch.bfloat16)
    lat = mi["latent"].to(dev)
    tiers = {sc: mi["w_tier"][sc].t().contiguous().to(dev) for sc in set(wp.scales)}
    w_tier = [tiers[sc] for sc in wp.scales]
    w_out = mi["w_out"].t().contiguous().to(dev)
    N, E = plan.info.n_tokens, wp.embed_dim
    tok = torch.empty((wp.batch, N, E), dtype=torch.bfloat16, device=dev)
    lat_out = torch.empty((wp.batch, wp.latent_channels, wp.grid_h * wp.patch, wp.grid_w * wp.patch),
                          dtype=torch.bfloat16, device=dev)
    plan.kv_resample(t["k_win"], t["v_win"], msf.MSF_RESAMPLE_FULL)

    def one_pass():
        # Each layer as in the single step: the MSP embedding and the K/V
        # pyramid in one launch, attention, then the de-embedding.
        cur = torch.cuda.current_stream()
        for _ in range(wp.layers):
            plan.patchify_resample(lat, w_tier, tok, t["k_win"], t["v_win"], msf.MSF_RESAMPLE_WINDOW_ONLY,
                                   stream=cur)
            plan.mssa_forward(t["q"], t["k_win"], t["v_win"], t["out"], stream=cur)
            plan.unpatchify(0, t["out"].view(wp.batch, N, E), w_out, lat_out, stream=cur)

    pass_ms = _timed(one_pass, flush, reps=3, warm=1, sleep=False)
    fl = plan.info.attention_flops * wp.layers
    out["window_pass_30"] = {"workload": wp.name, "layers": wp.layers, "pass_ms": pass_ms,
                             "us_per_layer": pass_ms * 1e3 / wp.layers, "tflops": fl / (pass_ms * 1e-3) / 1e12}
    # The same pass replayed from a CUDA graph (120 launches, no host work per
    # launch): the pass holds no history update, so it is a static sequence.
    try:
        graph = torch.cuda.CUDAGraph()
        cap = torch.cuda.Stream(device=dev)
        cap.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(cap):
            one_pass()
        torch.cuda.current_stream().wait_stream(cap)
        torch.cuda.synchronize()
        with torch.cuda.graph(graph):
            one_pass()
        g_ms = _timed(graph.replay, flush, reps=3, warm=1)
        out["window_pass_30"].update({"graph_pass_ms": g_ms, "graph_us_per_layer": g_ms * 1e3 / wp.layers,
                                      "graph_tflops": fl / (g_ms * 1e-3) / 1e12})
        del graph
    except Exception as e:  # report the eager pass alone
        out["window_pass_30"]["graph_error"] = str(e)[:200]
    if plan.device_status() != msf.MSF_OK:
        raise RuntimeError("device status error (window pass)")

    # ---- bandwidth of the pyramid and embedding kernels (480p layer, B=1 and the B=4 streams)
    bw = {}
    for w in (synth.LAYER_480P, synth.STREAM_480P):
        plan_b, tb = setup(w, embed=True)
        G, H, D, B = w.grid_h * w.grid_w, w.heads, w.head_dim, w.batch
        row = H * D * 2
        # window part: every fine state read once, pooled to G/4 tokens per coarse group (K and V)
        fine_states = sum(1 for sc in w.scales if sc == 1)
        win_bytes = 2 * B * fine_states * G * row * (1 + 0.25)
        win_ms = _timed(lambda: plan_b.kv_resample(tb["k_win"], tb["v_win"], msf.MSF_RESAMPLE_WINDOW_ONLY),
                        flush)
        mi_b = synth.msp_inputs(w, torch.bfloat16)
        lat_b = mi_b["latent"].to(dev)
        tiers_b = {sc: mi_b["w_tier"][sc].t().contiguous().to(dev) for sc in set(w.scales)}
        tok_b = torch.empty((B, plan_b.info.n_tokens, w.embed_dim), dtype=torch.bfloat16, device=dev)
        emb_ms = _timed(lambda: plan_b.patchify(lat_b, [tiers_b[sc] for sc in w.scales], tok_b), flush)
        emb_bytes = lat_b.numel() * 2 + tok_b.numel() * 2
        for name, by, ms in (("pyramid_window", win_bytes, win_ms), ("embed", emb_bytes, emb_ms)):
            gbs = by / (ms * 1e-3) / 1e9
            bw[f"{name}_{w.name}"] = {"us": ms * 1e3, "bytes": by, "gbs": gbs, "frac_of_measured": gbs / hbm,
                                     "frac_of_8tbs": gbs / 8000.0}
        plan_b.close()
    out["bandwidth"] = bw
    out["bandwidth_note"] = ("event time per call including ~4 us of launch latency; bytes are the "
                             "algorithmic reads + writes")

    # ---- tier modules (Sec. 4.1): coarse tiers with rank-32 LoRA on the embedding and
    # de-embedding and a latent residual branch, beside the plain tier projections
    tier = {}
    rank = 32
    for w in (synth.LAYER_480P, synth.STREAM_480P):
        plan_t, tt = setup(w, embed=True)
        B, N, E, C = w.batch, plan_t.info.n_tokens, w.embed_dim, w.latent_channels
        mi_t = synth.msp_inputs(w, torch.bfloat16)
        ti = synth.tier_inputs(w, rank, torch.bfloat16)
        lat_t = mi_t["latent"].to(dev)
        keep, mods, plain_w = [], {}, {}
        for sc in sorted(set(w.scales)):
            w_emb = mi_t["w_tier"][sc].t().contiguous().to(dev)
            plain_w[sc] = w_emb
            if sc == 1:
                w_o = mi_t["w_out"].t().contiguous().to(dev)
                mods[sc] = msf.tier_module(w_emb, w_o)
                keep += [w_emb, w_o]
                continue
            t = {k: (v.t().contiguous().to(dev) if torch.is_tensor(v) else v) for k, v in ti[sc].items()}
            mods[sc] = msf.tier_module(w_emb, t["w_out"], embed_down=t["lora_a"], embed_up=t["lora_b"],
                                       out_down=t["out_a"], out_up=t["out_b"], residual=t["residual"],
                                       lora_rank=rank, lora_scale=t["gamma"])
            keep += [w_emb] + [v for v in t.values() if torch.is_tensor(v)]
            plain_w[("out", sc)] = t["w_out"]
        tok_t = torch.empty((B, N, E), dtype=torch.bfloat16, device=dev)
        emb_base = _timed(lambda: plan_t.patchify(lat_t, [plain_w[sc] for sc in w.scales], tok_t), flush)
        emb_tier = _timed(lambda: plan_t.patchify_tiers(lat_t, [mods[sc] for sc in w.scales], tok_t), flush)
        pos = w.scales.index(2)
        Hl, Wl = w.grid_h * w.patch, w.grid_w * w.patch
        lat_o = torch.empty((B, C, Hl, Wl), dtype=torch.bfloat16, device=dev)
        de_base = _timed(lambda: plan_t.unpatchify(pos, tok_t, plain_w[("out", 2)], lat_o), flush)
        de_tier = _timed(lambda: plan_t.unpatchify_tier(pos, tok_t, lat_t, mods[2], lat_o), flush)
        if plan_t.device_status() != msf.MSF_OK:
            raise RuntimeError("device status error (tier modules)")
        n_coarse = sum(plan_t.info.state_tokens[l] for l, sc in enumerate(w.scales) if sc > 1)
        M = plan_t.info.state_tokens[pos]
        emb_bytes = lat_t.numel() * 2 + tok_t.numel() * 2 + 2 * B * n_coarse * 64 * 2
        de_bytes = B * M * E * 2 + 2 * B * C * Hl * Wl * 2 + B * M * 64 * 2 * 2
        tier[w.name] = {
            "lora_rank": rank, "embed_plain_us": emb_base * 1e3, "embed_tier_us": emb_tier * 1e3,
            "embed_tier_gbs": emb_bytes / (emb_tier * 1e-3) / 1e9,
            "deembed_position": pos, "deembed_plain_us": de_base * 1e3, "deembed_tier_us": de_tier * 1e3,
            "deembed_tier_gbs": de_bytes / (de_tier * 1e-3) / 1e9,
            "launches": {"embed_tier": 2, "deembed_tier": 3},
        }
        del keep
        plan_t.close()
    out["tier_module"] = tier
    return out


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3)

    world, rank, local = _dist()
    from paper_2607_20940_gb300 import synth
    w = synth.LAYER_480P

    if args.impl == "reference":
        if rank == 0:
            run_reference(args, w)
        return

    import torch
    import torch.distributed as dist

    from paper_2607_20940_gb300 import msf
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl")
    dev = torch.device("cuda", local)
    stream = torch.cuda.current_stream()

    # ------------------------------------------------------------ set-up
    x = synth.attention_inputs(w, torch.bfloat16, seed=w.seed + 1000 * rank)
    mi = synth.msp_inputs(w, torch.bfloat16, seed=w.seed + 1000 * rank)
    # The history update is fused into the K/V resample: the ring has one
    # spare slot, the resample stages the head there (copy and pooled levels
    # from one read) and a host-side commit makes it a history frame.
    plan = msf.Plan(msf.make_desc(w.scales, w.grid_h, w.grid_w, w.heads, w.head_dim,
                                  w.sink_tokens, w.history_frames, w.history_capacity,
                                  batch=w.batch, latent_channels=w.latent_channels, patch=w.patch,
                                  embed_dim=w.embed_dim, fused_append=1))
    info = plan.info
    d = {k: v.to(dev) for k, v in x.items() if k not in ("k_hist", "v_hist")}
    for k in ("k_hist", "v_hist"):
        ring = torch.zeros((w.batch, w.history_capacity + 1) + tuple(x[k].shape[2:]),
                           dtype=x[k].dtype, device=dev)
        ring[:, :w.history_frames] = x[k].to(dev)
        d[k] = ring
    ws = plan.workspace(dev)
    plan.bind(ws, d["k_sink"], d["v_sink"], d["k_hist"], d["v_hist"])
    lat = mi["latent"].to(dev)
    tiers = {s: mi["w_tier"][s].t().contiguous().to(dev) for s in set(w.scales)}
    w_tier = [tiers[s] for s in w.scales]  # positions of one tier share its weight
    w_out = mi["w_out"].t().contiguous().to(dev)
    N, E = info.n_tokens, w.embed_dim
    tok = torch.empty((w.batch, N, E), dtype=torch.bfloat16, device=dev)
    out = torch.empty_like(d["q"])
    lat_out = torch.empty((w.batch, w.latent_channels, w.grid_h * w.patch, w.grid_w * w.patch),
                          dtype=torch.bfloat16, device=dev)
    flush = torch.empty(FLUSH_BYTES, dtype=torch.uint8, device=dev)
    flops = info.attention_flops

    ev_a = []  # attention start/end events of the attention-timing steps

    def step(q, k, v, latent, timed_attn=False, lat_dst=None):
        lat_dst = lat_out if lat_dst is None else lat_dst
        # One stream: the MSP embedding and the window's K/V pyramid (with the
        # staged history head) in one launch, their pooling CTAs on the SM
        # slots the embedding tiles leave free; attention; the host-side
        # commit of the head to the history; the de-embedding of the head.
        # The next step's launch, which overwrites the new spare slot, follows
        # this attention in stream order.
        plan.patchify_resample(latent, w_tier, tok, k, v, msf.MSF_RESAMPLE_WINDOW_ONLY, stream=stream)
        if timed_attn:
            a0 = torch.cuda.Event(enable_timing=True)
            a1 = torch.cuda.Event(enable_timing=True)
            a0.record(stream)
        plan.mssa_forward(q, k, v, out, stream=stream)
        if timed_attn:
            a1.record(stream)
            ev_a.append((a0, a1))
        plan.history_commit()
        plan.unpatchify(0, out.view(w.batch, N, E), w_out, lat_dst, stream=stream)

    plan.kv_resample(d["k_win"], d["v_win"], msf.MSF_RESAMPLE_FULL)
    for _ in range(args.warmup):
        step(d["q"], d["k_win"], d["v_win"], lat)
    torch.cuda.synchronize()
    if plan.device_status() != msf.MSF_OK:
        raise RuntimeError("device status error during warm-up")

    # ------------------------------------------------------- timed steps
    clocks = ClockSampler(local)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    clocks.start()
    time.sleep(0.3)
    launches0 = msf.msf_kernel_launches()
    ev = []
    for _ in range(args.steps):
        flush.fill_(1)
        # The GPU idles ~100 us before the step's first event so that the
        # host has enqueued the step's launches by then: device time of the
        # step, not Python's launch rate (the streamed e2e below includes it).
        torch.cuda._sleep(200000)
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        step(d["q"], d["k_win"], d["v_win"], lat)
        e1.record(stream)
        ev.append((e0, e1))
    torch.cuda.synchronize()
    launches = msf.msf_kernel_launches() - launches0
    # The same steps again with events around the attention launch: its own
    # device time for the roofline. (Events between two launches cost the
    # step the overlap of their programmatic dependent launch, so the step
    # time above is taken without them.)
    for _ in range(args.steps):
        flush.fill_(1)
        torch.cuda._sleep(200000)
        step(d["q"], d["k_win"], d["v_win"], lat, timed_attn=True)
    torch.cuda.synchronize()
    clk = clocks.stop()
    if world > 1:
        dist.barrier()
    step_ms = [a.elapsed_time(b) for a, b in ev]
    attn_ms = [a.elapsed_time(b) for a, b in ev_a]
    tot_ms = max_over_ranks(sum(step_ms), dev)
    status = plan.device_status()

    # ------------------------------------------- end to end (host buffers)
    pin = {k: x[k].pin_memory() for k in ("q", "k_win", "v_win")}
    pin_lat = mi["latent"].pin_memory()
    host_out = torch.empty(lat_out.shape, dtype=lat_out.dtype).pin_memory()
    dq, dk, dv, dl = (torch.empty_like(d["q"]), torch.empty_like(d["k_win"]),
                      torch.empty_like(d["v_win"]), torch.empty_like(lat))
    h2d = sum(t.numel() * t.element_size() for t in list(pin.values()) + [pin_lat])
    d2h = host_out.numel() * host_out.element_size()
    ev2 = []
    for i in range(args.warmup + args.steps):
        flush.fill_(1)
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        dq.copy_(pin["q"], non_blocking=True)
        dk.copy_(pin["k_win"], non_blocking=True)
        dv.copy_(pin["v_win"], non_blocking=True)
        dl.copy_(pin_lat, non_blocking=True)
        step(dq, dk, dv, dl)
        host_out.copy_(lat_out, non_blocking=True)
        e1.record(stream)
        if i >= args.warmup:
            ev2.append((e0, e1))
    torch.cuda.synchronize()
    e2e_serial_ms = max_over_ranks(sum(a.elapsed_time(b) for a, b in ev2), dev)

    # The same steps as a stream: a copy stream uploads step i+1's inputs (two
    # device buffer sets) while step i computes, and reads back step i's
    # latent once it is done. Every step's copies stay inside the timed window.
    copy_s = torch.cuda.Stream(device=dev)
    dbuf = [(torch.empty_like(d["q"]), torch.empty_like(d["k_win"]), torch.empty_like(d["v_win"]),
             torch.empty_like(lat)) for _ in range(2)]
    dlat = [torch.empty_like(lat_out) for _ in range(2)]
    hout = [torch.empty(lat_out.shape, dtype=lat_out.dtype).pin_memory() for _ in range(2)]
    up = [torch.cuda.Event() for _ in range(2)]
    done = [torch.cuda.Event() for _ in range(2)]

    def upload(i):
        sl = i % 2
        if i >= 2:
            copy_s.wait_event(done[sl])  # step i-2 has finished with this buffer set
        with torch.cuda.stream(copy_s):
            for dst, src in zip(dbuf[sl], (pin["q"], pin["k_win"], pin["v_win"], pin_lat)):
                dst.copy_(src, non_blocking=True)
        up[sl].record(copy_s)

    def run_stream(n):
        upload(0)
        for i in range(n):
            sl = i % 2
            if i + 1 < n:
                upload(i + 1)
            stream.wait_event(up[sl])
            step(*dbuf[sl], lat_dst=dlat[sl])
            done[sl].record(stream)
            copy_s.wait_event(done[sl])
            with torch.cuda.stream(copy_s):
                hout[sl].copy_(dlat[sl], non_blocking=True)
        stream.wait_stream(copy_s)

    run_stream(args.warmup)
    torch.cuda.synchronize()
    flush.fill_(1)
    s0 = torch.cuda.Event(enable_timing=True)
    s1 = torch.cuda.Event(enable_timing=True)
    s0.record(stream)
    copy_s.wait_event(s0)
    run_stream(args.steps)
    s1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = max_over_ranks(s0.elapsed_time(s1), dev)
    if plan.device_status() != msf.MSF_OK:
        raise RuntimeError("device status error (end to end)")

    # ------------------------------------------------- all-fine baseline
    wf = w.with_scales((1, 1, 1, 1, 1))
    plan_f = msf.Plan(msf.make_desc(wf.scales, wf.grid_h, wf.grid_w, wf.heads, wf.head_dim,
                                    wf.sink_tokens, wf.history_frames, wf.history_capacity,
                                    batch=wf.batch))
    xf = synth.attention_inputs(wf, torch.bfloat16, seed=wf.seed + 1000 * rank)
    df = {k: v.to(dev) for k, v in xf.items()}
    wsf = plan_f.workspace(dev)
    plan_f.bind(wsf, df["k_sink"], df["v_sink"], df["k_hist"], df["v_hist"])
    outf = torch.empty_like(df["q"])
    plan_f.kv_resample(df["k_win"], df["v_win"])
    fine_ms = []
    for i in range(args.warmup + max(5, args.steps // 2)):
        flush.fill_(1)
        a0 = torch.cuda.Event(enable_timing=True)
        a1 = torch.cuda.Event(enable_timing=True)
        a0.record(stream)
        plan_f.mssa_forward(df["q"], df["k_win"], df["v_win"], outf)
        a1.record(stream)
        if i >= args.warmup:
            fine_ms.append((a0, a1))
    torch.cuda.synchronize()
    fine_attn_ms = statistics.mean(a.elapsed_time(b) for a, b in fine_ms)
    fine_flops = plan_f.info.attention_flops
    plan_f.close()
    del df, wsf, outf
    peaks, peak_src = _peaks()
    others = other_configs(msf, synth, dev, flush, peaks, rank)

    if rank != 0:
        if world > 1:
            dist.barrier()
            dist.destroy_process_group()
        return

    # ------------------------------------------------------- CPU baseline
    cpu = None
    parity = None
    if world == 1 and not args.no_cpu_baseline:
        t0 = time.perf_counter()
        ref = _oracle_step(w, x, mi)
        dt = time.perf_counter() - t0
        host = _host_info()
        cpu = {"value": flops / dt / 1e12, "unit": UNIT,
               "cores": host["blas_threads"] or os.cpu_count(), "kind": "oracle",
               "sample": f"one full 480p step (all 12 heads) in fp64 numpy, {dt:.1f} s",
               "host": host, "other_configs": oracle_other_configs()}
        parity = _parity_check(msf, w, x, ref)

    peaks, peak_src = _peaks()
    attn_avg_ms = statistics.mean(attn_ms)
    achieved = flops / (attn_avg_ms * 1e-3) / 1e12
    peak = float(peaks["bf16_tflops"])
    traffic = _traffic_from_profile(os.path.join(ROOT, "paper_2607_20940_gb300", "csrc", "attn_tc.cu"))
    ms_per_step = tot_ms / args.steps
    line = {
        "metric": METRIC,
        "value": world * flops * args.steps / (tot_ms * 1e-3) / 1e12,
        "unit": UNIT,
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": ms_per_step,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic",
        "config": {
            "workload": w.name, "T": w.T, "scales": list(w.scales), "grid": [w.grid_h, w.grid_w],
            "heads": w.heads, "head_dim": w.head_dim, "sink_tokens": w.sink_tokens,
            "history_frames": w.history_frames, "history_update": "fused into the resample",
            "batch_per_gpu": w.batch,
            "latent": [w.latent_channels, w.grid_h * w.patch, w.grid_w * w.patch],
            "embed_dim": w.embed_dim, "attention_gflop": flops / 1e9,
            "us_per_layer": ms_per_step * 1e3,
            "l2": "flushed between steps (256 MiB write), outside the timed events",
            "parallelism": f"replica x{world}",
        },
        "roofline": {
            "bound": "tensor", "kernel": "mssa_tc_kernel<128>", "achieved": achieved, "peak": peak,
            "unit": "TFLOP/s", "frac": achieved / peak, "traffic": traffic,
            "peak_source": f"{peak_src} bf16_tflops (burst)",
            "frac_of_sustained": achieved / float(peaks.get("bf16_tflops_sustained", peak)),
            "attention_us": attn_avg_ms * 1e3,
        },
        "all_fine": {"attention_us": fine_attn_ms * 1e3, "gflop": fine_flops / 1e9,
                     "tflops": fine_flops / (fine_attn_ms * 1e-3) / 1e12,
                     "speedup_vs_all_fine": fine_attn_ms / attn_avg_ms},
        "cpu_baseline": cpu,
        "parity": parity,
        "other_configs": others,
        "e2e": {"value": world * flops * args.steps / (e2e_ms * 1e-3) / 1e12, "unit": UNIT,
                "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                "ms_per_step": e2e_ms / args.steps,
                "mode": "streamed: step i+1's pinned host-to-device copies overlap step i on a copy "
                        "stream; each step's latent is read back; all copies inside the timed window",
                "serial_ms_per_step": e2e_serial_ms / args.steps,
                "serial_value": world * flops * args.steps / (e2e_serial_ms * 1e-3) / 1e12},
        "step_us": {"mean": ms_per_step * 1e3, "p50": 1e3 * statistics.median(step_ms),
                    "p99": 1e3 * sorted(step_ms)[min(len(step_ms) - 1, int(0.99 * len(step_ms)))]},
        "gpu_launches": launches,
        "clocks": clk,
        "device_status": msf.msf_status_string(status),
    }
    print(json.dumps(line))
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
