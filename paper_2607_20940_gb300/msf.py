"""Thin ctypes binding of libmsf.so (include/msf.h).

Argument marshalling only: every step of the window pass runs in the CUDA
kernels behind the C ABI. Tensors are passed by device pointer; torch is used
for device memory and streams. If the library is missing the import fails:
there is no fallback path.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Sequence

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libmsf.so")

MSF_OK = 0
MSF_ERR_INVALID_ARG = 1
MSF_ERR_UNSUPPORTED = 2
MSF_ERR_CUDA = 3
MSF_ERR_TIMEOUT = 4
MSF_ERR_STATE = 5
MSF_ERR_WORKSPACE = 6
MSF_DTYPE_BF16 = 0
MSF_DTYPE_F32 = 1
MSF_RESAMPLE_AVG = 0
MSF_RESAMPLE_STRIDED = 1
MSF_RESAMPLE_FULL = 0
MSF_RESAMPLE_WINDOW_ONLY = 1
MSF_MAX_STATES = 16
MSF_MAX_GROUPS = 8

EXPORTS = (
    "msf_status_string", "msf_last_cuda_error", "msf_plan_create", "msf_plan_destroy",
    "msf_plan_query", "msf_plan_index_map", "msf_plan_bind", "msf_patchify", "msf_unpatchify",
    "msf_kv_resample", "msf_mssa_forward", "msf_mssa_forward_simt", "msf_history_append",
    "msf_plan_device_status", "msf_kernel_launches", "msf_unpatchify_noalloc",
    "msf_selftest_wait_timeout", "msf_history_commit", "msf_mssa_forward_lse",
    "msf_mssa_backward", "msf_mssa_backward_simt", "msf_history_get", "msf_history_set",
    "msf_noalloc_device_status", "msf_noalloc_selftest_wait_timeout", "msf_patchify_tiers",
    "msf_unpatchify_tier", "msf_patchify_resample", "msf_mssa_forward_resample",
)


class msf_plan_desc(ctypes.Structure):
    _fields_ = [
        ("T", ctypes.c_int32), ("scales", ctypes.c_int32 * MSF_MAX_STATES),
        ("grid_h", ctypes.c_int32), ("grid_w", ctypes.c_int32), ("heads", ctypes.c_int32),
        ("head_dim", ctypes.c_int32), ("sink_tokens", ctypes.c_int32),
        ("history_frames", ctypes.c_int32), ("history_capacity", ctypes.c_int32),
        ("batch", ctypes.c_int32), ("dtype", ctypes.c_int32), ("resample", ctypes.c_int32),
        ("softmax_scale", ctypes.c_float), ("latent_channels", ctypes.c_int32),
        ("patch", ctypes.c_int32), ("embed_dim", ctypes.c_int32),
        ("frames_per_state", ctypes.c_int32), ("fused_append", ctypes.c_int32),
    ]


class msf_tier_module(ctypes.Structure):
    _fields_ = [
        ("w_embed", ctypes.c_void_p), ("embed_down", ctypes.c_void_p), ("embed_up", ctypes.c_void_p),
        ("w_out", ctypes.c_void_p), ("out_down", ctypes.c_void_p), ("out_up", ctypes.c_void_p),
        ("residual", ctypes.c_void_p), ("lora_rank", ctypes.c_int32), ("lora_scale", ctypes.c_float),
    ]


class msf_history_state(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in ("count", "oldest", "spare", "_pad")]


class msf_group_info(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in
                ("scale", "q_begin", "q_end", "n_kv", "n_pyramid", "pyr_offset")]


class msf_plan_info(ctypes.Structure):
    _fields_ = [
        ("T", ctypes.c_int32), ("n_tokens", ctypes.c_int32), ("n_tokens_fine", ctypes.c_int32),
        ("fine_tokens", ctypes.c_int32),
        ("state_offset", ctypes.c_int32 * MSF_MAX_STATES),
        ("state_tokens", ctypes.c_int32 * MSF_MAX_STATES),
        ("state_grid_h", ctypes.c_int32 * MSF_MAX_STATES),
        ("state_grid_w", ctypes.c_int32 * MSF_MAX_STATES),
        ("n_groups", ctypes.c_int32), ("groups", msf_group_info * MSF_MAX_GROUPS),
        ("history_count", ctypes.c_int32), ("history_next_slot", ctypes.c_int32),
        ("pyramid_tokens", ctypes.c_int32), ("frames_per_state", ctypes.c_int32),
        ("workspace_bytes", ctypes.c_uint64), ("attention_flops", ctypes.c_uint64),
        ("dense_flops", ctypes.c_uint64), ("resample_bytes", ctypes.c_uint64),
        ("pyramid_k_offset", ctypes.c_uint64), ("pyramid_v_offset", ctypes.c_uint64),
        ("backward_workspace_bytes", ctypes.c_uint64), ("backward_flops", ctypes.c_uint64),
        ("attention_counter_offset", ctypes.c_uint64), ("attention_counter_bytes", ctypes.c_uint64),
    ]


def _load():
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"{LIB_PATH} is missing: run __graft_entry__.build() first")
    lib = ctypes.CDLL(LIB_PATH)
    P, VP, I32, SZ = ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int32, ctypes.c_size_t
    sig = {
        "msf_status_string": (ctypes.c_char_p, [ctypes.c_int]),
        "msf_last_cuda_error": (ctypes.c_int, []),
        "msf_plan_create": (ctypes.c_int, [ctypes.POINTER(msf_plan_desc), ctypes.POINTER(P)]),
        "msf_plan_destroy": (None, [P]),
        "msf_plan_query": (ctypes.c_int, [P, ctypes.POINTER(msf_plan_info)]),
        "msf_plan_index_map": (ctypes.c_int, [P, I32, ctypes.POINTER(ctypes.c_int32), SZ,
                                              ctypes.POINTER(SZ)]),
        "msf_plan_bind": (ctypes.c_int, [P, VP, SZ, VP, VP, VP, VP]),
        "msf_patchify": (ctypes.c_int, [P, VP, ctypes.POINTER(VP), VP, VP]),
        "msf_unpatchify": (ctypes.c_int, [P, I32, VP, VP, VP, VP]),
        "msf_patchify_resample": (ctypes.c_int, [P, VP, ctypes.POINTER(VP), VP, VP, VP, I32, VP]),
        "msf_kv_resample": (ctypes.c_int, [P, VP, VP, I32, VP]),
        "msf_mssa_forward": (ctypes.c_int, [P, VP, VP, VP, VP, VP]),
        "msf_mssa_forward_simt": (ctypes.c_int, [P, VP, VP, VP, VP, VP]),
        "msf_mssa_forward_resample": (ctypes.c_int, [P, VP, VP, VP, VP, I32, VP]),
        "msf_history_append": (ctypes.c_int, [P, VP, VP, VP]),
        "msf_plan_device_status": (ctypes.c_int, [P, VP]),
        "msf_kernel_launches": (ctypes.c_uint64, []),
        "msf_unpatchify_noalloc": (ctypes.c_int, [P, I32, VP, VP, VP, VP]),
        "msf_selftest_wait_timeout": (ctypes.c_int, [P, ctypes.c_int64, VP]),
        "msf_noalloc_device_status": (ctypes.c_int, [VP]),
        "msf_patchify_tiers": (ctypes.c_int, [P, VP, ctypes.POINTER(ctypes.POINTER(msf_tier_module)), VP,
                                              VP]),
        "msf_unpatchify_tier": (ctypes.c_int, [P, I32, VP, VP, ctypes.POINTER(msf_tier_module), VP, VP]),
        "msf_noalloc_selftest_wait_timeout": (ctypes.c_int, [ctypes.c_int64, VP]),
        "msf_history_commit": (ctypes.c_int, [P]),
        "msf_history_get": (ctypes.c_int, [P, ctypes.POINTER(msf_history_state)]),
        "msf_history_set": (ctypes.c_int, [P, ctypes.POINTER(msf_history_state)]),
        "msf_mssa_forward_lse": (ctypes.c_int, [P, VP, VP, VP, VP, VP, VP]),
        "msf_mssa_backward": (ctypes.c_int, [P, VP, VP, VP, VP, VP, VP, VP, VP, VP, VP, SZ, VP]),
        "msf_mssa_backward_simt": (ctypes.c_int, [P, VP, VP, VP, VP, VP, VP, VP, VP, VP, VP, SZ, VP]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    return lib


_lib = _load()


class MsfError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        msg = _lib.msf_status_string(status).decode()
        if status == MSF_ERR_CUDA:
            msg += f" (cudaError {_lib.msf_last_cuda_error()})"
        super().__init__(f"{where}: {msg}")


def _check(status: int, where: str) -> None:
    if status != MSF_OK:
        raise MsfError(status, where)


def _ptr(t) -> Optional[int]:
    if t is None:
        return None
    return t.data_ptr()


def _stream(stream) -> Optional[int]:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    return stream if isinstance(stream, int) else stream.cuda_stream


# ---------------------------------------------------------------- functions
# One Python function per C entry point, same name, same argument order.

def msf_status_string(status: int) -> str:
    return _lib.msf_status_string(status).decode()


def msf_plan_create(desc: msf_plan_desc) -> int:
    h = ctypes.c_void_p()
    _check(_lib.msf_plan_create(ctypes.byref(desc), ctypes.byref(h)), "msf_plan_create")
    return h.value


def msf_plan_destroy(plan: int) -> None:
    _lib.msf_plan_destroy(plan)


def msf_plan_query(plan: int) -> msf_plan_info:
    info = msf_plan_info()
    _check(_lib.msf_plan_query(plan, ctypes.byref(info)), "msf_plan_query")
    return info


def msf_plan_index_map(plan: int, group: int):
    import numpy as np
    n = ctypes.c_size_t()
    _check(_lib.msf_plan_index_map(plan, group, None, 0, ctypes.byref(n)), "msf_plan_index_map")
    out = np.zeros((n.value, 5), dtype=np.int32)
    _check(_lib.msf_plan_index_map(plan, group, out.ctypes.data_as(ctypes.POINTER(ctypes.c_int32)),
                                   n.value, ctypes.byref(n)), "msf_plan_index_map")
    return out


def msf_plan_bind(plan: int, workspace, k_sink, v_sink, k_hist, v_hist) -> None:
    nbytes = workspace.numel() * workspace.element_size()
    _check(_lib.msf_plan_bind(plan, _ptr(workspace), nbytes, _ptr(k_sink), _ptr(v_sink),
                              _ptr(k_hist), _ptr(v_hist)), "msf_plan_bind")


def msf_patchify(plan: int, latent, w_tier: Optional[Sequence], tokens, stream=None) -> None:
    arr = None
    if w_tier is not None:
        arr = (ctypes.c_void_p * len(w_tier))(*[_ptr(w) for w in w_tier])
    _check(_lib.msf_patchify(plan, _ptr(latent), arr, _ptr(tokens), _stream(stream)),
           "msf_patchify")


def msf_patchify_resample(plan: int, latent, w_tier: Sequence, tokens, k_win, v_win,
                          flags: int = MSF_RESAMPLE_FULL, stream=None) -> None:
    arr = (ctypes.c_void_p * len(w_tier))(*[_ptr(w) for w in w_tier])
    _check(_lib.msf_patchify_resample(plan, _ptr(latent), arr, _ptr(tokens), _ptr(k_win), _ptr(v_win), flags,
                                      _stream(stream)), "msf_patchify_resample")


def msf_unpatchify(plan: int, position: int, tokens, w_out, latent_out, stream=None) -> None:
    _check(_lib.msf_unpatchify(plan, position, _ptr(tokens), _ptr(w_out), _ptr(latent_out),
                               _stream(stream)), "msf_unpatchify")


def tier_module(w_embed, w_out, embed_down=None, embed_up=None, out_down=None, out_up=None,
                residual=None, lora_rank=0, lora_scale=1.0) -> msf_tier_module:
    """An msf_tier_module of device tensors (nn.Linear layouts, see msf.h)."""
    return msf_tier_module(_ptr(w_embed), _ptr(embed_down), _ptr(embed_up), _ptr(w_out),
                           _ptr(out_down), _ptr(out_up), _ptr(residual), int(lora_rank),
                           float(lora_scale))


def msf_patchify_tiers(plan: int, latent, tiers: Sequence[msf_tier_module], tokens, stream=None) -> None:
    """tiers: one msf_tier_module per window position (the same object for
    positions that share a tier)."""
    ptrs = (ctypes.POINTER(msf_tier_module) * len(tiers))(*[ctypes.pointer(t) for t in tiers])
    _check(_lib.msf_patchify_tiers(plan, _ptr(latent), ptrs, _ptr(tokens), _stream(stream)),
           "msf_patchify_tiers")


def msf_unpatchify_tier(plan: int, position: int, tokens, latent_in, tier: msf_tier_module,
                        latent_out, stream=None) -> None:
    _check(_lib.msf_unpatchify_tier(plan, position, _ptr(tokens), _ptr(latent_in), ctypes.byref(tier),
                                    _ptr(latent_out), _stream(stream)), "msf_unpatchify_tier")


def msf_kv_resample(plan: int, k_win, v_win, flags: int = MSF_RESAMPLE_FULL, stream=None) -> None:
    _check(_lib.msf_kv_resample(plan, _ptr(k_win), _ptr(v_win), flags, _stream(stream)),
           "msf_kv_resample")


def msf_mssa_forward(plan: int, q, k_win, v_win, out, stream=None) -> None:
    _check(_lib.msf_mssa_forward(plan, _ptr(q), _ptr(k_win), _ptr(v_win), _ptr(out),
                                 _stream(stream)), "msf_mssa_forward")


def msf_mssa_forward_simt(plan: int, q, k_win, v_win, out, stream=None) -> None:
    _check(_lib.msf_mssa_forward_simt(plan, _ptr(q), _ptr(k_win), _ptr(v_win), _ptr(out),
                                      _stream(stream)), "msf_mssa_forward_simt")


def msf_mssa_forward_resample(plan: int, q, k_win, v_win, out, flags: int = MSF_RESAMPLE_FULL,
                              stream=None) -> None:
    _check(_lib.msf_mssa_forward_resample(plan, _ptr(q), _ptr(k_win), _ptr(v_win), _ptr(out),
                                          int(flags), _stream(stream)), "msf_mssa_forward_resample")


def msf_history_append(plan: int, k_win, v_win, stream=None) -> None:
    _check(_lib.msf_history_append(plan, _ptr(k_win), _ptr(v_win), _stream(stream)),
           "msf_history_append")


def msf_mssa_forward_lse(plan: int, q, k_win, v_win, out, lse, stream=None) -> None:
    _check(_lib.msf_mssa_forward_lse(plan, _ptr(q), _ptr(k_win), _ptr(v_win), _ptr(out),
                                     _ptr(lse), _stream(stream)), "msf_mssa_forward_lse")


def msf_mssa_backward(plan: int, q, k_win, v_win, out, dout, lse, dq, dk_win, dv_win, bwd_ws,
                      stream=None) -> None:
    nbytes = bwd_ws.numel() * bwd_ws.element_size()
    _check(_lib.msf_mssa_backward(plan, _ptr(q), _ptr(k_win), _ptr(v_win), _ptr(out), _ptr(dout),
                                  _ptr(lse), _ptr(dq), _ptr(dk_win), _ptr(dv_win), _ptr(bwd_ws),
                                  nbytes, _stream(stream)), "msf_mssa_backward")


def msf_mssa_backward_simt(plan: int, q, k_win, v_win, out, dout, lse, dq, dk_win, dv_win, bwd_ws,
                           stream=None) -> None:
    nbytes = bwd_ws.numel() * bwd_ws.element_size()
    _check(_lib.msf_mssa_backward_simt(plan, _ptr(q), _ptr(k_win), _ptr(v_win), _ptr(out),
                                       _ptr(dout), _ptr(lse), _ptr(dq), _ptr(dk_win), _ptr(dv_win),
                                       _ptr(bwd_ws), nbytes, _stream(stream)),
           "msf_mssa_backward_simt")


def msf_history_get(plan: int) -> msf_history_state:
    st = msf_history_state()
    _check(_lib.msf_history_get(plan, ctypes.byref(st)), "msf_history_get")
    return st


def msf_history_set(plan: int, st: msf_history_state) -> None:
    _check(_lib.msf_history_set(plan, ctypes.byref(st)), "msf_history_set")


def msf_history_commit(plan: int) -> None:
    _check(_lib.msf_history_commit(plan), "msf_history_commit")


def msf_plan_device_status(plan: int, stream=None) -> int:
    return _lib.msf_plan_device_status(plan, _stream(stream))


def msf_unpatchify_noalloc(plan: int, position: int, tokens, w_out, latent_out, stream=None) -> None:
    _check(_lib.msf_unpatchify_noalloc(plan, position, _ptr(tokens), _ptr(w_out), _ptr(latent_out),
                                       _stream(stream)), "msf_unpatchify_noalloc")


def msf_noalloc_device_status(stream=None) -> int:
    return _lib.msf_noalloc_device_status(_stream(stream))


def msf_noalloc_selftest_wait_timeout(limit_cycles: int, stream=None) -> None:
    _check(_lib.msf_noalloc_selftest_wait_timeout(limit_cycles, _stream(stream)),
           "msf_noalloc_selftest_wait_timeout")


def msf_selftest_wait_timeout(plan: int, limit_cycles: int, stream=None) -> None:
    _check(_lib.msf_selftest_wait_timeout(plan, limit_cycles, _stream(stream)), "msf_selftest_wait_timeout")


def msf_kernel_launches() -> int:
    return int(_lib.msf_kernel_launches())


# ------------------------------------------------------------ convenience

def make_desc(scales, grid_h, grid_w, heads, head_dim, sink_tokens, history_frames,
              history_capacity=None, batch=1, dtype=MSF_DTYPE_BF16, resample=MSF_RESAMPLE_AVG,
              softmax_scale=0.0, latent_channels=0, patch=0, embed_dim=0,
              frames_per_state=1, fused_append=0) -> msf_plan_desc:
    d = msf_plan_desc()
    d.T = len(scales)
    for i, s in enumerate(scales):
        d.scales[i] = int(s)
    d.grid_h, d.grid_w, d.heads, d.head_dim = grid_h, grid_w, heads, head_dim
    d.sink_tokens, d.history_frames = sink_tokens, history_frames
    d.history_capacity = history_frames if history_capacity is None else history_capacity
    d.batch, d.dtype, d.resample, d.softmax_scale = batch, dtype, resample, softmax_scale
    d.latent_channels, d.patch, d.embed_dim = latent_channels, patch, embed_dim
    d.frames_per_state = frames_per_state
    d.fused_append = fused_append
    return d


class Plan:
    """Owns a plan handle and the device buffers bound to it (torch tensors)."""

    def __init__(self, desc: msf_plan_desc):
        self.desc = desc
        self.handle = msf_plan_create(desc)
        self.info = msf_plan_query(self.handle)
        self._keep = ()

    def close(self):
        if self.handle:
            msf_plan_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def refresh(self) -> msf_plan_info:
        self.info = msf_plan_query(self.handle)
        return self.info

    def bind(self, workspace, k_sink, v_sink, k_hist, v_hist):
        msf_plan_bind(self.handle, workspace, k_sink, v_sink, k_hist, v_hist)
        self._keep = (workspace, k_sink, v_sink, k_hist, v_hist)
        self.refresh()

    def workspace(self, device="cuda"):
        import torch
        return torch.zeros(int(self.info.workspace_bytes), dtype=torch.uint8, device=device)

    def index_map(self, group: int):
        return msf_plan_index_map(self.handle, group)

    def patchify(self, latent, w_tier, tokens, stream=None):
        msf_patchify(self.handle, latent, w_tier, tokens, stream)

    def unpatchify(self, position, tokens, w_out, latent_out, stream=None):
        msf_unpatchify(self.handle, position, tokens, w_out, latent_out, stream)

    def patchify_resample(self, latent, w_tier, tokens, k_win, v_win, flags=MSF_RESAMPLE_FULL, stream=None):
        msf_patchify_resample(self.handle, latent, w_tier, tokens, k_win, v_win, flags, stream)

    def patchify_tiers(self, latent, tiers, tokens, stream=None):
        msf_patchify_tiers(self.handle, latent, tiers, tokens, stream)

    def unpatchify_tier(self, position, tokens, latent_in, tier, latent_out, stream=None):
        msf_unpatchify_tier(self.handle, position, tokens, latent_in, tier, latent_out, stream)

    def kv_resample(self, k_win, v_win, flags=MSF_RESAMPLE_FULL, stream=None):
        msf_kv_resample(self.handle, k_win, v_win, flags, stream)

    def mssa_forward(self, q, k_win, v_win, out, stream=None):
        msf_mssa_forward(self.handle, q, k_win, v_win, out, stream)

    def mssa_forward_resample(self, q, k_win, v_win, out, flags=MSF_RESAMPLE_FULL, stream=None):
        msf_mssa_forward_resample(self.handle, q, k_win, v_win, out, flags, stream)

    def mssa_forward_lse(self, q, k_win, v_win, out, lse, stream=None):
        msf_mssa_forward_lse(self.handle, q, k_win, v_win, out, lse, stream)

    def mssa_backward(self, q, k_win, v_win, out, dout, lse, dq, dk_win, dv_win, bwd_ws,
                      stream=None):
        msf_mssa_backward(self.handle, q, k_win, v_win, out, dout, lse, dq, dk_win, dv_win, bwd_ws,
                          stream)

    def mssa_backward_simt(self, q, k_win, v_win, out, dout, lse, dq, dk_win, dv_win, bwd_ws,
                           stream=None):
        msf_mssa_backward_simt(self.handle, q, k_win, v_win, out, dout, lse, dq, dk_win, dv_win,
                               bwd_ws, stream)

    def backward_workspace(self, device="cuda"):
        import torch
        return torch.empty(int(self.info.backward_workspace_bytes), dtype=torch.uint8,
                           device=device)

    def mssa_forward_simt(self, q, k_win, v_win, out, stream=None):
        msf_mssa_forward_simt(self.handle, q, k_win, v_win, out, stream)

    def history_append(self, k_win, v_win, stream=None):
        msf_history_append(self.handle, k_win, v_win, stream)
        self.refresh()

    def history_state(self) -> msf_history_state:
        return msf_history_get(self.handle)

    def set_history_state(self, st: msf_history_state):
        msf_history_set(self.handle, st)
        self.refresh()

    def history_commit(self):
        msf_history_commit(self.handle)
        self.refresh()

    def device_status(self, stream=None) -> int:
        return msf_plan_device_status(self.handle, stream)

    def selftest_wait_timeout(self, limit_cycles, stream=None):
        msf_selftest_wait_timeout(self.handle, limit_cycles, stream)
