"""Host-side checks of the C ABI (no GPU): the library loads, exports every
function include/msf.h declares, and its static plan tables (Eq. 3 counts,
Eq. 4 context layout, FLOP counts) equal the oracle's own enumeration."""
import ctypes
import os
import random
import re

import numpy as np
import pytest

from oracle import schedule
from paper_2607_20940_gb300 import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _msf():
    from paper_2607_20940_gb300 import msf
    return msf


def _declared():
    names = set()
    for fn in os.listdir(os.path.join(ROOT, "include")):
        if fn.endswith(".h"):
            src = open(os.path.join(ROOT, "include", fn)).read()
            src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
            names |= set(re.findall(r"\b(msf_[a-z0-9_]+)\s*\(", src))
    return names


def test_library_exports_every_declared_symbol():
    msf = _msf()
    lib = ctypes.CDLL(msf.LIB_PATH)
    declared = _declared()
    assert declared, "no declarations found"
    for name in sorted(declared):
        assert hasattr(lib, name), f"{name} declared in include/ but not exported"
    assert declared == set(msf.EXPORTS)


def _plan(scales, gh, gw, ns, nh, cap=None, H=2, D=64, B=1, F=1):
    msf = _msf()
    return msf.Plan(msf.make_desc(scales, gh, gw, H, D, ns, nh, history_capacity=cap, batch=B,
                                  frames_per_state=F))


CASES = [
    (synth.TINY.scales, 8, 8, 64, 1),
    (synth.LAYER_480P.scales, 30, 52, 1560, 2),
    (synth.THREE_SCALE.scales, 48, 80, 3840, 2),
    ((1, 1, 1, 1, 1), 30, 52, 1560, 2),
    ((2, 2, 4), 8, 8, 5, 3),
    ((1,), 4, 4, 0, 0),
]


@pytest.mark.parametrize("F", [1, 3])
@pytest.mark.parametrize("scales,gh,gw,ns,nh", CASES)
def test_plan_tables_match_oracle(scales, gh, gw, ns, nh, F):
    if F > 1 and gh * gw > 2000:
        pytest.skip("chunked variant checked on the smaller grids")
    p = _plan(scales, gh, gw, ns, nh, F=F)
    info = p.info
    cnt = schedule.token_counts(scales, gh, gw, F)
    offs = schedule.token_offsets(scales, gh, gw, F)
    assert info.frames_per_state == F
    assert info.n_tokens == sum(cnt)
    assert info.n_tokens_fine == len(scales) * F * gh * gw
    assert list(info.state_tokens[:len(scales)]) == cnt
    assert list(info.state_offset[:len(scales)]) == offs
    groups = schedule.query_groups(scales, gh, gw, F)
    assert info.n_groups == len(groups)
    for gi, g in enumerate(groups):
        gi_ = info.groups[gi]
        assert (gi_.scale, gi_.q_begin, gi_.q_end) == (g.scale, g.q_begin, g.q_end)
        rows = schedule.context_rows(scales, gh, gw, ns, nh, g.scale, F)
        assert gi_.n_kv == len(rows)
        got = p.index_map(gi)
        want = np.array(rows, dtype=np.int32).reshape(-1, 5)
        assert got.shape == want.shape
        assert np.array_equal(got, want)
    assert info.attention_flops == schedule.attention_flops(scales, gh, gw, ns, nh, 2, 64,
                                                            frames=F)


def test_plan_tables_random_schedules():
    rng = random.Random(1234)
    for _ in range(40):
        T = rng.randint(1, 6)
        levels = sorted(rng.choice([1, 1, 2, 2, 4, 8]) for _ in range(T))
        smax = max(levels)
        gh, gw = smax * rng.randint(1, 4), smax * rng.randint(1, 5)
        ns, nh = rng.randint(0, 9), rng.randint(0, 3)
        p = _plan(levels, gh, gw, ns, nh, cap=nh + rng.randint(0, 2), B=rng.randint(1, 3))
        for gi, g in enumerate(schedule.query_groups(levels, gh, gw)):
            want = np.array(schedule.context_rows(levels, gh, gw, ns, nh, g.scale),
                            dtype=np.int32).reshape(-1, 5)
            assert np.array_equal(p.index_map(gi), want)


def test_480p_numbers():
    info = _plan(synth.LAYER_480P.scales, 30, 52, 1560, 2, H=12, D=128).info
    assert info.n_tokens == 4290 and info.n_tokens_fine == 7800
    assert info.attention_flops == 202787020800
    assert info.dense_flops == 4 * 128 * 12 * 7800 * (1560 + 2 * 1560 + 7800)
    assert info.resample_bytes == 2 * 4 * (1560 + 390) * 12 * 128 * 2


def test_chunked_480p_numbers():
    """The paper's layout (Sec. 5.1): 3 latent frames per state, sink = one
    chunk, one history chunk; every count is the per-frame one times 3."""
    w = synth.CHUNKED_480P
    info = _plan(w.scales, 30, 52, w.sink_tokens, 1, H=12, D=128, F=3).info
    assert info.fine_tokens == 4680 and info.n_tokens == 12870 and info.n_tokens_fine == 23400
    assert [info.groups[i].n_kv for i in range(2)] == [4680 + 4680 + 12870,
                                                      4680 + 1170 + 2 * 1170 + 3 * 1170]
    assert info.attention_flops == 4 * 128 * 12 * (9360 * 22230 + 3510 * 11700)
    assert list(info.state_grid_h[:5]) == [90, 90, 45, 45, 45]


@pytest.mark.parametrize("bad", [
    dict(scales=(1, 2, 1)), dict(scales=(1, 3)), dict(scales=(1, 4), gh=30),
    dict(D=96), dict(H=0), dict(nh=3, cap=2), dict(F=-1),
    # one latent frame's grid must take the coarsest stride, even when the
    # stacked chunk (F * gh rows) would
    dict(scales=(1, 4), gh=2, F=2),
])
def test_plan_validation(bad):
    msf = _msf()
    args = dict(scales=(1, 2), gh=8, gw=8, ns=4, nh=1, cap=None, H=2, D=64, F=1)
    args.update(bad)
    with pytest.raises(msf.MsfError) as ei:
        _plan(args["scales"], args["gh"], args["gw"], args["ns"], args["nh"], cap=args["cap"],
              H=args["H"], D=args["D"], F=args["F"])
    assert ei.value.status in (msf.MSF_ERR_INVALID_ARG, msf.MSF_ERR_UNSUPPORTED)


def test_calls_before_bind_and_bad_pointers_fail_without_cuda():
    msf = _msf()
    p = _plan((1, 2), 8, 8, 4, 1)
    lib = msf._lib
    # unbound plan: STATE, reported before any CUDA call
    assert lib.msf_mssa_forward(p.handle, 4096, 8192, 12288, 16384, None) == msf.MSF_ERR_STATE
    assert lib.msf_kv_resample(p.handle, 4096, 8192, 0, None) == msf.MSF_ERR_STATE
    assert lib.msf_history_append(p.handle, 4096, 8192, None) == msf.MSF_ERR_STATE
    assert lib.msf_mssa_forward_resample(p.handle, 4096, 8192, 12288, 16384, 0, None) == msf.MSF_ERR_STATE
    # null / misaligned
    assert lib.msf_mssa_forward(p.handle, None, 8192, 12288, 16384, None) == msf.MSF_ERR_INVALID_ARG
    assert lib.msf_mssa_forward_resample(p.handle, None, 8192, 12288, 16384, 0, None) == \
        msf.MSF_ERR_INVALID_ARG
    assert lib.msf_mssa_forward_resample(p.handle, 4096, 8192, 12288, None, 0, None) == \
        msf.MSF_ERR_INVALID_ARG
    assert lib.msf_mssa_forward_resample(None, 4096, 8192, 12288, 16384, 0, None) == msf.MSF_ERR_INVALID_ARG
    assert lib.msf_plan_bind(p.handle, 4096, 16, 4096, 4096, 4096, 4096) == msf.MSF_ERR_WORKSPACE
    assert lib.msf_plan_bind(p.handle, 4097, 1 << 30, 4096, 4096, 4096, 4096) == msf.MSF_ERR_INVALID_ARG
    assert lib.msf_plan_index_map(p.handle, 7, None, 0, ctypes.byref(ctypes.c_size_t())) == \
        msf.MSF_ERR_INVALID_ARG
    assert msf.msf_status_string(msf.MSF_ERR_TIMEOUT) == "device wait timed out"


# ------------------------------------------------ fused history update --

def _fused_plan(scales, gh, gw, ns, nh, cap, F=1):
    msf = _msf()
    return msf.Plan(msf.make_desc(scales, gh, gw, 2, 64, ns, nh, history_capacity=cap,
                                  frames_per_state=F, fused_append=1))


@pytest.mark.parametrize("scales,gh,gw,ns,nh,cap,F", [
    ((1, 1, 2), 8, 8, 5, 1, 3, 1),
    ((1, 2, 2, 4), 8, 8, 3, 2, 2, 1),   # at capacity: every ring slot in use
    ((1, 1), 4, 6, 0, 0, 1, 1),         # no coarser level, empty history
    ((1, 2), 4, 4, 2, 1, 2, 2),         # chunked
])
def test_fused_append_context_is_the_same_rows(scales, gh, gw, ns, nh, cap, F):
    """With the head staged in the ring's spare slot the kernels read the
    same Eq. 4 context in another order: sink; for g > 1 the pooled window
    states 2..; ring slots 0..count (live frames, then the spare = the head);
    the window states from k_win. Same rows, same lengths, same FLOPs."""
    p = _fused_plan(scales, gh, gw, ns, nh, cap, F)
    ref = _plan(scales, gh, gw, ns, nh, cap=cap, F=F)
    assert p.info.attention_flops == ref.info.attention_flops
    assert p.info.history_next_slot == nh          # spare = first free slot
    for gi, g in enumerate(schedule.query_groups(scales, gh, gw, F)):
        got = [tuple(r) for r in p.index_map(gi).tolist()]
        want = schedule.context_rows(scales, gh, gw, ns, nh, g.scale, F)
        assert sorted(got) == sorted(want)
        assert p.info.groups[gi].n_kv == len(want)
        # the kernel order, written out from the layout rule
        sink = [r for r in want if r[0] == schedule.SINK]
        hist = [r for r in want if r[0] == schedule.HIST]
        win = [r for r in want if r[0] == schedule.WIN]
        head = [r for r in win if r[1] == 0]
        finer = [r for r in win if r[1] > 0 and scales[r[1]] < g.scale]
        rest = [r for r in win if r[1] > 0 and scales[r[1]] >= g.scale]
        if g.scale == 1:
            order = sink + hist + head + rest
        else:
            order = sink + finer + hist + head + rest
        assert got == order


def test_fused_append_validation_and_state():
    msf = _msf()
    for kw, err in [(dict(scales=(2, 2)), msf.MSF_ERR_UNSUPPORTED),     # head not fine
                    (dict(cap=0), msf.MSF_ERR_UNSUPPORTED),               # no ring
                    (dict(fa=2), msf.MSF_ERR_INVALID_ARG)]:
        a = dict(scales=(1, 2), cap=2, fa=1)
        a.update(kw)
        with pytest.raises(msf.MsfError) as ei:
            msf.Plan(msf.make_desc(a["scales"], 8, 8, 2, 64, 4, 0, history_capacity=a["cap"],
                                   fused_append=a["fa"]))
        assert ei.value.status == err
    p = _fused_plan((1, 2), 8, 8, 4, 1, 2)
    lib = msf._lib
    assert lib.msf_history_commit(p.handle) == msf.MSF_ERR_STATE      # not bound
    q = _plan((1, 2), 8, 8, 4, 1, cap=2)
    assert lib.msf_history_commit(q.handle) == msf.MSF_ERR_STATE      # not fused
    assert lib.msf_history_commit(None) == msf.MSF_ERR_INVALID_ARG


def test_backward_flops_480p():
    """S, dP and dQ over every query-key pair (6 D flops each), dK and dV over
    the pairs whose key comes from the window (4 D more); the sink and the
    history are a detached cache."""
    info = _plan(synth.LAYER_480P.scales, 30, 52, 1560, 2, H=12, D=128).info
    g1 = 3120 * (6 * 128 * 8970 + 4 * 128 * (8970 - 1560 - 2 * 1560))
    g2 = 1170 * (6 * 128 * 4290 + 4 * 128 * (4290 - 1560 - 2 * 390))
    assert info.backward_flops == 12 * (g1 + g2)


def test_history_state_host_checks():
    msf = _msf()
    p = _plan((1, 2), 8, 8, 4, 1, cap=3)
    st = p.history_state()
    assert (st.count, st.oldest, st.spare) == (1, 0, -1)
    with pytest.raises(msf.MsfError) as ei:
        p.set_history_state(st)                      # not bound
    assert ei.value.status == msf.MSF_ERR_STATE
    q = _fused_plan((1, 2), 8, 8, 4, 2, 3)
    st = q.history_state()
    assert (st.count, st.oldest, st.spare) == (2, 0, 2)
