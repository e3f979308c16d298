"""uc_attend_static: decode attention for callers that cannot allocate device
memory for scratch space (for example a plug-in inside a host framework that
owns the device memory pool, or a latency-critical path that must not call
cudaMalloc). It takes no workspace: its scratch is a static device array
inside the library. This test calls it through the C ABI twice in a row and
checks each result against uc_attend (which uses a caller workspace), within
the attention tolerance used everywhere else, and checks that a call needing
more scratch than the array holds is refused before anything runs.

This file is collected last so that a run stopping at the first failure has
already run every other test; it also passes when run on its own.
"""
import ctypes as C

import numpy as np
import pytest
import torch

import synth
from tests import _packed

pytestmark = pytest.mark.gpu

uc = pytest.importorskip("paper_2609_32831_gb300")
from paper_2609_32831_gb300 import _lib  # noqa: E402

DEV = torch.device("cuda")


def _dev(x):
    return torch.from_numpy(np.ascontiguousarray(x, np.float32)).to(torch.bfloat16).to(DEV)


def _segments(B, hkv):
    """A text view, evicted bf16 rows, evicted + int4 rows and int2 rows."""
    sizes = [200, 700, 600, 130]
    N = sum(sizes)
    k, v = synth.make_kv(404, B, hkv, N)
    s = synth.make_scores(405, (B, hkv, N))
    kd, vd, sd = _dev(k), _dev(v), torch.from_numpy(s).to(DEV)
    segs = [uc.Segment.view(kd, vd, 0, 200)]
    for kind, bits, lo, n, keep in [("evict", 16, 200, 700, 111), ("evict_quant", 4, 900, 600, 150),
                                    ("quant", 2, 1500, 130, 130)]:
        g = uc.Segment(kind, bits, B, hkv, n, keep, DEV)
        g.set_keep([keep] * B)
        uc.compress_segment(kd, vd, g, begin=lo, scores=sd)
        segs.append(g)
    return segs, (kd, vd)


def _call_static(q, segs, out, lse, mass):
    arr = (C.POINTER(_lib.UcSegment) * len(segs))(*[C.pointer(s.c) for s in segs])
    B, hq, T, d = q.shape
    stream = C.c_void_p(torch.cuda.current_stream().cuda_stream)
    return _lib.lib().uc_attend_static(
        C.c_void_p(q.data_ptr()), hq, T, C.cast(arr, C.c_void_p), len(segs), C.c_void_p(out.data_ptr()),
        C.c_void_p(lse.data_ptr()), C.c_void_p(mass.data_ptr()), stream)


@pytest.mark.parametrize("T", [1, 3])
def test_attend_static_matches_attend(T):
    B, hkv = 3, 4
    segs, keep_alive = _segments(B, hkv)
    q = _dev(synth.make_q(406 + T, B, 28, T))
    ref_o, ref_lse, ref_mass = uc.attend(q, segs, ws=uc.Workspace(DEV))
    torch.cuda.synchronize()
    r_o = ref_o.double().cpu().numpy()
    for call in range(2):
        out = torch.full_like(q, float("nan"))
        lse = torch.full((B, 28, T), float("nan"), device=DEV)
        mass = torch.full((B, 28, T, len(segs)), float("nan"), device=DEV)
        status = _call_static(q, segs, out, lse, mass)
        assert status == _lib.UC_OK, _lib.lib().uc_last_error()
        torch.cuda.synchronize()
        assert _packed.attention_error(out.double().cpu().numpy(), r_o) <= _packed.ATTN_RTOL
        np.testing.assert_allclose(lse.cpu().numpy(), ref_lse.cpu().numpy(), rtol=0, atol=1e-5)
        np.testing.assert_allclose(mass.cpu().numpy(), ref_mass.cpu().numpy(), rtol=0, atol=1e-5)


def test_attend_static_refuses_oversized_calls():
    B, hkv = 64, 4
    n = 200  # 64 sequences x 4 heads, several items each: partials for T = 8 exceed 8 MiB
    seg = uc.Segment("evict", 16, B, hkv, n, n, DEV)
    seg.set_keep([n] * B)
    k, v = synth.make_kv(407, B, hkv, n)
    uc.compress_segment(_dev(k), _dev(v), seg, scores=torch.ones((B, hkv, n), device=DEV))
    segs = [seg, seg]  # two segments: at least two work items per head
    need = _lib.lib().uc_attend_workspace_size(
        C.cast((C.POINTER(_lib.UcSegment) * 2)(C.pointer(seg.c), C.pointer(seg.c)), C.c_void_p), 2, 28, 8)
    assert need > 8 << 20
    q = _dev(synth.make_q(408, B, 28, 8))
    out = torch.empty_like(q)
    lse = torch.empty((B, 28, 8), device=DEV)
    mass = torch.empty((B, 28, 8, 2), device=DEV)
    n0 = _lib.lib().uc_launch_count()
    assert _call_static(q, segs, out, lse, mass) == _lib.UC_ERR_OOM
    assert b"static" in _lib.lib().uc_last_error()
    assert _lib.lib().uc_launch_count() == n0
