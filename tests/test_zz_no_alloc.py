"""uc_attend_static: decode attention for callers that cannot allocate device
memory for scratch space (for example a plug-in inside a host framework that
owns the device memory pool, or a latency-critical path that must not call
cudaMalloc). It takes no workspace: its scratch is a static device array
inside the library. These tests call it through the C ABI twice in a row and
check each result against uc_attend (which uses a caller workspace) and the
CPU oracle, within the attention tolerance used everywhere else; check that
invalid arguments get exactly uc_attend's status with nothing launched, that
a call needing more scratch than the array holds is refused before anything
runs and the next call still works, and that a small many-query call (the
tensor-core path, whose rebuilt rows also fit the array) matches uc_attend.

This file is collected last so that a run stopping at the first failure has
already run every other test; it also passes when run on its own.
"""
import ctypes as C

import numpy as np
import pytest
import torch

import synth
from oracle import attention as oattn
from oracle import segment as oseg
from tests import _packed

pytestmark = pytest.mark.gpu

uc = pytest.importorskip("paper_2609_32831_gb300")
from paper_2609_32831_gb300 import _lib  # noqa: E402

DEV = torch.device("cuda")


def _dev(x):
    return torch.from_numpy(np.ascontiguousarray(x, np.float32)).to(torch.bfloat16).to(DEV)


SIZES = [("view", 16, 0, 200, 200), ("evict", 16, 200, 700, 111), ("evict_quant", 4, 900, 600, 150),
         ("quant", 2, 1500, 130, 130)]


def _segments(B, hkv):
    """A text view, evicted bf16 rows, evicted + int4 rows and int2 rows.
    Returns the segments, the device tensors they view, and the host inputs."""
    N = sum(x[3] for x in SIZES)
    k, v = synth.make_kv(404, B, hkv, N)
    s = synth.make_scores(405, (B, hkv, N))
    kd, vd, sd = _dev(k), _dev(v), torch.from_numpy(s).to(DEV)
    segs = [uc.Segment.view(kd, vd, 0, 200)]
    for kind, bits, lo, n, keep in SIZES[1:]:
        g = uc.Segment(kind, bits, B, hkv, n, keep, DEV)
        g.set_keep([keep] * B)
        uc.compress_segment(kd, vd, g, begin=lo, scores=sd)
        segs.append(g)
    return segs, (kd, vd), (k, v, s)


def _oracle_segments(host_in, B, hkv):
    k, v, s = host_in
    out = []
    for kind, bits, lo, n, keep in SIZES:
        if kind == "view":
            out.append([[oattn.Plain(k[b, j, lo:lo + n], v[b, j, lo:lo + n]) for j in range(hkv)] for b in range(B)])
        else:
            out.append([[oseg.compress(k[b, j, lo:lo + n], v[b, j, lo:lo + n], s[b, j, lo:lo + n], kind, keep, bits)
                         for j in range(hkv)] for b in range(B)])
    return out


def _arr(segs):
    return (C.POINTER(_lib.UcSegment) * len(segs))(*[None if x is None else C.pointer(x.c) for x in segs])


def _call_attend(q, hq, T, segs, n_seg, out, lse, mass, ws):
    stream = C.c_void_p(torch.cuda.current_stream().cuda_stream)
    wp, wn = ws.get(64 << 20)
    return _lib.lib().uc_attend(C.c_void_p(q), hq, T, C.cast(_arr(segs), C.c_void_p), n_seg, C.c_void_p(out),
                                C.c_void_p(lse), C.c_void_p(mass), wp, wn, stream)


def _call_static(q, segs, out, lse, mass):
    B, hq, T, d = q.shape
    stream = C.c_void_p(torch.cuda.current_stream().cuda_stream)
    return _lib.lib().uc_attend_static(
        C.c_void_p(q.data_ptr()), hq, T, C.cast(_arr(segs), C.c_void_p), len(segs), C.c_void_p(out.data_ptr()),
        C.c_void_p(lse.data_ptr()), C.c_void_p(mass.data_ptr()), stream)


@pytest.mark.parametrize("T", [1, 3])
def test_attend_static_matches_attend(T):
    B, hkv = 3, 4
    segs, keep_alive, host_in = _segments(B, hkv)
    qh = synth.make_q(406 + T, B, 28, T)
    q = _dev(qh)
    ref_o, ref_lse, ref_mass = uc.attend(q, segs, ws=uc.Workspace(DEV))
    torch.cuda.synchronize()
    r_o = ref_o.double().cpu().numpy()
    # the oracle: uc_attend itself and the static entry point's first call
    osegs = _oracle_segments(host_in, B, hkv)
    o_o, o_lse, o_mass = oattn.attend(qh, osegs, hkv)
    bound = _packed.logit_error_bound(qh, osegs, hkv, [False, False, True, True])
    assert _packed.attention_error(r_o, o_o) <= _packed.ATTN_RTOL
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
        assert _packed.attention_error(out.double().cpu().numpy(), o_o) <= _packed.ATTN_RTOL
        assert (np.abs(lse.cpu().numpy() - o_lse) <= bound).all()
        assert (np.abs(mass.cpu().numpy() - o_mass) <= 2 * bound[..., None]).all()


def test_attend_static_refuses_oversized_calls_and_recovers():
    B, hkv = 64, 4
    n = 200  # 64 sequences x 4 heads, several items each: partials for T = 8 exceed 8 MiB
    seg = uc.Segment("evict", 16, B, hkv, n, n, DEV)
    seg.set_keep([n] * B)
    k, v = synth.make_kv(407, B, hkv, n)
    uc.compress_segment(_dev(k), _dev(v), seg, scores=torch.ones((B, hkv, n), device=DEV))
    segs = [seg, seg]  # two segments: at least two work items per head
    need = _lib.lib().uc_attend_workspace_size(C.cast(_arr(segs), C.c_void_p), 2, 28, 8)
    assert need > 8 << 20
    q = _dev(synth.make_q(408, B, 28, 8))
    out = torch.empty_like(q)
    lse = torch.empty((B, 28, 8), device=DEV)
    mass = torch.empty((B, 28, 8, 2), device=DEV)
    n0 = _lib.lib().uc_launch_count()
    assert _call_static(q, segs, out, lse, mass) == _lib.UC_ERR_OOM
    assert b"static" in _lib.lib().uc_last_error()
    assert _lib.lib().uc_launch_count() == n0
    # the call right after the refusal: the status word and merge counters
    # it clears give the same result as uc_attend
    q1 = _dev(synth.make_q(409, B, 28, 1))
    out1 = torch.full_like(q1, float("nan"))
    lse1 = torch.empty((B, 28, 1), device=DEV)
    mass1 = torch.empty((B, 28, 1, 2), device=DEV)
    assert _call_static(q1, segs, out1, lse1, mass1) == _lib.UC_OK, _lib.lib().uc_last_error()
    ref_o, ref_lse, _ = uc.attend(q1, segs, ws=uc.Workspace(DEV))
    torch.cuda.synchronize()
    assert _packed.attention_error(out1.double().cpu().numpy(), ref_o.double().cpu().numpy()) <= _packed.ATTN_RTOL
    np.testing.assert_allclose(lse1.cpu().numpy(), ref_lse.cpu().numpy(), rtol=0, atol=1e-5)


def test_attend_static_invalid_arguments_match_attend():
    """Every rejection happens before anything is launched or cleared, with
    uc_attend's status: a null segment pointer, segments of different batch,
    no segments, a null query, a query-head count that is not a multiple of
    the KV heads, and more than 64 query rows per KV head."""
    B, hkv = 2, 4
    segs, keep_alive, _ = _segments(B, hkv)
    other = uc.Segment("evict", 16, B + 1, hkv, 50, 50, DEV)
    other.set_keep([50] * (B + 1))
    k, v = synth.make_kv(410, B + 1, hkv, 50)
    uc.compress_segment(_dev(k), _dev(v), other, scores=torch.ones((B + 1, hkv, 50), device=DEV))
    q = _dev(synth.make_q(411, B, 28, 1))
    q10 = _dev(synth.make_q(412, B, 28, 10))
    out = torch.empty_like(q10)
    lse = torch.empty((B, 28, 10), device=DEV)
    mass = torch.empty((B, 28, 10, 4), device=DEV)
    ws = uc.Workspace(DEV)
    stream = C.c_void_p(torch.cuda.current_stream().cuda_stream)
    cases = [
        ("null segment", q.data_ptr(), 28, 1, [segs[0], None], 2),
        ("batch mismatch", q.data_ptr(), 28, 1, [segs[0], other], 2),
        ("no segments", q.data_ptr(), 28, 1, segs, 0),
        ("null query", 0, 28, 1, segs, 4),
        ("heads", q.data_ptr(), 30, 1, segs, 4),
        ("rows", q10.data_ptr(), 112, 3, segs, 4),   # 28 query heads per KV head x 3 tokens = 84 rows
    ]
    for name, qp, hq, T, ss, ns in cases:
        n0 = _lib.lib().uc_launch_count()
        a = _call_attend(qp, hq, T, ss, ns, out.data_ptr(), lse.data_ptr(), mass.data_ptr(), ws)
        b = _lib.lib().uc_attend_static(C.c_void_p(qp), hq, T, C.cast(_arr(ss), C.c_void_p), ns,
                                        C.c_void_p(out.data_ptr()), C.c_void_p(lse.data_ptr()),
                                        C.c_void_p(mass.data_ptr()), stream)
        assert a != _lib.UC_OK and a == b, (name, a, b)
        assert _lib.lib().uc_launch_count() == n0, name


def test_attend_static_many_queries():
    """16 query tokens per head take the tensor-core dense path; its rebuilt
    fp16 rows of this small cache fit the static array."""
    B, hkv = 1, 4
    segs, keep_alive, host_in = _segments(B, hkv)
    qh = synth.make_q(413, B, 28, 16)
    q = _dev(qh)
    need = _lib.lib().uc_attend_workspace_size(C.cast(_arr(segs), C.c_void_p), len(segs), 28, 16)
    assert 0 < need <= 8 << 20
    ref_o, ref_lse, ref_mass = uc.attend(q, segs, ws=uc.Workspace(DEV))
    o_o, _, _ = oattn.attend(qh, _oracle_segments(host_in, B, hkv), hkv)
    for call in range(2):
        out = torch.full_like(q, float("nan"))
        lse = torch.full((B, 28, 16), float("nan"), device=DEV)
        mass = torch.full((B, 28, 16, len(segs)), float("nan"), device=DEV)
        assert _call_static(q, segs, out, lse, mass) == _lib.UC_OK, _lib.lib().uc_last_error()
        torch.cuda.synchronize()
        assert torch.equal(out, ref_o)
        np.testing.assert_allclose(lse.cpu().numpy(), ref_lse.cpu().numpy(), rtol=0, atol=1e-6)
        assert _packed.attention_error(out.double().cpu().numpy(), o_o) <= _packed.ATTN_RTOL
