"""Failure handling without a GPU fault: every wait inside the decode and
quantization kernels is bounded. A test hook withholds one tile's copies (one
K row of a group, for the quantizer), so the waits for it give up after the
wait limit (shortened here to 20 ms); the call must report UC_ERR_TIMEOUT
through its workspace status word, the launch must finish (every warp left:
the stream synchronises well inside a second), and the next call on the
same context must be correct again."""
import time

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


def _case(B=2, hkv=4):
    n_text, n_img = 300, 2000
    k, v = synth.make_kv(71, B, hkv, n_text + n_img)
    kd, vd = _dev(k), _dev(v)
    text = uc.Segment.view(kd, vd, 0, n_text)
    img = uc.Segment("quant", 4, B, hkv, n_img, n_img, DEV)
    img.set_keep([n_img] * B)
    uc.compress_segment(kd, vd, img, begin=n_text)
    q = synth.make_q(72, B, 28, 1)
    osegs = [[[oattn.Plain(k[b, j, :n_text], v[b, j, :n_text]) for j in range(hkv)] for b in range(B)],
             [[oseg.compress(k[b, j, n_text:], v[b, j, n_text:], None, "quant", n_img, 4) for j in range(hkv)]
              for b in range(B)]]
    return q, [text, img], osegs, (kd, vd)


@pytest.mark.parametrize("pos", [0, 5])
def test_bounded_wait_runs_out_and_reports_timeout(pos):
    q, segs, osegs, keep = _case()
    qd = _dev(q)
    ws = uc.Workspace(DEV)
    uc.attend(qd, segs, ws=ws)               # warm: library loaded, plan cached
    assert ws.status() == _lib.UC_OK
    prev = uc.set_wait_limit(20_000_000)
    try:
        uc.debug_withhold_tile(pos)
        t0 = time.perf_counter()
        uc.attend(qd, segs, ws=ws)
        status = ws.status()                  # synchronises the stream
        elapsed = time.perf_counter() - t0
    finally:
        uc.set_wait_limit(prev)
        uc.debug_withhold_tile(-1)
    assert status == _lib.UC_ERR_TIMEOUT
    assert elapsed < 1.0, elapsed             # a few 20 ms limits, not a hang
    # the context is usable and the next call is correct
    O, lse, mass = uc.attend(qd, segs, ws=ws)
    assert ws.status() == _lib.UC_OK
    rO, _, _ = oattn.attend(q, osegs, 4)
    assert _packed.attention_error(O.double().cpu().numpy(), rO) <= _packed.ATTN_RTOL


@pytest.mark.parametrize("bits", [4, 2])
def test_quantizer_wait_runs_out_and_reports_timeout(bits):
    from tests.test_gpu_kernels import _check_quant_block
    B, hkv, n = 2, 4, 256
    k, v = synth.make_kv(73 + bits, B, hkv, n)
    kd, vd = _dev(k), _dev(v)
    seg = uc.Segment("quant", bits, B, hkv, n, n, DEV)
    seg.set_keep([n] * B)
    ws = uc.Workspace(DEV)
    uc.compress_segment(kd, vd, seg, ws=ws)
    assert ws.status() == _lib.UC_OK
    prev = uc.set_wait_limit(20_000_000)
    try:
        uc.debug_withhold_tile(3)              # group 3 of the first (sequence, KV head)
        t0 = time.perf_counter()
        uc.compress_segment(kd, vd, seg, ws=ws)
        status = ws.status()
        elapsed = time.perf_counter() - t0
    finally:
        uc.set_wait_limit(prev)
        uc.debug_withhold_tile(-1)
    assert status == _lib.UC_ERR_TIMEOUT
    assert elapsed < 1.0, elapsed
    uc.compress_segment(kd, vd, seg, ws=ws)
    assert ws.status() == _lib.UC_OK
    kb = torch.from_numpy(np.ascontiguousarray(k)).to(torch.bfloat16).float().numpy()
    vb = torch.from_numpy(np.ascontiguousarray(v)).to(torch.bfloat16).float().numpy()
    for b in range(B):
        for j in range(hkv):
            ref = oseg.compress(kb[b, j], vb[b, j], None, "quant", n, bits)
            _check_quant_block(seg, b, j, ref)
