"""Dense multi-query attention (the tensor-core path of uc_attend, T > 8)
against the CPU oracle.

Queries attend without a mask to every stored token of every segment (the
denoising / editing calls: latent queries over the compressed cache and the
current latents themselves). Checked element-wise within 2e-3 of the row's
max |O| beyond each element's own bf16 output rounding; lse and segment mass
within the fp32 / hi-lo key bound.
"""
import numpy as np
import pytest
import torch

import synth
from oracle import attention as oattn
from oracle import segment as oseg
from tests import _packed

pytestmark = pytest.mark.gpu
uc = pytest.importorskip("paper_2609_32831_gb300")
DEV = "cuda"


def dev(x):
    return torch.from_numpy(np.ascontiguousarray(x, np.float32)).to(torch.bfloat16).to(DEV)


def host(t):
    return t.detach().float().cpu().numpy()


def _mix(seed, B, hkv, spec):
    """spec: list of (n, kind, keep, bits) -> GPU segments and oracle twins."""
    N = sum(s[0] for s in spec)
    k, v = synth.make_kv(seed, B, hkv, N)
    sc = synth.make_scores(seed, (B, hkv, N))
    kd, vd, sd = dev(k), dev(v), torch.from_numpy(sc).to(DEV)
    gs, os_ = [], []
    off = 0
    for n, kind, keep, bits in spec:
        if kind == "full":
            gs.append(uc.Segment.view(kd, vd, off, n))
            os_.append([[oattn.Plain(k[b, j, off:off + n], v[b, j, off:off + n]) for j in range(hkv)]
                        for b in range(B)])
        else:
            kp = keep if hasattr(keep, "__len__") else [keep] * B
            g = uc.Segment(kind, bits, B, hkv, n, max(kp), DEV)
            g.set_keep(kp)
            uc.compress_segment(kd, vd, g, begin=off, scores=sd)
            gs.append(g)
            os_.append([[oseg.compress(k[b, j, off:off + n], v[b, j, off:off + n], sc[b, j, off:off + n], kind,
                                       kp[b], bits) for j in range(hkv)] for b in range(B)])
        off += n
    return gs, os_


CASES = {
    "one_tile_bf16": (1, 128, [(64, "full", 64, 16)]),
    "partial_tiles_bf16": (2, 200, [(100, "full", 100, 16), (77, "full", 77, 16)]),
    "quant_int4": (1, 128, [(96, "quant", 96, 4)]),
    "text_latent_self": (2, 256, [(64, "full", 64, 16), (300, "quant", 300, 4), (256, "full", 256, 16)]),
    "editing_mix": (2, 130, [(40, "full", 40, 16), (320, "quant", 320, 4), (400, "evict", 80, 16),
                             (192, "full", 192, 16)]),
    "int2_ragged": (3, 160, [(90, "evict_quant", [33, 64, 1], 2), (70, "full", 70, 16)]),
}


@pytest.mark.parametrize("case", list(CASES))
def test_dense_parity(case):
    B, T, spec = CASES[case]
    hkv = 4
    gs, os_ = _mix(sum(map(ord, case)), B, hkv, spec)
    q = synth.make_q(7, B, 28, T)
    O, lse, mass = uc.attend(dev(q), gs)
    rO, rl, rm = oattn.attend(q, os_, hkv)
    assert _packed.attention_error(host(O), rO) <= _packed.ATTN_RTOL
    bound = _packed.logit_error_bound(q, os_, hkv, [False] * len(spec))
    assert (np.abs(host(lse) - rl) <= bound + 1e-5).all()
    assert (np.abs(host(mass) - rm) <= 2 * bound[..., None] + 1e-5).all()


def test_dense_issue_orders_agree_bitwise():
    """P(j) shares tensor memory with S(j+1) of its Q tile; the default issue
    order relies on the tensor pipe reading P before the next Q K^T writes
    there. Waiting for P V to complete first must give the same bits."""
    B, T, spec = 2, 700, CASES["editing_mix"][2]
    gs, _ = _mix(99, B, 4, spec)
    q = dev(synth.make_q(8, B, 28, T))
    runs = []
    for serial in (False, True, False):
        prev = uc.set_dense_serial_pv(serial)
        try:
            O, lse, mass = uc.attend(q, gs)
            torch.cuda.synchronize()
            runs.append((O.view(torch.int16).cpu(), lse.cpu(), mass.cpu()))
        finally:
            uc.set_dense_serial_pv(prev)
    for r in runs[1:]:
        assert all(torch.equal(a, b) for a, b in zip(runs[0], r))


@pytest.mark.parametrize("name", ["denoise_4k", "edit_4k"])
def test_dense_full_size_sampled(name):
    """One layer of the denoising / editing workload at full size (batch 4,
    4096 latent queries, every segment of the workload, int4 latent cache),
    in the launch configuration the benchmark times; 16 query positions of
    every (sequence, head) checked against the oracle."""
    wl = synth.workload(name)
    B, T, hkv = wl.batch, wl.q_tokens, 4
    spec = []
    for s in wl.segments:
        if s.name == "latent":
            continue
        keep = s.n if s.kind in ("full", "quant") else max(1, int(np.floor(s.keep_frac * s.n)))
        spec.append((s.n, s.kind, keep, s.bits))
    gs, os_ = _mix(404 + len(name), B, hkv, spec)
    kl, vl = synth.make_kv(405, B, hkv, T)
    kld, vld = dev(kl), dev(vl)
    gs.append(uc.Segment.view(kld, vld, 0, T))
    os_.append([[oattn.Plain(kl[b, j], vl[b, j]) for j in range(hkv)] for b in range(B)])
    q = synth.make_q(406, B, 28, T)
    O, lse, mass = uc.attend(dev(q), gs)
    torch.cuda.synchronize()
    idx = np.sort(np.random.default_rng(7).choice(T, 16, replace=False))
    idx[0], idx[-1] = 0, T - 1
    qs = np.ascontiguousarray(q[:, :, idx])
    rO, rl, rm = oattn.attend(qs, os_, hkv)
    assert _packed.attention_error(host(O)[:, :, idx], rO) <= _packed.ATTN_RTOL
    bound = _packed.logit_error_bound(qs, os_, hkv, [False] * len(gs))
    assert (np.abs(host(lse)[:, :, idx] - rl) <= bound + 1e-5).all()
    assert (np.abs(host(mass)[:, :, idx] - rm) <= 2 * bound[..., None] + 1e-5).all()
