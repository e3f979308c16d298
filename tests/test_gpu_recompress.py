"""GPU parity of progressive re-compression and of the Eq. 1 mass reduction.

A source segment is compressed on the GPU and by the oracle from the same
seeded inputs (their parity is covered elsewhere), then compressed further on
both sides. Kept indices, bf16 rows, codes, scales and zero-points must match
bit for bit; the source must be left untouched.
"""
import numpy as np
import pytest
import torch

import synth
from oracle import attention as oattn
from oracle import scores as oscores
from oracle import segment as oseg
from tests import _packed
from tests.test_gpu_kernels import _check_quant_block, dev, host

pytestmark = pytest.mark.gpu

uc = pytest.importorskip("paper_2609_32831_gb300")
DEV = "cuda"
B, HKV = 2, 4


def _source(kind, bits, n, keep, k, v, s):
    """GPU segment + oracle slices for one source configuration."""
    if kind == "full":
        kd, vd = dev(k), dev(v)
        seg = uc.Segment.view(kd, vd, 0, n)
        seg._keepalive = (kd, vd)
        refs = [[oseg.compress(k[b, j], v[b, j], None, "full", n, 16) for j in range(HKV)] for b in range(B)]
        return seg, refs
    seg = uc.Segment(kind, bits, B, HKV, n, max(keep), DEV)
    seg.set_keep(keep)
    uc.compress_segment(dev(k), dev(v), seg, scores=torch.from_numpy(s).to(DEV))
    refs = [[oseg.compress(k[b, j], v[b, j], s[b, j], kind, keep[b], bits) for j in range(HKV)]
            for b in range(B)]
    return seg, refs


def _check(seg, refs):
    cap = seg.c.cap
    assert seg.tensor("n_kept").cpu().tolist() == [refs[b][0].n_kept for b in range(B)]
    if seg.c.bits < 16:
        for b in range(B):
            for j in range(HKV):
                _check_quant_block(seg, b, j, refs[b][j])
        return
    kk = host(seg.tensor("k").view(B * HKV, cap, 128))
    vv = host(seg.tensor("v").view(B * HKV, cap, 128))
    idx = seg.tensor("kept_idx").view(B * HKV, cap).cpu().numpy()
    for b in range(B):
        for j in range(HKV):
            r = refs[b][j]
            np.testing.assert_array_equal(idx[b * HKV + j, :r.n_kept], r.kept_idx)
            np.testing.assert_array_equal(kk[b * HKV + j, :r.n_kept], r.k_kept)
            np.testing.assert_array_equal(vv[b * HKV + j, :r.n_kept], r.v_kept)


def _snapshot(seg):
    return {name: t.clone() for name, t in seg._t.items() if t is not None}


CASES = [
    # src kind, src bits, src keep fraction, dst kind, dst bits, dst keep fraction, n_recent
    ("evict", 16, 0.5, "evict", 16, 0.3, 0),
    ("evict", 16, 0.5, "evict", 16, 0.25, 8),
    ("evict", 16, 0.6, "evict_quant", 4, 0.4, 0),
    ("quant", 4, 1.0, "quant", 2, 1.0, 0),
    ("quant", 4, 1.0, "evict_quant", 2, 0.3, 0),
    ("quant", 2, 1.0, "evict", 16, 0.1, 3),
    ("evict_quant", 4, 0.5, "evict_quant", 2, 0.2, 0),
    ("evict_quant", 4, 0.5, "quant", 4, None, 0),
    ("full", 16, 1.0, "quant", 4, 1.0, 0),
    ("full", 16, 1.0, "evict", 16, 0.2, 0),
]


@pytest.mark.parametrize("case", CASES, ids=lambda c: f"{c[0]}{c[1]}-{c[3]}{c[4]}-r{c[6]}")
@pytest.mark.parametrize("n", [1000, 77])
def test_recompress_parity(case, n):
    skind, sbits, sfrac, dkind, dbits, dfrac, recent = case
    k, v = synth.make_kv(300 + n, B, HKV, n)
    s = synth.make_scores(301 + n, (B, HKV, n), tie_frac=0.3)
    skeep = [max(1, int(n * sfrac)), max(1, int(n * sfrac * 0.7))] if skind in ("evict", "evict_quant") \
        else [n, n]
    src, srefs = _source(skind, sbits, n, skeep, k, v, s)
    if dfrac is None or dkind == "quant":
        dkeep = list(skeep)
    else:
        dkeep = [max(1, int(x * dfrac / sfrac)) for x in skeep]
        dkeep = [min(a, b) for a, b in zip(dkeep, skeep)]
    dst = uc.Segment(dkind, dbits, B, HKV, n, max(dkeep), DEV)
    dst.set_keep(dkeep)
    before = _snapshot(src)
    uc.recompress_segment(src, dst, scores=torch.from_numpy(s).to(DEV), n_recent=recent)
    torch.cuda.synchronize()
    for name, t in before.items():
        assert torch.equal(t, src.tensor(name)), name
    drefs = [[oseg.recompress(srefs[b][j], s[b, j], dkind, dkeep[b], dbits, recent) for j in range(HKV)]
             for b in range(B)]
    _check(dst, drefs)
    assert dst.n_kept() == dkeep


def test_recompress_after_appends_and_to_nothing():
    n, steps = 150, 37
    k, v = synth.make_kv(41, B, HKV, n)
    s = synth.make_scores(42, (B, HKV, n + steps))
    src = uc.Segment("quant", 4, B, HKV, n, n + steps, DEV)
    src.set_keep([n] * B)
    uc.compress_segment(dev(k), dev(v), src)
    refs = [[oseg.compress(k[b, j], v[b, j], None, "quant", n, 4) for j in range(HKV)] for b in range(B)]
    kn, vn = synth.make_kv(43, B, HKV, steps)
    for t in range(steps):
        uc.append_next(src, dev(kn[:, :, t]), dev(vn[:, :, t]), 0)
        refs = [[oseg.append(refs[b][j], kn[b, j, t:t + 1], vn[b, j, t:t + 1], n + t) for j in range(HKV)]
                for b in range(B)]
    src.sync_host()
    assert src.n_kept() == [n + steps] * B
    keep = [60, 0]
    dst = uc.Segment("evict_quant", 2, B, HKV, n, 64, DEV)
    dst.set_keep(keep)
    sd = torch.from_numpy(s).to(DEV)
    uc.recompress_segment(src, dst, scores=sd)
    drefs = [[oseg.recompress(refs[b][j], s[b, j], "evict_quant", keep[b], 2) for j in range(HKV)]
             for b in range(B)]
    _check(dst, drefs)
    # the shrunken segment still attends like its oracle (sequence 0 only)
    q = synth.make_q(44, 1, 28, 1)
    one = uc.Segment("evict_quant", 2, 1, HKV, n + steps, 64, DEV)
    one.set_keep([keep[0]])
    src1 = uc.Segment("evict", 16, 1, HKV, n + steps, n + steps, DEV)
    src1.set_keep([n + steps])
    kk = np.concatenate([k, kn], axis=2)[:1]
    vv = np.concatenate([v, vn], axis=2)[:1]
    uc.compress_segment(dev(kk), dev(vv), src1, scores=sd[:1])
    uc.recompress_segment(src1, one, scores=sd[:1])
    r1 = [[oseg.recompress(oseg.compress(kk[0, j], vv[0, j], s[0, j], "evict", n + steps, 16), s[0, j],
                           "evict_quant", keep[0], 2) for j in range(HKV)]]
    O, lse, _ = uc.attend(dev(q), [one])
    rO, rl, _ = oattn.attend(q, [r1], HKV)
    assert _packed.attention_error(host(O), rO) <= _packed.ATTN_RTOL


def test_recompress_rejects_bad_calls():
    n = 64
    k, v = synth.make_kv(51, B, HKV, n)
    src = uc.Segment("quant", 4, B, HKV, n, n, DEV)
    src.set_keep([n] * B)
    uc.compress_segment(dev(k), dev(v), src)
    too_many = uc.Segment("evict", 16, B, HKV, n, n + 8, DEV)
    too_many.set_keep([n + 1, 3])
    with pytest.raises(uc.UniCacheError):
        uc.recompress_segment(src, too_many, scores=torch.zeros((B, HKV, n), device=DEV))
    no_scores = uc.Segment("evict", 16, B, HKV, n, n, DEV)
    no_scores.set_keep([3, 3])
    with pytest.raises(uc.UniCacheError):
        uc.recompress_segment(src, no_scores)
    with pytest.raises(uc.UniCacheError):
        uc.recompress_segment(src, src)
    other_b = uc.Segment("quant", 2, 1, HKV, n, n, DEV)
    other_b.set_keep([n])
    with pytest.raises(uc.UniCacheError):
        uc.recompress_segment(src, other_b)
    # a logical index outside the score array is reported, not read
    short = uc.Segment("evict", 16, B, HKV, n, n, DEV)
    short.set_keep([3, 3])
    ws = uc.Workspace(DEV)
    uc.recompress_segment(src, short, scores=torch.zeros((B, HKV, n - 10), device=DEV), ws=ws)
    assert ws.status() == 4            # UC_ERR_RANGE


@pytest.mark.parametrize("shape", [(1, 28, 1, 3), (2, 28, 4096, 4), (3, 8, 37, 8)])
def test_attention_mass_parity(shape):
    Bm, hq, T, ns = shape
    rng = np.random.default_rng(sum(shape))
    m = rng.random(shape, dtype=np.float32)
    m /= m.sum(axis=-1, keepdims=True)
    md = torch.from_numpy(m).to(DEV)
    got = uc.attention_mass(md)
    want = oscores.attention_type_mass(m)
    np.testing.assert_allclose(host(got), want, rtol=2e-6, atol=0)
    again = uc.attention_mass(md)
    assert torch.equal(got, again)          # fixed summation order
    uc.attention_mass(md, out=got, weight=0.5, accumulate=True)
    np.testing.assert_allclose(host(got), 1.5 * want, rtol=3e-6, atol=0)


def test_attention_mass_of_attend_output():
    n_text, n_vit = 60, 300
    k, v = synth.make_kv(61, B, HKV, n_text + n_vit)
    q = synth.make_q(62, B, 28, 5)
    kd, vd = dev(k), dev(v)
    segs = [uc.Segment.view(kd, vd, 0, n_text), uc.Segment.view(kd, vd, n_text, n_vit)]
    _, _, mass = uc.attend(dev(q), segs)
    got = host(uc.attention_mass(mass))
    ref = [[[oattn.Plain(k[b, j, lo:hi], v[b, j, lo:hi]) for j in range(HKV)] for b in range(B)]
           for lo, hi in ((0, n_text), (n_text, n_text + n_vit))]
    _, _, rmass = oattn.attend(q, ref, HKV)
    np.testing.assert_allclose(got, oscores.attention_type_mass(rmass), atol=1e-4)
