"""GPU parity of each kernel against the CPU oracle, through the C ABI.

Codes, scales, zero-points and kept indices must match bit for bit; scores
within fp32 accumulation error; attention within 2e-3 of the row's max |O|
beyond each element's own bf16 output rounding.
"""
import numpy as np
import pytest
import torch

import synth
from oracle import attention as oattn
from oracle import scores as oscores
from oracle import segment as oseg
from oracle import select as osel
from tests import _packed

pytestmark = pytest.mark.gpu

uc = pytest.importorskip("paper_2609_32831_gb300")
DEV = "cuda"


def dev(x):
    return torch.from_numpy(np.ascontiguousarray(x, np.float32)).to(torch.bfloat16).to(DEV)


def host(t):
    return t.detach().float().cpu().numpy()


def _check_quant_block(seg, b, j, ref):
    """Compare one (b, kvh) block of a quantized GPU segment with an oracle Seg."""
    bits = seg.bits
    bh = b * seg.n_kv_heads + j
    ng = ref.n_groups
    cap = seg.cap
    kc = seg.tensor("k_codes").view(seg.batch * seg.n_kv_heads, -1)[bh].cpu().numpy()
    vc = seg.tensor("v_codes").view(seg.batch * seg.n_kv_heads, -1)[bh].cpu().numpy()
    kp = seg.tensor("k_params").view(seg.batch * seg.n_kv_heads, -1)[bh].cpu().numpy()
    vp = seg.tensor("v_params").view(seg.batch * seg.n_kv_heads, -1)[bh].cpu().numpy()
    if ng:
        np.testing.assert_array_equal(_packed.unpack_k_codes(kc, ng, bits), ref.k_codes)
        np.testing.assert_array_equal(_packed.unpack_v_codes(vc, ng, bits), ref.v_codes)
        s, z = _packed.unpack_k_params(kp, ng)
        np.testing.assert_array_equal(s.view(np.uint16), ref.k_scale.view(np.uint16))
        np.testing.assert_array_equal(z.view(np.uint16), ref.k_zero.view(np.uint16))
        s, z = _packed.unpack_v_params(vp, ng)
        np.testing.assert_array_equal(s.view(np.uint16), ref.v_scale.view(np.uint16))
        np.testing.assert_array_equal(z.view(np.uint16), ref.v_zero.view(np.uint16))
    tail = ref.tail
    if tail:
        kt = host(seg.tensor("k").view(-1, 32, 128)[bh, :tail])
        vt = host(seg.tensor("v").view(-1, 32, 128)[bh, :tail])
        np.testing.assert_array_equal(kt, ref.k_kept[32 * ng:])
        np.testing.assert_array_equal(vt, ref.v_kept[32 * ng:])
    idx = seg.tensor("kept_idx").view(-1, cap)[bh, :ref.n_kept].cpu().numpy()
    np.testing.assert_array_equal(idx, ref.kept_idx)


@pytest.mark.parametrize("bits", [4, 2])
@pytest.mark.parametrize("n", [32, 75, 200, 1000])
def test_quantize_parity(bits, n):
    B, hkv = 2, 4
    k, v = synth.make_kv(100 + n + bits, B, hkv, n)
    seg = uc.Segment("quant", bits, B, hkv, n, n, DEV)
    seg.set_keep([n] * B)
    uc.compress_segment(dev(k), dev(v), seg)
    assert seg.tensor("n_kept").cpu().tolist() == [n] * B
    for b in range(B):
        for j in range(hkv):
            _check_quant_block(seg, b, j, oseg.compress(k[b, j], v[b, j], None, "quant", n, bits))


@pytest.mark.parametrize("bits", [4, 2])
def test_quantize_signed_zero_minimum(bits):
    """Groups whose minimum is +0 or -0 (both present, either first): the
    zero-point is stored as +0, bit-exact with the oracle."""
    B, hkv, n = 1, 2, 64
    k, v = synth.make_kv(41 + bits, B, hkv, n)
    bf = lambda x: torch.from_numpy(x).to(torch.bfloat16).float().numpy()   # inputs exact in bf16
    k, v = bf(np.abs(k) + np.float32(0.25)), bf(np.abs(v) + np.float32(0.25))
    k[0, 0, 3, :] = -0.0
    k[0, 0, 7, :] = 0.0
    k[0, 1, 40, :64] = -0.0
    k[0, 1, 35, :] = 0.0
    v[0, 0, 2, :] = -0.0
    v[0, 0, 3, 32:] = 0.0
    v[0, 0, 3, :32] = -0.0
    v[0, 1, 50, ::2] = -0.0
    v[0, 1, 50, 1::2] = 0.0
    seg = uc.Segment("quant", bits, B, hkv, n, n, DEV)
    seg.set_keep([n])
    uc.compress_segment(dev(k), dev(v), seg)
    for j in range(hkv):
        ref = oseg.compress(k[0, j], v[0, j], None, "quant", n, bits)
        assert (ref.k_zero.view(np.uint16)[j] == 0).all()   # head j's group j holds the zero rows
        _check_quant_block(seg, 0, j, ref)


@pytest.mark.parametrize("bits", [4, 2])
def test_quantize_zero_scale_and_clamped_codes(bits):
    """Groups of zeros of both signs (scale and zero-point +0, codes 0) and
    groups whose fp16 scale rounds far below range / qmax (fp16 subnormals),
    so that their largest element's quotient rounds above qmax and clamps:
    bit-exact with the oracle."""
    B, hkv, n = 1, 2, 64
    k, v = synth.make_kv(43 + bits, B, hkv, n)
    bf = lambda x: torch.from_numpy(np.ascontiguousarray(x)).to(torch.bfloat16).float().numpy()
    k, v = bf(k), bf(v)
    zeros = np.zeros(32, np.float32)
    zeros[1::2] = -0.0
    k[0, 0, :32, 5] = zeros                  # key channel 5, group 0
    v[0, 1, 40, 64:96] = zeros               # value token 40, channel group 2
    qmax = 2 ** bits - 1
    lo = np.float32(2.0 ** -20)
    hi = bf(np.array([2.0 ** -20 + 1.4 * qmax * 2.0 ** -24], np.float32))[0]   # s rounds to 2^-24
    ramp = np.where(np.arange(32) % 3 == 0, hi, lo).astype(np.float32)
    k[0, 1, 32:, 9] = ramp                   # key channel 9, group 1
    v[0, 0, 7, 32:64] = ramp                 # value token 7, channel group 1
    s16 = ((hi - lo) / np.float32(qmax) + np.float32(0)).astype(np.float16)
    assert s16 == np.float16(2.0 ** -24) and (hi - lo) / np.float32(s16) > qmax + 0.5   # the largest element clamps
    seg = uc.Segment("quant", bits, B, hkv, n, n, DEV)
    seg.set_keep([n])
    uc.compress_segment(dev(k), dev(v), seg)
    for j in range(hkv):
        ref = oseg.compress(k[0, j], v[0, j], None, "quant", n, bits)
        _check_quant_block(seg, 0, j, ref)
    ref0 = oseg.compress(k[0, 0], v[0, 0], None, "quant", n, bits)
    assert ref0.k_scale.view(np.uint16)[0, 5] == 0 and (ref0.k_codes[:32, 5] == 0).all()
    assert ref0.v_codes[7, 32:64].max() == qmax


@pytest.mark.parametrize("bits", [4, 2])
def test_evict_quant_parity(bits):
    B, hkv, n = 3, 4, 768
    k, v = synth.make_kv(7 + bits, B, hkv, n)
    s = synth.make_scores(8, (B, hkv, n), tie_frac=0.3)
    keep = [153, 64, 31]
    seg = uc.Segment("evict_quant", bits, B, hkv, n, max(keep), DEV)
    seg.set_keep(keep)
    uc.compress_segment(dev(k), dev(v), seg, scores=torch.from_numpy(s).to(DEV))
    assert seg.tensor("n_kept").cpu().tolist() == keep
    for b in range(B):
        for j in range(hkv):
            _check_quant_block(seg, b, j, oseg.compress(k[b, j], v[b, j], s[b, j], "evict_quant", keep[b], bits))


@pytest.mark.parametrize("n,keep,recent,ties", [(700, 140, 0, 0.5), (30000, 9000, 0, 0.2),
                                                (5000, 1500, 16, 0.0), (64, 64, 0, 0.9), (9, 1, 0, 1.0)])
def test_evict_topk_parity(n, keep, recent, ties):
    B, hkv = 2, 4
    begin = 17
    k, v = synth.make_kv(n + keep, B, hkv, n + begin)
    s = synth.make_scores(n, (B, hkv, n + begin), tie_frac=ties)
    if ties >= 1.0:
        s[:] = 1.0
    s[0, 1, begin + 3] = -0.0          # signed zero equals +0
    s[0, 1, begin + 4] = 0.0
    seg = uc.Segment("evict", 16, B, hkv, n, keep, DEV)
    seg.set_keep([keep, max(1, keep // 2)])
    uc.compress_segment(dev(k), dev(v), seg, begin=begin, scores=torch.from_numpy(s).to(DEV),
                        n_recent=recent)
    kk = host(seg.tensor("k").view(B * hkv, keep, 128))
    for b in range(B):
        kb = seg.n_kept()[b]
        for j in range(hkv):
            ref = osel.topk_keep(s[b, j, begin:], kb, recent)
            idx = seg.tensor("kept_idx").view(B * hkv, keep)[b * hkv + j, :kb].cpu().numpy()
            np.testing.assert_array_equal(idx, ref)
            np.testing.assert_array_equal(kk[b * hkv + j, :kb], k[b, j, begin + ref])


@pytest.mark.parametrize("n,keeps,recent,ties", [(118000, (23600, 35400), 0, 0.3), (20000, (6000, 19999), 16, 0.5),
                                                 (16384, (16384, 1), 0, 0.9)])
def test_evict_topk_parity_long(n, keeps, recent, ties):
    """Candidate lists of 16K and more with few (sequence, KV head) pairs take
    the cluster top-k (one cluster of CTAs per pair): kept indices bit-exact
    with the oracle's full sort, ties to the lower index, -0 equal to +0,
    recent tokens kept."""
    B, hkv = 2, 4
    begin = 17
    s = synth.make_scores(n + 3, (B, hkv, n + begin), tie_frac=ties)
    s[0, 1, begin + 3] = -0.0
    s[0, 1, begin + 4] = 0.0
    k = torch.zeros((B, hkv, n + begin, 128), dtype=torch.bfloat16, device=DEV)
    seg = uc.Segment("evict", 16, B, hkv, n, max(keeps), DEV)
    seg.set_keep(list(keeps))
    uc.compress_segment(k, k, seg, begin=begin, scores=torch.from_numpy(s).to(DEV), n_recent=recent)
    assert seg.tensor("n_kept").cpu().tolist() == list(keeps)
    idx = seg.tensor("kept_idx").view(B * hkv, max(keeps)).cpu().numpy()
    for b in range(B):
        for j in range(hkv):
            ref = osel.topk_keep(s[b, j, begin:], keeps[b], recent)
            np.testing.assert_array_equal(idx[b * hkv + j, :keeps[b]], ref)


def test_evict_nan_score_reports_range():
    B, hkv, n = 1, 4, 100
    k, v = synth.make_kv(5, B, hkv, n)
    s = synth.make_scores(5, (B, hkv, n))
    s[0, 2, 50] = np.nan
    seg = uc.Segment("evict", 16, B, hkv, n, 20, DEV)
    seg.set_keep([20])
    ws = uc.Workspace(DEV)
    uc.compress_segment(dev(k), dev(v), seg, scores=torch.from_numpy(s).to(DEV), ws=ws)
    assert ws.status() == 4            # UC_ERR_RANGE
    assert ws.status() == 0            # cleared


def test_quantize_overflow_reports_range():
    B, hkv, n = 1, 1, 32
    k = np.zeros((B, hkv, n, 128), np.float32)
    v = np.zeros_like(k)
    k[0, 0, 0, 0], k[0, 0, 1, 0] = -60000.0, 150000.0
    seg = uc.Segment("quant", 2, B, hkv, n, n, DEV)
    seg.set_keep([n])
    ws = uc.Workspace(DEV)
    uc.compress_segment(dev(k), dev(v), seg, ws=ws)
    assert ws.status() == 4


@pytest.mark.parametrize("B,W,N", [(1, 32, 1024), (2, 32, 3000), (1, 8, 77), (2, 16, 1)])
def test_scores_parity(B, W, N):
    q = synth.make_q(11 + N, B, 28, W)
    k, _ = synth.make_kv(12 + N, B, 4, N)
    got = host(uc.score_accumulate(dev(q), dev(k)))
    ref = oscores.observation_scores(q, k)
    np.testing.assert_allclose(got, ref, rtol=2e-5, atol=1e-7 * 7 * W)
    np.testing.assert_allclose(got.sum(-1), 7 * W, rtol=1e-5)


def test_segment_mass_parity():
    B, W, N = 2, 32, 1500
    q = synth.make_q(21, B, 28, W)
    k, _ = synth.make_kv(22, B, 4, N)
    sc = uc.score_accumulate(dev(q), dev(k))
    ranges = [(0, 150), (150, 1500), (10, 20)]
    got = host(uc.segment_mass(sc, ranges, 28, W))
    ref = oscores.observation_scores(q, k)
    for b in range(B):
        for s, (lo, hi) in enumerate(ranges):
            assert got[b, s] == pytest.approx(oscores.type_mass(ref[b], lo, hi, 28, W), rel=2e-5, abs=1e-9)


# ------------------------------------------------------------------ attention

def _build_mix(seed, B, hkv, sizes, kinds, keeps, bits):
    """GPU segments and their oracle twins over one shared context."""
    N = sum(sizes)
    k, v = synth.make_kv(seed, B, hkv, N)
    s = synth.make_scores(seed, (B, hkv, N), tie_frac=0.1)
    kd, vd, sd = dev(k), dev(v), torch.from_numpy(s).to(DEV)
    gsegs, osegs = [], []
    off = 0
    for n, kind, keep, bt in zip(sizes, kinds, keeps, bits):
        if kind == "full":
            g = uc.Segment.view(kd, vd, off, n)
            o = [[oattn.Plain(k[b, j, off:off + n], v[b, j, off:off + n]) for j in range(hkv)] for b in range(B)]
        else:
            kp = keep if hasattr(keep, "__len__") else [keep] * B
            g = uc.Segment(kind, bt, B, hkv, n, max(kp), DEV)
            g.set_keep(kp)
            uc.compress_segment(kd, vd, g, begin=off, scores=sd)
            o = [[oseg.compress(k[b, j, off:off + n], v[b, j, off:off + n], s[b, j, off:off + n], kind,
                                kp[b], bt) for j in range(hkv)] for b in range(B)]
        gsegs.append(g)
        osegs.append(o)
        off += n
    return gsegs, osegs


MIXES = {
    "text_full+vit_evict_int4": ([256, 768], ["full", "evict_quant"], [256, 153], [16, 4]),
    "four_kinds": ([200, 700, 300, 130], ["full", "evict", "evict_quant", "quant"], [200, 100, 150, 130], [16, 16, 2, 2]),
    "bf16_only": ([1000, 3000], ["evict", "full"], [333, 3000], [16, 16]),
    "quant_only_tail": ([77, 40], ["quant", "quant"], [77, 40], [4, 2]),
    "ragged_batch": ([300, 900], ["evict", "evict_quant"], [[1, 250, 37], [0 + 45, 600, 31]], [16, 4]),
}


@pytest.mark.parametrize("mix", list(MIXES))
@pytest.mark.parametrize("T", [1, 2, 5, 8])
def test_attend_parity(mix, T):
    sizes, kinds, keeps, bits = MIXES[mix]
    B = 3 if mix == "ragged_batch" else 2
    hkv = 4
    gsegs, osegs = _build_mix(sum(map(ord, mix)) + T, B, hkv, sizes, kinds, keeps, bits)
    q = synth.make_q(T, B, 28, T)
    O, lse, mass = uc.attend(dev(q), gsegs)
    rO, rl, rm = oattn.attend(q, osegs, hkv)
    assert _packed.attention_error(host(O), rO) <= _packed.ATTN_RTOL
    bound = _packed.logit_error_bound(q, osegs, hkv, [kd in ("quant", "evict_quant") for kd in kinds])
    assert (np.abs(host(lse) - rl) <= bound).all()
    assert (np.abs(host(mass) - rm) <= 2 * bound[..., None]).all()


LONG_MIXES = {
    # few (sequence, KV head) pairs and long segments: more than 32 items per
    # pair, merged by the separate merge kernel
    "four_long": (1, [3000, 40000, 20000, 500], ["full", "quant", "evict_quant", "evict"],
                  [3000, 40000, 6000, 300], [16, 2, 4, 16]),
    "ragged_two": (2, [1000, 60000], ["evict", "evict_quant"], [[1000, 400], [30000, 21000]], [16, 2]),
}


@pytest.mark.parametrize("mix", list(LONG_MIXES))
def test_attend_many_items_merge(mix):
    B, sizes, kinds, keeps, bits = LONG_MIXES[mix]
    hkv = 4
    gsegs, osegs = _build_mix(sum(map(ord, mix)), B, hkv, sizes, kinds, keeps, bits)
    plan = uc.attend_plan(gsegs, 28, 1)
    assert plan["items_per_bh"] > 32 and plan["merge_kernel"]
    q = synth.make_q(3, B, 28, 1)
    rO, rl, rm = oattn.attend(q, osegs, hkv)
    bound = _packed.logit_error_bound(q, osegs, hkv, [kd in ("quant", "evict_quant") for kd in kinds])
    ws = uc.Workspace(DEV)
    for _ in range(2):   # a second call on the same workspace
        O, lse, mass = uc.attend(dev(q), gsegs, ws=ws)
        assert ws.status() == 0
        assert _packed.attention_error(host(O), rO) <= _packed.ATTN_RTOL
        assert (np.abs(host(lse) - rl) <= bound).all()
        assert (np.abs(host(mass) - rm) <= 2 * bound[..., None]).all()


@pytest.mark.parametrize("bits", [2, 4, 16])
@pytest.mark.parametrize("T", [1, 3])
def test_attend_two_segments_ragged(bits, T):
    """Two long segments of one tile kind at batch 16 (seven items per
    (sequence, KV head) split between them) and a short bf16 segment of
    generated tokens (light: it takes no item from the long ones), lengths
    differing per sequence so every item boundary moves; one sequence's first
    segment holds a single token (its tail tile only)."""
    B, hkv = 16, 4
    rng = np.random.default_rng(11 + bits + T)
    kind = "evict" if bits == 16 else "evict_quant"
    sizes = [1500, 6000, 120]
    keeps = [[1] + [int(x) for x in rng.integers(1, 1400, B - 1)], [int(x) for x in rng.integers(1000, 6000, B)],
             [int(x) for x in rng.integers(1, 120, B)]]
    gsegs, osegs = _build_mix(60 + bits + T, B, hkv, sizes, [kind, kind, "evict"], keeps, [bits, bits, 16])
    q = synth.make_q(61 + T, B, 28, T)
    O, lse, mass = uc.attend(dev(q), gsegs)
    rO, rl, rm = oattn.attend(q, osegs, hkv)
    assert _packed.attention_error(host(O), rO) <= _packed.ATTN_RTOL
    bound = _packed.logit_error_bound(q, osegs, hkv, [bits != 16, bits != 16, False])
    assert (np.abs(host(lse) - rl) <= bound).all()
    assert (np.abs(host(mass) - rm) <= 2 * bound[..., None]).all()


def test_attend_empty_segment_and_repeat_calls():
    B, hkv = 2, 4
    gsegs, osegs = _build_mix(5, B, hkv, [100, 500], ["evict", "evict_quant"], [[1, 7], [64, 1]], [16, 4])
    empty = uc.Segment("evict", 16, B, hkv, 64, 64, DEV)      # never filled: 0 tokens
    gsegs.append(empty)
    osegs.append([[oattn.Plain(np.zeros((0, 128)), np.zeros((0, 128))) for j in range(hkv)] for b in range(B)])
    q = synth.make_q(3, B, 28, 1)
    ws = uc.Workspace(DEV)
    for _ in range(3):                      # counters re-arm between calls
        O, lse, mass = uc.attend(dev(q), gsegs, ws=ws)
        rO, rl, rm = oattn.attend(q, osegs, hkv)
        assert _packed.attention_error(host(O), rO) <= _packed.ATTN_RTOL
        bound = _packed.logit_error_bound(q, osegs, hkv, [False, True, False])
        assert (np.abs(host(mass) - rm) <= 2 * bound[..., None]).all()
        assert (np.abs(host(lse) - rl) <= bound).all()
        assert (host(mass)[..., 2] == 0).all()
    assert ws.status() == 0


@pytest.mark.parametrize("kind,bits", [("quant", 2), ("quant", 4), ("evict", 16), ("evict_quant", 4)])
def test_append_parity(kind, bits):
    B, hkv, n, steps = 2, 4, 90, 45
    k, v = synth.make_kv(31, B, hkv, n)
    s = synth.make_scores(31, (B, hkv, n))
    keep = n if kind == "quant" else 50
    seg = uc.Segment(kind, bits, B, hkv, n, keep + steps, DEV)
    seg.set_keep([keep] * B)
    uc.compress_segment(dev(k), dev(v), seg, scores=torch.from_numpy(s).to(DEV))
    refs = [[oseg.compress(k[b, j], v[b, j], s[b, j], kind, keep, bits) for j in range(hkv)] for b in range(B)]
    kn, vn = synth.make_kv(32, B, hkv, steps)
    q = synth.make_q(33, B, 28, 1)
    for t in range(steps):
        uc.append(seg, dev(kn[:, :, t]), dev(vn[:, :, t]), n + t)
        refs = [[oseg.append(refs[b][j], kn[b, j, t:t + 1], vn[b, j, t:t + 1], n + t) for j in range(hkv)]
                for b in range(B)]
        if t % 15 == 14:
            O, _, _ = uc.attend(dev(q), [seg])
            rO, _, _ = oattn.attend(q, [refs], hkv)
            assert _packed.attention_error(host(O), rO) <= _packed.ATTN_RTOL
    assert seg.n_kept() == [keep + steps] * B
    assert seg.tensor("n_kept").cpu().tolist() == [keep + steps] * B
    if bits < 16:
        for b in range(B):
            for j in range(hkv):
                _check_quant_block(seg, b, j, refs[b][j])
    else:
        kk = host(seg.tensor("k").view(B * hkv, seg.cap, 128))
        for b in range(B):
            for j in range(hkv):
                np.testing.assert_array_equal(kk[b * hkv + j, :keep + steps], refs[b][j].k_kept)


def test_attend_max_batch_and_heads():
    # 64 sequences x 8 KV heads (512 (b, kvh) pairs, more than the CTA slots):
    # merge counters, item plan and workspace layout at their largest
    B, hkv, hq = 64, 8, 56
    gsegs, osegs = _build_mix(77, B, hkv, [40, 70], ["full", "quant"], [40, 70], [16, 2])
    q = synth.make_q(78, B, hq, 1)
    ws = uc.Workspace(DEV)
    for _ in range(2):
        O, lse, mass = uc.attend(dev(q), gsegs, ws=ws)
    rO, rl, rm = oattn.attend(q, osegs, hkv)
    assert _packed.attention_error(host(O), rO) <= _packed.ATTN_RTOL
    assert ws.status() == 0
