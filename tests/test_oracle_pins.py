"""Pins of the CPU oracle to facts outside itself (no GPU needed).

Each test checks the oracle against brute force, a closed form, a library
routine or a hand-worked case, chosen so that a dropped term, a wrong sign or
index, or a transposed operand in the oracle fails at least one of them.
"""
import itertools
import json
import math
import os

import numpy as np
import pytest
import torch

import synth
from oracle import attention, policy, quant, scores, segment, select

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def _gold(name):
    with open(os.path.join(GOLD, name)) as f:
        return json.load(f)


# ------------------------------------------------------------------ scores

def test_scores_sum_to_heads_times_window():
    q = synth.make_q(1, 2, 8, 5)          # B=2, Hq=8, W=5
    k, _ = synth.make_kv(2, 2, 2, 37)     # Hkv=2 -> g=4
    s = scores.observation_scores(q, k)
    np.testing.assert_allclose(s.sum(axis=2), 4 * 5, rtol=1e-12)
    assert (s > 0).all()


def test_scores_single_key_is_exact():
    q = synth.make_q(3, 1, 28, 32)
    k, _ = synth.make_kv(4, 1, 4, 1)
    s = scores.observation_scores(q, k)
    np.testing.assert_allclose(s, 7 * 32, rtol=0, atol=1e-12)


def test_scores_match_library_attention_column_sums():
    """Column sums of the probability matrix from torch's SDPA (fp64, V = I)."""
    B, hq, hkv, W, N, d = 1, 6, 2, 4, 19, 16
    rng = np.random.default_rng(5)
    q = rng.standard_normal((B, hq, W, d))
    k = rng.standard_normal((B, hkv, N, d)) * 2
    s = scores.observation_scores(q, k)
    g = hq // hkv
    eye = torch.eye(N, dtype=torch.float64)
    for j in range(hkv):
        qt = torch.from_numpy(q[0, j * g:(j + 1) * g])           # [g, W, d]
        kt = torch.from_numpy(k[0, j]).expand(g, N, d)
        p = torch.nn.functional.scaled_dot_product_attention(qt, kt, eye.expand(g, N, N))
        np.testing.assert_allclose(s[0, j], p.sum(dim=(0, 1)).numpy(), rtol=1e-12)


def test_scores_dominant_key():
    q = np.zeros((1, 7, 3, 8))
    q[..., 0] = 1.0
    k = np.zeros((1, 1, 10, 8))
    k[0, 0, 6, 0] = 200.0                  # logit 200/sqrt(8) >> others
    s = scores.observation_scores(q, k)
    assert abs(s[0, 0, 6] - 21.0) < 1e-9


def test_type_mass_is_mean_over_heads_and_queries():
    q = synth.make_q(6, 1, 28, 32)
    k, _ = synth.make_kv(7, 1, 4, 64)
    s = scores.observation_scores(q, k)
    parts = [scores.type_mass(s[0], 0, 20, 28, 32), scores.type_mass(s[0], 20, 64, 28, 32)]
    assert abs(sum(parts) - 1.0) < 1e-12
    assert scores.chunk_mass([0.2, 0.4]) == pytest.approx(0.3)


def test_attention_type_mass_equals_observation_type_mass():
    B, hq, hkv, T, n = 2, 8, 2, 6, 90
    q = synth.make_q(31, B, hq, T)
    k, v = synth.make_kv(32, B, hkv, n)
    cuts = [(0, 25), (25, 31), (31, 90)]
    segs = [[[attention.Plain(k[b, j, lo:hi], v[b, j, lo:hi]) for j in range(hkv)] for b in range(B)]
            for lo, hi in cuts]
    _, _, mass = attention.attend(q, segs, hkv)
    got = scores.attention_type_mass(mass)
    s = scores.observation_scores(q, k)
    for b in range(B):
        want = [scores.type_mass(s[b], lo, hi, hq, T) for lo, hi in cuts]
        np.testing.assert_allclose(got[b], want, rtol=1e-12)
    np.testing.assert_allclose(got.sum(axis=1), 1.0, rtol=1e-12)


# ------------------------------------------------------------------ policy

def test_concentration_closed_forms():
    for n in (1, 9, 10, 11, 30, 768):
        c = policy.concentration(np.ones(n))
        assert c == pytest.approx(math.ceil(n / 10) / n, rel=1e-12)
    one_hot = np.zeros(50)
    one_hot[17] = 3.0
    assert policy.concentration(one_hot) == 1.0
    v = np.arange(1, 21, dtype=float)                 # top 2 of 20: 20 + 19
    assert policy.concentration(v) == pytest.approx(39 / 210)
    assert policy.assign_policy([0.5]) == "evict"
    assert policy.assign_policy([0.49, 0.5]) == "quant"
    assert policy.assign_policy([0.9, 0.2]) == "evict"


@pytest.mark.parametrize("case", _gold("eq2_budget_cases.json")["cases"])
def test_eq2_hand_worked(case):
    b = policy.allocate_budget(case["mass"], case["prev"], case["total"])
    np.testing.assert_allclose(b, case["expect"], rtol=1e-12, atol=1e-9)


def _water_level(m, cap, total):
    """Independent solution of Eq. 2's redistribution: b = min(cap, lam m)."""
    m = np.asarray(m, float)
    cap = np.asarray(cap, float)
    live = m > 0
    target = min(total, cap[live].sum())
    lo, hi = 0.0, 1.0
    while np.minimum(cap, hi * m)[live].sum() < target:
        hi *= 2
        if hi > 1e30:
            break
    for _ in range(200):
        mid = 0.5 * (lo + hi)
        if np.minimum(cap, mid * m)[live].sum() < target:
            lo = mid
        else:
            hi = mid
    return np.where(live, np.minimum(cap, hi * m), 0.0)


def test_eq2_matches_water_level_and_invariants():
    rng = np.random.default_rng(11)
    for _ in range(300):
        n = int(rng.integers(1, 7))
        m = rng.random(n) * (rng.random(n) > 0.2)
        cap = rng.random(n) * 100
        total = float(rng.random() * 150)
        b = policy.allocate_budget(m, cap, total)
        assert b.sum() <= total * (1 + 1e-9) + 1e-9
        assert (b <= cap + 1e-9).all()
        assert (b[m == 0] == 0).all()
        if m.sum() > 0:
            np.testing.assert_allclose(b, _water_level(m, cap, total), rtol=1e-7, atol=1e-7)
            free = (b < cap - 1e-7) & (m > 0)
            if free.sum() >= 2:
                r = b[free] / m[free]
                assert r.max() - r.min() <= 1e-7 * r.max()


@pytest.mark.parametrize("case", _gold("eq3_schedule_cases.json")["cases"])
def test_eq3_hand_worked(case):
    M = case["M"]
    rho = [case["rho_init"]]
    for c in range(1, len(case["expect_rho"])):
        rho.append(policy.retention_schedule(rho[-1], case["rho_init"], case["rho_min"], M[c], M[0]))
    np.testing.assert_allclose(rho, case["expect_rho"], rtol=1e-12)


def test_budget_mapping():
    n = 768
    keep, bits = policy.budget_to_policy("evict", 0.2 * n * 512, n)
    assert (keep, bits) == (153, 16)
    assert policy.budget_to_policy("quant", 0.35 * n * 512, n) == (n, 4)
    assert policy.budget_to_policy("quant", 0.2 * n * 512, n) == (n, 2)
    keep, bits = policy.budget_to_policy("quant", 0.1 * n * 512, n)
    assert bits == 2 and keep == math.floor(0.1 * n * 512 / 96)
    assert policy.bytes_per_token(16) == 512
    assert policy.bytes_per_token(4) == 160
    assert policy.bytes_per_token(2) == 96
    assert policy.keep_count(768, 0.2) == 153
    assert policy.keep_count(7168, 0.3) == 2150
    assert policy.keep_count(1792, 0.2) == 358
    assert policy.keep_count(100, 0.29) == 29
    assert policy.keep_count(3, 0.1) == 1


# ------------------------------------------------------------------ top-k

def _brute_topk(s, k):
    """The unique k-subset in which every kept token beats every dropped one
    (larger score, or equal score and lower index)."""
    n = len(s)
    found = []
    for sub in itertools.combinations(range(n), k):
        kept = set(sub)
        ok = all((s[i] > s[j]) or (s[i] == s[j] and i < j)
                 for i in kept for j in range(n) if j not in kept)
        if ok:
            found.append(sub)
    assert len(found) == 1
    return np.array(found[0])


@pytest.mark.parametrize("seed", range(12))
def test_topk_brute_force(seed):
    rng = np.random.default_rng(seed)
    n = int(rng.integers(1, 11))
    s = rng.integers(0, 4, size=n).astype(np.float32)     # many ties
    if seed % 3 == 0:
        s = rng.random(n).astype(np.float32)
    if seed == 5:
        s[:] = 1.0
    for k in range(1, n + 1):
        np.testing.assert_array_equal(select.topk_keep(s, k), _brute_topk(s, k))


def test_topk_signed_zero_and_nan():
    s = np.array([0.0, -0.0, 1.0, -0.0], dtype=np.float32)
    np.testing.assert_array_equal(select.topk_keep(s, 2), [0, 2])
    np.testing.assert_array_equal(select.topk_keep(s, 3), [0, 1, 2])
    with pytest.raises(ValueError):
        select.topk_keep(np.array([1.0, np.nan], np.float32), 1)


def test_topk_recent_tokens_forced():
    s = np.array([9, 8, 7, 0, 0], dtype=np.float32)
    np.testing.assert_array_equal(select.topk_keep(s, 3, n_recent=2), [0, 3, 4])
    np.testing.assert_array_equal(select.topk_keep(s, 2, n_recent=5), [3, 4])


# ------------------------------------------------------------------ quantizer

def test_fp16_rounding_reference_values():
    def f(x):
        with np.errstate(over="ignore"):
            return float(np.float32(x).astype(np.float16))
    assert f(65504.0) == 65504.0
    assert math.isinf(f(65520.0))
    assert f(65519.0) == 65504.0
    assert f(2.0 ** -24) == 2.0 ** -24            # smallest subnormal
    assert f(1.0 + 2.0 ** -11) == 1.0             # tie -> even
    assert f(1.0 + 3 * 2.0 ** -11) == 1.0 + 2.0 ** -9


def _check_codes(x, codes, s16, z16, bits, axis_params):
    qmax = 2 ** bits - 1
    xs = x.astype(np.float64)
    s = np.broadcast_to(s16.astype(np.float64), xs.shape)
    z = np.broadcast_to(z16.astype(np.float64), xs.shape)
    with np.errstate(divide="ignore", invalid="ignore"):
        r = (xs - z) / s
    zero = s == 0
    frac = r - np.floor(r)
    near_tie = np.abs(frac - 0.5) <= 8 * 2.0 ** -24 * np.maximum(np.abs(r), 1)
    exact = np.clip(np.where(np.abs(frac - 0.5) < 1e-300, 2 * np.round(r / 2), np.round(r)), 0, qmax)
    ok = zero | near_tie
    assert (codes[zero] == 0).all()
    assert (codes[~ok] == exact[~ok]).all()
    lo = np.clip(np.floor(r), 0, qmax)
    hi = np.clip(np.ceil(r), 0, qmax)
    assert ((codes[near_tie & ~zero] == lo[near_tie & ~zero]) |
            (codes[near_tie & ~zero] == hi[near_tie & ~zero])).all()
    # error bound: s/2 inside the range, fp16 slack of s and z at the ends
    deq = codes * s + z
    err = np.abs(xs - deq)
    inside = (r >= 0) & (r <= qmax) & ~zero
    assert (err[inside] <= s[inside] / 2 * (1 + 1e-6)).all()
    ulp = lambda v: np.spacing(np.abs(v).astype(np.float16)).astype(np.float64)
    slack = qmax * ulp(s) / 2 + ulp(z) / 2 + s / 2
    assert (err[~zero] <= slack[~zero] * (1 + 1e-6) + 1e-30).all()


@pytest.mark.parametrize("bits", [4, 2])
def test_quantize_k_nearest_level(bits):
    k, _ = synth.make_kv(21, 1, 1, 96)
    x = k[0, 0]
    codes, s16, z16 = quant.quantize_k(x, bits)
    assert codes.shape == (96, 128) and s16.shape == (3, 128)
    xg = x.reshape(3, 32, 128)
    _check_codes(xg, codes.reshape(3, 32, 128), s16[:, None, :], z16[:, None, :], bits, 1)
    # the oracle's dequantization reproduces x within the quantization bound
    deq = quant.dequantize_k(codes, s16, z16).reshape(3, 32, 128)
    bound = np.broadcast_to(s16.astype(np.float64)[:, None, :], deq.shape) * (2 ** bits) / 2
    assert (np.abs(deq - xg) <= bound + 1e-30).all()
    # zero-point is the group minimum rounded to fp16
    np.testing.assert_array_equal(z16, xg.min(axis=1).astype(np.float16))


@pytest.mark.parametrize("bits", [4, 2])
def test_quantize_v_nearest_level(bits):
    _, v = synth.make_kv(22, 1, 1, 40)
    x = v[0, 0]
    codes, s16, z16 = quant.quantize_v(x, bits)
    assert codes.shape == (40, 128) and s16.shape == (40, 4)
    xg = x.reshape(40, 4, 32)
    _check_codes(xg, codes.reshape(40, 4, 32), s16[:, :, None], z16[:, :, None], bits, 2)
    deq = quant.dequantize_v(codes, s16, z16).reshape(40, 4, 32)
    inside = np.abs(deq - xg) <= np.broadcast_to(s16.astype(np.float64)[:, :, None], deq.shape) * 0.5 * (1 + 1e-6)
    assert inside.mean() > 0.9


def test_quantize_degenerate_groups():
    x = np.zeros((32, 128), np.float32)
    x[:, 5] = 3.0                          # constant channel -> s = 0
    x[:, 6] = np.linspace(0, 1e-7, 32)     # range below fp16 resolution
    codes, s16, z16 = quant.quantize_k(x, 4)
    assert (codes[:, 5] == 0).all() and float(z16[0, 5]) == 3.0
    assert float(s16[0, 6]) == 0.0 and (codes[:, 6] == 0).all()
    with pytest.raises(quant.RangeError):
        quant.quantize_k(np.full((32, 128), 1e6, np.float32), 4)
    big = np.zeros((32, 128), np.float32)
    big[0, 0] = -60000.0
    big[1, 0] = 150000.0
    with pytest.raises(quant.RangeError):     # (mx - mn) / 3 > 65504 at int2
        quant.quantize_k(big, 2)
    with pytest.raises(quant.RangeError):
        quant.quantize_v(np.full((32, 128), np.nan, np.float32), 4)


def test_plan_batch_hand_worked():
    """The batch reading of §3.4 on hand-worked configurations."""
    n = 100
    assert policy.plan_batch([("full", n, 16)] * 3, n) == ("full", 16, True, [n] * 3)
    # one sequence evicts: the segment evicts, the others keep everything
    assert policy.plan_batch([("full", n, 16), ("evict", 40, 16)], n) == ("evict", 16, False, [n, 40])
    # int4 for one sequence, int2 for another: int2 for both, still every token
    assert policy.plan_batch([("quant", n, 4), ("quant", n, 2)], n) == ("quant", 2, False, [n, n])
    # one sequence had to evict under int2: evict then quantize, per-sequence keeps
    assert policy.plan_batch([("quant", n, 4), ("evict_quant", 70, 2)], n) == ("evict_quant", 2, False, [n, 70])
    assert policy.config_kind("evict", n, 16, n) == "full"
    assert policy.config_kind("quant", 10, 2, n) == "evict_quant"
    assert policy.chunk_mass([0.25, 0.5, 0.125], [True, False, True]) == 0.375


def test_quantize_zero_minimum_is_plus_zero():
    """Groups whose minimum is a signed zero store z = +0 (0x0000) whichever
    zero comes first, with codes that still dequantize within s / 2."""
    rng = np.random.default_rng(3)
    x = np.abs(rng.standard_normal((32, 128))).astype(np.float32) + np.float32(0.25)
    x[5, :] = 0.0
    x[9, :] = -0.0
    x[0, :64] = -0.0          # a -0 first in half of the channels' groups
    for bits in (4, 2):
        codes, s16, z16 = quant.quantize_k(x, bits)
        assert (z16.view(np.uint16) == 0).all()
        deq = quant.dequantize_k(codes, s16, z16)
        assert (np.abs(deq - x) <= s16.astype(np.float64)[0] / 2 * (1 + 2 ** -10) + 1e-12).all()
        codes, s16, z16 = quant.quantize_v(x, bits)
        zb = z16.view(np.uint16)
        assert (zb[5] == 0).all() and (zb[9] == 0).all() and (zb[0, :2] == 0).all()
        assert (z16[1:5].astype(np.float32) > 0).all()    # other tokens: a positive minimum
        assert ((codes[5] == 0) & (codes[9] == 0)).all()  # all-zero tokens (s = 0)


def test_quantize_zero_scale_is_plus_zero():
    """A group of zeros of both signs has scale +0 (0x0000) and zero-point +0
    whichever zero the minimum and maximum searches return: the parameters
    are formed from mx = -0, mn = +0 directly (the order that gives -0)."""
    for bits in (4, 2):
        s16, z16 = quant._params(np.float32([-0.0, 0.0, -0.0]), np.float32([-0.0, -0.0, 0.0]), bits)
        assert (s16.view(np.uint16) == 0).all() and (z16.view(np.uint16) == 0).all()
        x = np.zeros((32, 128), np.float32)
        x[::2, :] = -0.0
        x[:, 64:] = -0.0
        for fn in (quant.quantize_k, quant.quantize_v):
            codes, s16, z16 = fn(x, bits)
            assert (s16.view(np.uint16) == 0).all() and (z16.view(np.uint16) == 0).all()
            assert (codes == 0).all()


def test_quantize_handpicked_values():
    x = np.zeros((1, 128), np.float32)
    x[0, :32] = np.arange(32, dtype=np.float32) / 2     # 0 .. 15.5
    codes, s16, z16 = quant.quantize_v(x, 4)
    # s = 15.5 / 15 rounded to fp16, z = 0
    s = float(np.float16(np.float32(15.5) / np.float32(15)))
    assert float(s16[0, 0]) == s and float(z16[0, 0]) == 0.0
    expect = np.clip(np.rint((np.arange(32) / 2) / s), 0, 15)
    np.testing.assert_array_equal(codes[0, :32], expect)
    assert codes[0, 0] == 0 and codes[0, 31] == 15


# ------------------------------------------------------------------ segments

def test_packed_bytes_hand_worked():
    gold = _gold("packed_bytes_cases.json")
    for c in gold["cases"]:
        n = c["n_kept"]
        k, v = synth.make_kv(31, 1, 1, n)
        seg = segment.compress(k[0, 0], v[0, 0], None,
                               "full" if c["kind"] in ("full", "evict") else "quant", n, c["bits"])
        assert segment.stored_bytes(seg) == c["expect_bytes"]
    a, b = gold["ratios"]["single_layer_1k_overall"]
    assert a / b == pytest.approx(3.19, abs=0.005)


@pytest.mark.parametrize("bits", [4, 2])
def test_append_equals_one_shot(bits):
    k, v = synth.make_kv(41, 1, 1, 100)
    s = synth.make_scores(3, (100,))
    seg = segment.compress(k[0, 0], v[0, 0], s, "evict_quant", 30, bits)
    kn, vn = synth.make_kv(42, 1, 1, 40)
    grown = seg
    for i in range(40):
        grown = segment.append(grown, kn[0, 0, i:i + 1], vn[0, 0, i:i + 1], 100 + i)
    kept = np.concatenate([seg.kept_idx, 100 + np.arange(40)])
    kk = np.concatenate([k[0, 0], kn[0, 0]])
    vv = np.concatenate([v[0, 0], vn[0, 0]])
    once = segment._build("evict_quant", bits, kept, kk[kept], vv[kept])
    assert grown.n_groups == 2 and grown.tail == 6
    np.testing.assert_array_equal(grown.k_codes, once.k_codes)
    np.testing.assert_array_equal(grown.v_scale, once.v_scale)
    np.testing.assert_array_equal(grown.kept_idx, kept)


# ------------------------------------------------------------------ attention

def _sdpa(q_rows, k, v):
    qt = torch.from_numpy(q_rows)[None]
    return torch.nn.functional.scaled_dot_product_attention(
        qt, torch.from_numpy(k)[None], torch.from_numpy(v)[None])[0].numpy()


def test_attention_ratio_one_equals_library():
    q = synth.make_q(51, 2, 8, 3)
    k, v = synth.make_kv(52, 2, 2, 50)
    segs = [[[attention.Plain(k[b, j, :20], v[b, j, :20]) for j in range(2)] for b in range(2)],
            [[attention.Plain(k[b, j, 20:], v[b, j, 20:]) for j in range(2)] for b in range(2)]]
    O, lse, mass = attention.attend(q, segs, 2)
    for b in range(2):
        for h in range(8):
            j = h // 4
            ref = _sdpa(q[b, h].astype(np.float64), k[b, j].astype(np.float64), v[b, j].astype(np.float64))
            np.testing.assert_allclose(O[b, h], ref, rtol=1e-10, atol=1e-12)
            logits = q[b, h].astype(np.float64) @ k[b, j].astype(np.float64).T / math.sqrt(128)
            np.testing.assert_allclose(lse[b, h], np.log(np.exp(logits).sum(axis=1)), rtol=1e-12)
    np.testing.assert_allclose(mass.sum(axis=3), 1.0, rtol=1e-12)


def test_attention_eviction_equals_subset():
    q = synth.make_q(61, 1, 28, 1)
    k, v = synth.make_kv(62, 1, 4, 300)
    s = synth.make_scores(63, (4, 300))
    segs = [[[segment.compress(k[0, j], v[0, j], s[j], "evict", 60, 16) for j in range(4)]]]
    O, _, mass = attention.attend(q, segs, 4)
    for h in range(28):
        j = h // 7
        kept = select.topk_keep(s[j], 60)
        ref = _sdpa(q[0, h].astype(np.float64), k[0, j, kept].astype(np.float64),
                    v[0, j, kept].astype(np.float64))
        np.testing.assert_allclose(O[0, h], ref, rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(mass[..., 0], 1.0)


def test_attention_quantized_equals_dequantized_library():
    q = synth.make_q(71, 1, 28, 2)
    k, v = synth.make_kv(72, 1, 4, 75)
    segs = [[[segment.compress(k[0, j], v[0, j], None, "quant", 75, 4) for j in range(4)]]]
    O, _, _ = attention.attend(q, segs, 4)
    for h in (0, 13, 27):
        sg = segs[0][0][h // 7]
        kh = np.concatenate([quant.dequantize_k(sg.k_codes, sg.k_scale, sg.k_zero),
                             k[0, h // 7, 64:].astype(np.float64)])
        vh = np.concatenate([quant.dequantize_v(sg.v_codes, sg.v_scale, sg.v_zero),
                             v[0, h // 7, 64:].astype(np.float64)])
        np.testing.assert_allclose(O[0, h], _sdpa(q[0, h].astype(np.float64), kh, vh), rtol=1e-10, atol=1e-12)


def test_attention_lse_merge_of_parts():
    """Two parts attended separately and merged by log-sum-exp equal the whole."""
    q = synth.make_q(81, 1, 28, 3)
    k, v = synth.make_kv(82, 1, 4, 90)
    mk = lambda lo, hi: [[[attention.Plain(k[0, j, lo:hi], v[0, j, lo:hi]) for j in range(4)]]]
    O, lse, mass = attention.attend(q, mk(0, 90), 4)
    O1, l1, _ = attention.attend(q, mk(0, 33), 4)
    O2, l2, _ = attention.attend(q, mk(33, 90), 4)
    L = np.logaddexp(l1, l2)
    merged = np.exp(l1 - L)[..., None] * O1 + np.exp(l2 - L)[..., None] * O2
    np.testing.assert_allclose(merged, O, rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(L, lse, rtol=1e-12)
    segs = [mk(0, 33)[0], mk(33, 90)[0]]
    _, _, m2 = attention.attend(q, [segs[0], segs[1]], 4)
    np.testing.assert_allclose(m2[..., 0], np.exp(l1 - lse), rtol=1e-10)


# ---------------------------------------------------------- re-compression

def test_round_bf16_matches_library_and_ties():
    rng = np.random.default_rng(11)
    x = np.concatenate([rng.standard_normal(20000).astype(np.float32) * np.float32(100),
                        rng.standard_normal(2000).astype(np.float32) * np.float32(1e-38),
                        np.float32([0.0, -0.0, 65504.0, 3.0e38])])
    ref = torch.from_numpy(x).to(torch.bfloat16).float().numpy()
    np.testing.assert_array_equal(quant.round_bf16(x).view(np.uint32), ref.view(np.uint32))
    # hand-worked ties in [1, 2), where one bf16 step is 2^-7
    cases = [(1 + 2**-8, 1.0), (1 + 3 * 2**-8, 1 + 2**-6), (-(1 + 2**-8), -1.0),
             (1 + 2**-8 + 2**-20, 1 + 2**-7), (1 + 2**-9, 1.0)]
    for val, want in cases:
        assert quant.round_bf16(np.float32([val]))[0] == np.float32(want)


def test_rebuild_rounds_through_fp32():
    # just above a bf16 tie by less than half an fp32 step: fp32 first lands
    # on the tie, which then goes to even (a single rounding would go up)
    assert quant.rebuild_bf16(np.array([1 + 2**-8 + 2**-30]))[0] == np.float32(1.0)
    assert quant.rebuild_bf16(np.array([1 + 2**-8 + 2**-22]))[0] == np.float32(1 + 2**-7)


def _on_grid(seed, n, bits):
    """K, V [n, 128] whose quantization groups sit exactly on a grid: scale
    2^-e and zero -m * scale vary per group, and every group holds codes 0
    and qmax, so quantization recovers scale, zero and codes exactly."""
    rng = np.random.default_rng(seed)
    qmax = 2 ** bits - 1
    ng = n // 32

    k = np.zeros((n, 128), np.float64)
    v = np.zeros((n, 128), np.float64)
    for g in range(ng):
        for ch in range(128):
            e, m = 2 + (ch + 3 * g) % 5, (7 * ch + g) % (qmax + 1)
            c = rng.integers(0, qmax + 1, size=32)
            lo, hi = rng.choice(32, size=2, replace=False)
            c[lo], c[hi] = 0, qmax
            k[32 * g:32 * g + 32, ch] = (c - m) * 2.0 ** -e
    for t in range(32 * ng):
        for grp in range(4):
            e, m = 2 + (t + grp) % 5, (5 * t + 3 * grp) % (qmax + 1)
            c = rng.integers(0, qmax + 1, size=32)
            lo, hi = rng.choice(32, size=2, replace=False)
            c[lo], c[hi] = 0, qmax
            v[t, 32 * grp:32 * grp + 32] = (c - m) * 2.0 ** -e
    tail = n - 32 * ng
    k[32 * ng:] = synth.bf16_round(rng.standard_normal((tail, 128)).astype(np.float32))
    v[32 * ng:] = synth.bf16_round(rng.standard_normal((tail, 128)).astype(np.float32))
    return k.astype(np.float32), v.astype(np.float32)


@pytest.mark.parametrize("bits", [4, 2])
def test_requantize_on_grid_is_exact(bits):
    n = 32 * 3 + 11
    k, v = _on_grid(40 + bits, n, bits)
    seg = segment.compress(k, v, None, "quant", n, bits)
    kr, vr = segment.stored_rows(seg)
    np.testing.assert_array_equal(kr, k)
    np.testing.assert_array_equal(vr, v)
    again = segment.recompress(seg, None, "quant", n, bits)
    for name in ("k_codes", "k_scale", "k_zero", "v_codes", "v_scale", "v_zero", "kept_idx"):
        np.testing.assert_array_equal(getattr(again, name), getattr(seg, name))


def test_requantize_on_grid_then_evict_equals_one_shot():
    n = 32 * 4 + 5
    k, v = _on_grid(44, n, 4)
    s = np.random.default_rng(45).permutation(n).astype(np.float32)
    src = segment.compress(k, v, None, "quant", n, 4)
    got = segment.recompress(src, s, "evict_quant", 70, 2)
    want = segment.compress(k, v, s, "evict_quant", 70, 2)
    np.testing.assert_array_equal(got.kept_idx, np.sort(np.argsort(-s)[:70]))
    for name in ("kept_idx", "k_codes", "k_scale", "k_zero", "v_codes", "v_scale", "v_zero", "k_kept"):
        np.testing.assert_array_equal(getattr(got, name), getattr(want, name))


@pytest.mark.parametrize("recent", [0, 5])
def test_nested_eviction_equals_one_shot(recent):
    n = 300
    k, v = synth.make_kv(21, 1, 1, n)
    k, v = k[0, 0], v[0, 0]
    s = np.random.default_rng(22).permutation(n).astype(np.float32)
    first = segment.compress(k, v, s, "evict", 120, 16, recent)
    for keep in (120, 77, 6, 1):
        got = segment.recompress(first, s, "evict", keep, 16, recent)
        want = segment.compress(k, v, s, "evict", keep, 16, recent)
        np.testing.assert_array_equal(got.kept_idx, want.kept_idx)
        np.testing.assert_array_equal(got.k_kept, want.k_kept)
        np.testing.assert_array_equal(got.v_kept, want.v_kept)
    got = segment.recompress(first, s, "evict_quant", 64, 4, recent)
    want = segment.compress(k, v, s, "evict_quant", 64, 4, recent)
    for name in ("kept_idx", "k_codes", "k_scale", "v_codes", "v_zero"):
        np.testing.assert_array_equal(getattr(got, name), getattr(want, name))
    full = segment.compress(k, v, None, "full", n, 16)
    got = segment.recompress(full, s, "evict", 50, 16)
    np.testing.assert_array_equal(got.kept_idx, np.sort(np.argsort(-s)[:50]))
    np.testing.assert_array_equal(got.k_kept, k[got.kept_idx])


# ------------------------------------------------- decode heavy-hitter scores

def test_token_probabilities_equal_observation_scores_and_mass():
    B, hq, hkv, T = 2, 14, 2, 3
    q = synth.make_q(61, B, hq, T)
    k, v = synth.make_kv(62, B, hkv, 120)
    cuts = [(0, 30), (30, 31), (31, 120)]
    segs = [[[attention.Plain(k[b, j, lo:hi], v[b, j, lo:hi]) for j in range(hkv)] for b in range(B)]
            for lo, hi in cuts]
    probs = attention.token_probabilities(q, segs, hkv)
    obs = scores.observation_scores(q, k)
    for (lo, hi), p in zip(cuts, probs):
        np.testing.assert_allclose(p, obs[:, :, lo:hi], rtol=1e-12, atol=1e-15)
    total = sum(p.sum(axis=2) for p in probs)
    np.testing.assert_allclose(total, (hq // hkv) * T, rtol=1e-12)
    _, _, mass = attention.attend(q, segs, hkv)
    g = hq // hkv
    for s, p in enumerate(probs):
        for j in range(hkv):
            np.testing.assert_allclose(p[:, j].sum(axis=1), mass[:, j * g:(j + 1) * g, :, s].sum(axis=(1, 2)),
                                       rtol=1e-12)


def test_streaming_reeviction_keeps_heavy_hitters_and_window():
    # accumulated scores by logical index; re-eviction keeps the window of
    # most recent stored tokens plus the highest-scoring older ones
    n = 50
    k, v = synth.make_kv(63, 1, 1, n)
    kept = np.sort(np.random.default_rng(64).choice(200, size=n, replace=False))
    seg = segment._build("evict", 16, kept.astype(np.int64), k[0, 0], v[0, 0])
    acc = np.random.default_rng(65).permutation(200).astype(np.float64)
    out = segment.recompress(seg, acc, "evict", 20, 16, n_recent=6)
    window = kept[-6:]
    older = kept[:-6]
    heavy = older[np.argsort(-acc[older])[:14]]
    np.testing.assert_array_equal(out.kept_idx, np.sort(np.concatenate([heavy, window])))
    rows = np.searchsorted(kept, out.kept_idx)
    np.testing.assert_array_equal(out.k_kept, k[0, 0][rows])
