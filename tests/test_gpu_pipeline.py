"""End-to-end parity of the hot path through the engine (C-ABI calls only).

The oracle runs the same workload independently from the same synthetic
inputs: its own fp64 scores, Eq. 1 masses, Eq. 2 budgets, top-k, quantizer
and attention. Kept-token sets may differ only between tokens whose oracle
scores tie with the k-th score to within fp32 accumulation error; where the
sets agree (the usual case) the attention outputs are compared element-wise.
At full workload sizes the comparison runs on sampled (layer, sequence)
slices.
"""
import numpy as np
import pytest
import torch

import synth
from oracle import attention as oattn
from oracle import policy as opol
from oracle import scores as osc
from oracle import segment as oseg
from tests import _packed

pytestmark = pytest.mark.gpu
uc = pytest.importorskip("paper_2609_32831_gb300")
from paper_2609_32831_gb300.engine import CacheType, RequestCache, fixed_keep  # noqa: E402

DEV = torch.device("cuda")


def host(t):
    return t.detach().float().cpu().numpy()


def _kept_sets_consistent(got_idx, ref_idx, ref_scores, rel=5e-5):
    diff = set(got_idx.tolist()) ^ set(ref_idx.tolist())
    if not diff:
        return True
    kth = np.sort(ref_scores)[::-1][len(ref_idx) - 1]
    assert all(abs(ref_scores[i] - kth) <= rel * abs(kth) + 1e-12 for i in diff), "kept tokens differ"
    return False


def _oracle_layer(k, v, qwin, types, begins, keeps, bits_of, kinds_of, b):
    """Oracle segments of one (layer, sequence) slice; k, v [Hkv, N, 128]."""
    s = osc.observation_scores(qwin[None], k[None])[0]
    segs = []
    for a, t in enumerate(types):
        lo, hi = begins[a], begins[a] + t.n
        if kinds_of[a] == "full":
            segs.append([oattn.Plain(k[j, lo:hi], v[j, lo:hi]) for j in range(k.shape[0])])
        else:
            segs.append([oseg.compress(k[j, lo:hi], v[j, lo:hi], s[j, lo:hi], kinds_of[a], keeps[a], bits_of[a])
                         for j in range(k.shape[0])])
    return s, segs


def test_single_layer_1k_end_to_end():
    """256 text tokens kept in bf16 + 768 image tokens: top 20 % by 32-query
    window scores, int4 (keys per channel, values per token); one decode
    query; batch 1, seed 0."""
    wl = synth.workload("single_layer_1k")
    k, v = synth.make_kv(0, 1, 4, wl.n_ctx)
    qwin = synth.make_q(0, 1, 28, 32)
    q = synth.make_q(1, 1, 28, 1)
    to = lambda x: torch.from_numpy(x).to(torch.bfloat16).to(DEV)
    types = [CacheType("text", 256, "full"), CacheType("vit", 768, "evict_quant", 0.2, 4)]
    cache = RequestCache(types, 1, 1, DEV)
    sc = []
    cache.prefill(to(k)[None], to(v)[None], to(qwin)[None], scores_out=sc)
    out = cache.decode_step([to(q)], lse=[torch.empty((1, 28, 1), device=DEV)],
                            mass=[torch.empty((1, 28, 1, 2), device=DEV)])
    keep = fixed_keep(768, 0.2)
    assert keep == 153
    ref_s, osegs = _oracle_layer(k[0], v[0], qwin[0], types, [0, 256], [256, keep], [16, 4],
                                 ["full", "evict_quant"], 0)
    np.testing.assert_allclose(host(sc[0])[0], ref_s, rtol=2e-5, atol=1e-6)
    vit = cache.layers[0][1]
    same = True
    for j in range(4):
        got = vit.tensor("kept_idx").view(4, -1)[j, :keep].cpu().numpy()
        same &= _kept_sets_consistent(got, osegs[1][j].kept_idx, ref_s[j, 256:])
    if same:
        rO, _, _ = oattn.attend(q, [[osegs[0]], [osegs[1]]], 4)
        assert _packed.attention_error(host(out[0]), rO) <= _packed.ATTN_RTOL
    # realized compression of the image segment and of the whole cache
    assert vit.stored_bytes() == 4 * 33280
    assert cache.full_bytes() / cache.stored_bytes() == pytest.approx(524288 / 164352)


def _full_size_inputs(wl, device, seed0):
    L, B, N = wl.layers, wl.batch, wl.n_ctx
    K = torch.empty((L, B, 4, N, 128), dtype=torch.bfloat16, device=device)
    V = torch.empty_like(K)
    Qw = torch.empty((L, B, 28, wl.window, 128), dtype=torch.bfloat16, device=device)
    for l in range(L):
        k, v = synth.torch_kv(seed0 + l, B, 4, N, device)
        K[l].copy_(k)
        V[l].copy_(v)
        Qw[l].copy_(synth.torch_q(seed0 + 50 + l, B, 28, wl.window, device))
    return K, V, Qw


def test_understanding_decode_8k_sampled():
    """28 layers, batch 8, 8192 tokens: 512 text (bf16) + 7168 image tokens
    evicted to 30 % then int4 + 512 generated tokens in int2; decode steps
    append to the int2 segment. Sampled slices against the oracle."""
    wl = synth.workload("understanding_decode_8k")
    steps = 40
    types = [CacheType("text", 512, "full"), CacheType("vit", 7168, "evict_quant", 0.3, 4),
             CacheType("gen", 512, "quant", 1.0, 2, headroom=steps)]
    K, V, Qw = _full_size_inputs(wl, DEV, 2000)
    cache = RequestCache(types, wl.layers, wl.batch, DEV, append_to="gen")
    sc = []
    cache.prefill(K, V, Qw, scores_out=sc)
    g = torch.Generator(device=DEV)
    g.manual_seed(5)
    Qd = torch.randn((steps, wl.layers, wl.batch, 28, 1, 128), generator=g, device=DEV).to(torch.bfloat16)
    Kn = torch.randn((steps, wl.layers, wl.batch, 4, 128), generator=g, device=DEV).to(torch.bfloat16)
    Vn = torch.randn((steps, wl.layers, wl.batch, 4, 128), generator=g, device=DEV).to(torch.bfloat16)
    outs = None
    for t in range(steps):
        outs = cache.decode_step(Qd[t], Kn[t], Vn[t])
    assert cache.layers[0][2].n_kept() == [512 + steps] * wl.batch
    keep = fixed_keep(7168, 0.3)
    assert keep == 2150
    for l, b in [(0, 0), (27, 7), (13, 3)]:
        k = host(K[l, b])
        v = host(V[l, b])
        ref_s, osegs = _oracle_layer(k, v, host(Qw[l, b]), types, [0, 512, 7680], [512, keep, 512], [16, 4, 2],
                                     ["full", "evict_quant", "quant"], b)
        np.testing.assert_allclose(host(sc[l][b]), ref_s, rtol=2e-5, atol=1e-6)
        same = True
        for j in range(4):
            got = cache.layers[l][1].tensor("kept_idx").view(wl.batch * 4, -1)[b * 4 + j, :keep].cpu().numpy()
            same &= _kept_sets_consistent(got, osegs[1][j].kept_idx, ref_s[j, 512:7680])
        if not same:
            continue
        kn, vn = host(Kn[:, l, b]), host(Vn[:, l, b])
        gsegs = osegs[2]
        for t in range(steps):
            gsegs = [oseg.append(gsegs[j], kn[t, j:j + 1], vn[t, j:j + 1], 8192 + t) for j in range(4)]
        q = host(Qd[steps - 1, l, b])[None]
        rO, _, _ = oattn.attend(q, [[osegs[0]], [osegs[1]], [gsegs]], 4)
        assert _packed.attention_error(host(outs[l][b:b + 1]), rO) <= _packed.ATTN_RTOL


@pytest.mark.parametrize("name", ["long_context_32k", "long_context_128k"])
def test_long_context_sampled(name):
    """28 layers, batch 16 x 32768 or batch 2 x 131072 tokens (10 % text,
    90 % image), both candidates with calibrated policies and Eq. 2 budgets at
    retention 0.2; decode steps append to a bf16 generated-token segment."""
    wl = synth.workload(name)
    types = [CacheType(s.name, s.n, "auto") for s in wl.segments]
    cache = RequestCache(types, wl.layers, wl.batch, DEV, rho=0.2, gen_capacity=8)

    def examples():
        for e in range(2):
            yield ([synth.torch_kv(90000 + 100 * e + l, 1, 4, wl.n_ctx, DEV)[0] for l in range(0, 28, 9)],
                   [synth.torch_q(95000 + 100 * e + l, 1, 28, 32, DEV) for l in range(0, 28, 9)])
    cache.calibrate(examples())
    pols = {k: ("evict" if p == 0 else "quant") for k, p in cache.policy.items()}
    K, V, Qw = _full_size_inputs(wl, DEV, 3000)
    sc = []
    cache.prefill(K, V, Qw, scores_out=sc)
    g = torch.Generator(device=DEV)
    g.manual_seed(6)
    Qd = torch.randn((3, wl.layers, wl.batch, 28, 1, 128), generator=g, device=DEV).to(torch.bfloat16)
    Kn = torch.randn((3, wl.layers, wl.batch, 4, 128), generator=g, device=DEV).to(torch.bfloat16)
    Vn = torch.randn((3, wl.layers, wl.batch, 4, 128), generator=g, device=DEV).to(torch.bfloat16)
    for t in range(3):
        outs = cache.decode_step(Qd[t], Kn[t], Vn[t])
    begins = [0, types[0].n]
    n_checked = 0
    for l, b in [(0, 0), (27, wl.batch - 1), (9, min(5, wl.batch - 1))]:
        k, v, qw = host(K[l, b]), host(V[l, b]), host(Qw[l, b])
        ref_s = osc.observation_scores(qw[None], k[None])[0]
        np.testing.assert_allclose(host(sc[l][b]), ref_s, rtol=3e-5, atol=1e-6)
        # Eq. 1 chunk mass and Eq. 2 keep counts from the oracle's own scores
        c = l // 4
        masses = []
        for ll in range(4 * c, min(4 * c + 4, wl.layers)):
            kk = host(K[ll, b])
            s_ll = osc.observation_scores(host(Qw[ll, b])[None], kk[None])[0]
            masses.append([osc.type_mass(s_ll, begins[a], begins[a] + types[a].n, 28, 32) for a in range(2)])
        m = np.mean(masses, axis=0)
        sizes = np.array([t.n * 512.0 for t in types])
        bud = opol.allocate_budget(m, sizes, 0.2 * sizes.sum())
        for a, t in enumerate(types):
            keep, bits = opol.budget_to_policy(pols[t.name], bud[a], t.n)
            seg = cache.layers[l][a]
            assert abs(seg.n_kept()[b] - keep) <= 1
            assert seg.bits == bits
        # kept sets and attention for this slice when the keep counts agree
        keeps = [cache.layers[l][a].n_kept()[b] for a in range(2)]
        ok_keep = all(abs(keeps[a] - opol.budget_to_policy(pols[types[a].name], bud[a], types[a].n)[0]) == 0
                      for a in range(2))
        if not ok_keep:
            continue
        osegs = []
        same = True
        for a, t in enumerate(types):
            lo, hi = begins[a], begins[a] + t.n
            kind = "evict" if cache.layers[l][a].bits == 16 else "evict_quant"
            segs = [oseg.compress(k[j, lo:hi], v[j, lo:hi], ref_s[j, lo:hi], kind, keeps[a],
                                  cache.layers[l][a].bits) for j in range(4)]
            for j in range(4):
                got = cache.layers[l][a].tensor("kept_idx").view(wl.batch * 4, -1)[b * 4 + j, :keeps[a]]
                same &= _kept_sets_consistent(got.cpu().numpy(), segs[j].kept_idx, ref_s[j, lo:hi])
            osegs.append(segs)
        if not same:
            continue
        kn, vn = host(Kn[:, l, b]), host(Vn[:, l, b])
        gen = [oattn.Plain(kn[:, j], vn[:, j]) for j in range(4)]
        q = host(Qd[2, l, b])[None]
        rO, _, _ = oattn.attend(q, [[osegs[0]], [osegs[1]], [gen]], 4)
        assert _packed.attention_error(host(outs[l][b:b + 1]), rO) <= _packed.ATTN_RTOL
        n_checked += 1
    assert n_checked >= 1
