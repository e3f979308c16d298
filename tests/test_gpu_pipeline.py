"""End-to-end parity of the hot path through the engine (C-ABI calls only).

The oracle runs the same workload independently from the same synthetic
inputs: its own fp64 scores, Eq. 1 masses, Eq. 2 budgets, top-k, quantizer
and attention. Where floating point decides an integer, both sides take the
decision on the same input: the oracle's top-k ranks the fp32 score array
the GPU produced (itself checked against the oracle's fp64 scores), and its
Eq. 2 keep counts come from the Eq. 1 masses the engine used (themselves
checked against the oracle's masses), so kept sets and keep counts are
compared bit-exactly and no slice is skipped. At full workload sizes the
comparison runs on sampled (layer, sequence) slices.
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


def _assert_kept_identical(got_idx, ref_idx):
    """Kept indices from the same fp32 score array: bit-exact (ties go to the
    lower token index on both sides)."""
    np.testing.assert_array_equal(np.asarray(got_idx), np.asarray(ref_idx))


def _oracle_layer(k, v, qwin, types, begins, keeps, bits_of, kinds_of, b, scores=None):
    """Oracle segments of one (layer, sequence) slice; k, v [Hkv, N, 128].
    Eviction ranks ``scores`` [Hkv, N] when given (the GPU's fp32 array),
    else the oracle's own observation scores; returns those scores too."""
    s = osc.observation_scores(qwin[None], k[None])[0] if scores is None else scores
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
    ref_s = osc.observation_scores(qwin[0][None], k[0][None])[0]
    np.testing.assert_allclose(host(sc[0])[0], ref_s, rtol=2e-5, atol=1e-6)
    vit = cache.layers[0][1]
    # the oracle's segments from the GPU's fp32 scores: identical kept sets
    _, osegs = _oracle_layer(k[0], v[0], qwin[0], types, [0, 256], [256, keep], [16, 4],
                             ["full", "evict_quant"], 0, scores=host(sc[0])[0])
    for j in range(4):
        _assert_kept_identical(vit.tensor("kept_idx").view(4, -1)[j, :keep].cpu().numpy(), osegs[1][j].kept_idx)
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
    n_checked = 0
    for l, b in [(0, 0), (27, 7), (13, 3)]:
        k = host(K[l, b])
        v = host(V[l, b])
        ref_s = osc.observation_scores(host(Qw[l, b])[None], k[None])[0]
        gpu_s = host(sc[l][b])
        np.testing.assert_allclose(gpu_s, ref_s, rtol=2e-5, atol=1e-6)
        _, osegs = _oracle_layer(k, v, None, types, [0, 512, 7680], [512, keep, 512], [16, 4, 2],
                                 ["full", "evict_quant", "quant"], b, scores=gpu_s)
        for j in range(4):
            got = cache.layers[l][1].tensor("kept_idx").view(wl.batch * 4, -1)[b * 4 + j, :keep].cpu().numpy()
            _assert_kept_identical(got, osegs[1][j].kept_idx)
        kn, vn = host(Kn[:, l, b]), host(Vn[:, l, b])
        gsegs = osegs[2]
        for t in range(steps):
            gsegs = [oseg.append(gsegs[j], kn[t, j:j + 1], vn[t, j:j + 1], 8192 + t) for j in range(4)]
        q = host(Qd[steps - 1, l, b])[None]
        rO, _, _ = oattn.attend(q, [[osegs[0]], [osegs[1]], [gsegs]], 4)
        assert _packed.attention_error(host(outs[l][b:b + 1]), rO) <= _packed.ATTN_RTOL
        n_checked += 1
    assert n_checked == 3


@pytest.mark.parametrize("name", ["long_context_32k", "long_context_128k"])
def test_long_context_graph_sampled(name):
    """The benchmark's own decode path: 28 layers, batch 16 x 32768 or batch
    2 x 131072 tokens (10 % text, 90 % image), both candidates with
    calibrated policies and Eq. 2 budgets at retention 0.2, a bf16
    generated-token segment that is empty when the 28-layer decode step is
    captured as CUDA graphs (two copies replayed in turn, attention events on
    two layers, as the benchmark does) and grows by one token per replay.
    Every replayed step's output, lse and per-segment mass are compared on
    sampled (layer, sequence) slices with the oracle's attention over its
    own compressed segments plus the appended rows."""
    wl = synth.workload(name)
    steps = 6
    types = [CacheType(s.name, s.n, "auto") for s in wl.segments]
    cache = RequestCache(types, wl.layers, wl.batch, DEV, rho=0.2, gen_capacity=16)

    def examples():
        for e in range(2):
            yield ([synth.torch_kv(90000 + 100 * e + l, 1, 4, wl.n_ctx, DEV)[0] for l in range(0, 28, 9)],
                   [synth.torch_q(95000 + 100 * e + l, 1, 28, 32, DEV) for l in range(0, 28, 9)])
    cache.calibrate(examples())
    pols = {k: ("evict" if p == 0 else "quant") for k, p in cache.policy.items()}
    K, V, Qw = _full_size_inputs(wl, DEV, 3000)
    sc = []
    cache.prefill(K, V, Qw, scores_out=sc)
    masses_used = host(cache.mass_buf)           # Eq. 1 chunk masses the engine fed to Eq. 2
    cache.capture_decode(want_lse=True, want_mass=True, events=True, copies=2, event_layers=(0, wl.layers // 2))
    assert [g.n_kept() for g in cache.gen] == [[0] * wl.batch] * wl.layers
    g = torch.Generator(device=DEV)
    g.manual_seed(6)
    Qd = torch.randn((steps, wl.layers, wl.batch, 28, 1, 128), generator=g, device=DEV).to(torch.bfloat16)
    Kn = torch.randn((steps, wl.layers, wl.batch, 4, 128), generator=g, device=DEV).to(torch.bfloat16)
    Vn = torch.randn((steps, wl.layers, wl.batch, 4, 128), generator=g, device=DEV).to(torch.bfloat16)

    begins = [0, types[0].n]
    slices = [(0, 0), (27, wl.batch - 1), (9, min(5, wl.batch - 1))]
    oracle = {}
    for l, b in slices:
        k, v, qw = host(K[l, b]), host(V[l, b]), host(Qw[l, b])
        ref_s = osc.observation_scores(qw[None], k[None])[0]
        gpu_s = host(sc[l][b])
        np.testing.assert_allclose(gpu_s, ref_s, rtol=3e-5, atol=1e-6)
        # Eq. 1: the chunk masses from the oracle's own scores match the ones
        # the engine used; Eq. 2 + budget -> (keep, bits) from the engine's
        # masses gives exactly the engine's configuration
        c = l // 4
        masses = []
        for ll in range(4 * c, min(4 * c + 4, wl.layers)):
            s_ll = osc.observation_scores(host(Qw[ll, b])[None], host(K[ll, b])[None])[0]
            masses.append([osc.type_mass(s_ll, begins[a], begins[a] + types[a].n, 28, 32) for a in range(2)])
        np.testing.assert_allclose(masses_used[c, b, :2], np.mean(masses, axis=0), rtol=1e-4)
        sizes = np.array([t.n * 512.0 for t in types])
        bud = opol.allocate_budget(masses_used[c, b, :2].astype(np.float64), sizes, 0.2 * sizes.sum())
        osegs = []
        for a, t in enumerate(types):
            keep, bits = opol.budget_to_policy(pols[t.name], bud[a], t.n)
            seg = cache.layers[l][a]
            assert seg.n_kept()[b] == keep
            assert seg.bits == bits
            lo, hi = begins[a], begins[a] + t.n
            kind = "evict" if bits == 16 else "evict_quant"
            segs = [oseg.compress(k[j, lo:hi], v[j, lo:hi], gpu_s[j, lo:hi], kind, keep, bits) for j in range(4)]
            for j in range(4):
                got = seg.tensor("kept_idx").view(wl.batch * 4, -1)[b * 4 + j, :keep].cpu().numpy()
                _assert_kept_identical(got, segs[j].kept_idx)
            osegs.append(segs)
        oracle[(l, b)] = osegs

    n_checked = 0
    for t in range(steps):
        out = cache.decode_step_graph(Qd[t], Kn[t], Vn[t], copy=t % 2)
        torch.cuda.synchronize()
        for l, b in slices:
            osegs = oracle[(l, b)]
            kn, vn = host(Kn[:t + 1, l, b]), host(Vn[:t + 1, l, b])
            gen = [oattn.Plain(kn[:, j], vn[:, j]) for j in range(4)]
            q = host(Qd[t, l, b])[None]
            segs = [[osegs[0]], [osegs[1]], [gen]]
            rO, rl, rm = oattn.attend(q, segs, 4)
            assert _packed.attention_error(host(out[l, b:b + 1]), rO) <= _packed.ATTN_RTOL, (t, l, b)
            quant = [cache.layers[l][a].bits != 16 for a in range(2)] + [False]
            bound = _packed.logit_error_bound(q, segs, 4, quant)
            assert (np.abs(host(cache.g_lse[l, b:b + 1]) - rl) <= bound).all(), (t, l, b)
            assert (np.abs(host(cache.g_mass[l, b:b + 1]) - rm) <= 2 * bound[..., None]).all(), (t, l, b)
            n_checked += 1
    assert n_checked == steps * len(slices)
    cache.sync_host_counts()
    assert [gg.n_kept() for gg in cache.gen] == [[steps] * wl.batch] * wl.layers
