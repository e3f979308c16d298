"""Decode-time heavy-hitter statistics (uc_accumulate_scores) and streaming
re-eviction in the decode loop, against the oracle.

The per-token increments must match the oracle's probabilities within the
logit error bound of the attention call whose lse they use; the engine's
re-evicted segments must hold exactly the tokens the oracle's own replay of
the same schedule keeps.
"""
import numpy as np
import pytest
import torch

import synth
from oracle import attention as oattn
from oracle import segment as oseg
from tests import _packed
from tests.test_gpu_kernels import dev, host

pytestmark = pytest.mark.gpu

uc = pytest.importorskip("paper_2609_32831_gb300")
from paper_2609_32831_gb300 import engine  # noqa: E402

DEV = "cuda"


@pytest.mark.parametrize("T", [1, 3])
def test_accumulate_scores_parity(T):
    B, hkv, hq = 2, 4, 28
    n_ctx, n_vit, keep_vit, gen_cap, steps = 500, 300, 90, 64, 20
    k, v = synth.make_kv(71 + T, B, hkv, n_ctx + n_vit)
    s = synth.make_scores(72, (B, hkv, n_ctx + n_vit))
    kd, vd = dev(k), dev(v)
    ctx = uc.Segment("quant", 2, B, hkv, n_ctx, n_ctx, DEV)
    ctx.set_keep([n_ctx] * B)
    uc.compress_segment(kd, vd, ctx)
    vit = uc.Segment("evict", 16, B, hkv, n_vit, keep_vit, DEV)
    vit.set_keep([keep_vit] * B)
    uc.compress_segment(kd, vd, vit, begin=n_ctx, scores=torch.from_numpy(s).to(DEV))
    gen = uc.Segment("evict", 16, B, hkv, 0, gen_cap, DEV)
    gen.set_keep([0] * B)
    kn, vn = synth.make_kv(73, B, hkv, steps)
    pos0 = n_ctx + n_vit
    for t in range(steps):
        uc.append(gen, dev(kn[:, :, t]), dev(vn[:, :, t]), pos0 + t)
    q = synth.make_q(74 + T, B, hq, T)
    O, lse, _ = uc.attend(dev(q), [ctx, vit, gen])
    rng = np.random.default_rng(75)
    acc_vit0 = rng.random((B, hkv, n_vit)).astype(np.float32)
    acc_gen0 = rng.random((B, hkv, pos0 + gen_cap)).astype(np.float32)
    acc_vit = torch.from_numpy(acc_vit0).to(DEV)
    acc_gen = torch.from_numpy(acc_gen0).to(DEV)
    ws = uc.Workspace(DEV)
    uc.accumulate_scores(dev(q), vit, lse, acc_vit, ws=ws)
    uc.accumulate_scores(dev(q), gen, lse, acc_gen, ws=ws)
    assert ws.status() == 0
    r_ctx = [[oseg.compress(k[b, j, :n_ctx], v[b, j, :n_ctx], None, "quant", n_ctx, 2) for j in range(hkv)]
             for b in range(B)]
    r_vit = [[oseg.compress(k[b, j, n_ctx:], v[b, j, n_ctx:], s[b, j, n_ctx:], "evict", keep_vit, 16)
              for j in range(hkv)] for b in range(B)]
    r_gen = [[oattn.Plain(kn[b, j], vn[b, j]) for j in range(hkv)] for b in range(B)]
    _, p_vit, p_gen = oattn.token_probabilities(q, [r_ctx, r_vit, r_gen], hkv)
    bound = _packed.logit_error_bound(q, [r_ctx, r_vit, r_gen], hkv, [True, False, False])
    g = hq // hkv
    got_vit = host(acc_vit) - acc_vit0
    got_gen = host(acc_gen) - acc_gen0
    for b in range(B):
        for j in range(hkv):
            # the lse error moves every probability of a row by a factor exp(+-bound)
            rel = float(np.expm1(2 * bound[b, j * g:(j + 1) * g].max())) + 1e-5
            idx = r_vit[b][j].kept_idx
            np.testing.assert_allclose(got_vit[b, j, idx], p_vit[b, j], rtol=rel, atol=1e-7)
            mask = np.ones(n_vit, bool)
            mask[idx] = False
            assert (got_vit[b, j, mask] == 0).all()
            np.testing.assert_allclose(got_gen[b, j, pos0:pos0 + steps], p_gen[b, j], rtol=rel, atol=1e-7)
            assert (got_gen[b, j, :pos0] == 0).all() and (got_gen[b, j, pos0 + steps:] == 0).all()


def test_streaming_reeviction_matches_oracle_replay():
    L, B, hkv, hq = 2, 2, 4, 28
    n_text, n_vit, gen_cap, steps = 64, 300, 64, 35
    types = [engine.CacheType("text", n_text, "full"), engine.CacheType("vit", n_vit, "full")]
    se = [engine.StreamEvict("gen", budget=24, window=8, interval=10),
          engine.StreamEvict("vit", budget=100, window=0, interval=10)]
    rc = engine.RequestCache(types, L, B, DEV, gen_capacity=gen_cap, stream_evict=se)
    N = n_text + n_vit
    k, v, qw = [], [], []
    for l in range(L):
        a, b = synth.make_kv(80 + l, B, hkv, N)
        k.append(a)
        v.append(b)
        qw.append(synth.make_q(90 + l, B, hq, 32))
    kd = [dev(x) for x in k]
    vd = [dev(x) for x in v]
    rc.prefill(kd, vd, [dev(x) for x in qw])
    kn = [synth.make_kv(100 + l, B, hkv, steps) for l in range(L)]
    qs = [[synth.make_q(200 + 7 * t + l, B, hq, 1) for l in range(L)] for t in range(steps)]
    # oracle state per layer: segment slices and accumulators by logical index
    o_text = [[[oattn.Plain(k[l][b, j, :n_text], v[l][b, j, :n_text]) for j in range(hkv)] for b in range(B)]
              for l in range(L)]
    o_vit = [[[oseg.compress(k[l][b, j, n_text:], v[l][b, j, n_text:], None, "full", n_vit, 16)
               for j in range(hkv)] for b in range(B)] for l in range(L)]
    o_gen = [[[oseg._build("evict", 16, np.zeros(0, np.int64), np.zeros((0, 128), np.float32),
                           np.zeros((0, 128), np.float32)) for j in range(hkv)] for b in range(B)] for l in range(L)]
    acc_vit = np.zeros((L, B, hkv, n_vit))
    acc_gen = np.zeros((L, B, hkv, N + gen_cap))
    for t in range(steps):
        kl = [dev(kn[l][0][:, :, t]) for l in range(L)]
        vl = [dev(kn[l][1][:, :, t]) for l in range(L)]
        outs = rc.decode_step([dev(qs[t][l]) for l in range(L)], kl, vl)
        for l in range(L):
            for b in range(B):
                for j in range(hkv):
                    o_gen[l][b][j] = oseg.append(o_gen[l][b][j], kn[l][0][b, j, t:t + 1], kn[l][1][b, j, t:t + 1],
                                                 N + t)
            segs = [o_text[l], o_vit[l], o_gen[l]]
            rO, _, _ = oattn.attend(qs[t][l], segs, hkv)
            assert _packed.attention_error(host(outs[l]), rO) <= _packed.ATTN_RTOL
            _, pv, pg = oattn.token_probabilities(qs[t][l], segs, hkv)
            for b in range(B):
                for j in range(hkv):
                    acc_vit[l, b, j, o_vit[l][b][j].kept_idx] += pv[b, j]
                    acc_gen[l, b, j, o_gen[l][b][j].kept_idx] += pg[b, j]
        if (t + 1) % 10 == 0:
            for l in range(L):
                for b in range(B):
                    for j in range(hkv):
                        if o_gen[l][b][j].n_kept > 24:
                            o_gen[l][b][j] = oseg.recompress(o_gen[l][b][j], acc_gen[l, b, j], "evict", 24, 16, 8)
                        if o_vit[l][b][j].n_kept > 100:
                            o_vit[l][b][j] = oseg.recompress(o_vit[l][b][j], acc_vit[l, b, j], "evict", 100, 16, 0)
    assert rc.evictions >= 2 * L
    for l in range(L):
        gen, vit = rc.layers[l][-1], rc.layers[l][1]
        for seg, ref in ((gen, o_gen[l]), (vit, o_vit[l])):
            cap = seg.c.cap
            idx = seg.tensor("kept_idx").view(B * hkv, cap).cpu().numpy()
            kk = host(seg.tensor("k").view(B * hkv, cap, 128))
            for b in range(B):
                for j in range(hkv):
                    r = ref[b][j]
                    assert seg.n_kept()[b] == r.n_kept
                    np.testing.assert_array_equal(idx[b * hkv + j, :r.n_kept], r.kept_idx)
                    np.testing.assert_array_equal(kk[b * hkv + j, :r.n_kept], r.k_kept)
