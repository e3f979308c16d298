"""The Eq. 3 temporal schedule driven through the library, against the same
schedule taken with the oracle's functions.

Both sides start from the same seeded context, latents, queries and eviction
scores. At every (layer, step) the GPU attention output and segment masses
must match the oracle's; at every chunk end the GPU's per-type configuration
(kind, bits, per-sequence keep) must equal the one the oracle's Eq. 3, Eq. 2
and budget mapping give from the oracle's own masses; the re-compressed
segments must match the oracle's bit for bit.
"""
import numpy as np
import pytest
import torch

import synth
from oracle import attention as oattn
from oracle import policy as opol
from oracle import scores as oscores
from oracle import segment as oseg
from tests import _packed
from tests.test_gpu_kernels import _check_quant_block, dev, host

pytestmark = pytest.mark.gpu

uc = pytest.importorskip("paper_2609_32831_gb300")
from paper_2609_32831_gb300 import engine  # noqa: E402

DEV = "cuda"
HQ, HKV = 28, 4
KIND = {uc.KIND_FULL: "full", uc.KIND_EVICT: "evict", uc.KIND_QUANT: "quant", uc.KIND_EVICT_QUANT: "evict_quant"}


def _oracle_config(policy, n, rows_keep_bits):
    """The engine's reading for one type of one layer chunk: per-sequence
    keep counts, one kind and the lowest bits any sequence's budget allows;
    an evicting type that keeps everything stays a full view."""
    keep = [k for k, _ in rows_keep_bits]
    bits = min(b for _, b in rows_keep_bits)
    if policy == "evict" and all(k == n for k in keep):
        return ("full", 16, keep)
    if bits == 16:
        return ("evict", 16, keep)
    return ("quant" if all(k == n for k in keep) else "evict_quant", bits, keep)


@pytest.mark.parametrize("rho_init,rho_min", [(0.6, 0.15), (0.35, 0.1)])
def test_temporal_schedule_matches_oracle(rho_init, rho_min):
    L, B, T, F = 2, 2, 64, 8
    types = [engine.CacheType("text", 40, "full"), engine.CacheType("vae", 256, "quant"),
             engine.CacheType("vit", 200, "evict")]
    cfg = engine.ScheduleConfig(rho_init=rho_init, rho_min=rho_min, layer_chunk=1, step_chunk=3)
    begin = [0, 40, 296]
    n_ctx = 496
    kc, vc, kl, vl, q, sc = [], [], [], [], [], []
    for l in range(L):
        a, b = synth.make_kv(700 + l, B, HKV, n_ctx)
        kc.append(a)
        vc.append(b)
        a, b = synth.make_kv(800 + l, B, HKV, T)
        kl.append(a)
        vl.append(b)
        q.append(synth.make_q(900 + l, B, HQ, T))
        sc.append(synth.make_scores(1000 + l, (B, HKV, n_ctx), tie_frac=0.2))
    kcd = [dev(x) for x in kc]
    vcd = [dev(x) for x in vc]
    latent = []
    for l in range(L):
        kd, vd = dev(kl[l]), dev(vl[l])
        seg = uc.Segment.view(kd, vd, 0, T)
        seg._keepalive = (kd, vd)
        latent.append(seg)
    qd = [dev(x) for x in q]
    scd = torch.from_numpy(np.stack(sc)).to(DEV)
    sched = engine.TemporalSchedule(types, L, B, DEV, cfg)
    sched.start(kcd, vcd, None, F, scores=scd)

    # oracle state: slices [l][a][b][j], per (layer chunk = layer, sequence) budgets, rho, M^(0)
    oseg_ = [[[[oseg.compress(kc[l][b, j, begin[a]:begin[a] + t.n], vc[l][b, j, begin[a]:begin[a] + t.n],
                              None, "full", t.n, 16) for j in range(HKV)] for b in range(B)]
              for a, t in enumerate(types)] for l in range(L)]
    ocfg = [[("full", 16, [t.n] * B) for t in types] for _ in range(L)]
    S = np.array([512.0 * t.n for t in types])
    cand = [1, 2]
    prev = [[S[cand].copy() for _ in range(B)] for _ in range(L)]
    rho = np.full((L, B), rho_init)
    m0 = np.zeros((L, B))
    macc = np.zeros((L, B, 4))
    recompressions = 0
    for f in range(F):
        c = 0 if f == 0 else 1 + (f - 1) // 3
        steps_in = 1 if c == 0 else min(3, F - (1 + (c - 1) * 3))
        for l in range(L):
            segs = list(sched.segments(l, f)) + [latent[l]]
            for a, t in enumerate(types):
                kind, bits, keep = ocfg[l][a]
                assert KIND[segs[a].c.kind] == kind and segs[a].c.bits == bits, (f, l, a)
                assert segs[a].n_kept() == keep, (f, l, a)
            O, lse, mass = uc.attend(qd[l], segs)
            sched.observe(l, f, mass)
            ref = [oseg_[l][a] for a in range(3)] + [[[oattn.Plain(kl[l][b, j], vl[l][b, j]) for j in range(HKV)]
                                                       for b in range(B)]]
            rO, _, rmass = oattn.attend(q[l], ref, HKV)
            assert _packed.attention_error(host(O), rO) <= _packed.ATTN_RTOL
            np.testing.assert_allclose(host(mass), rmass, atol=5e-5)
            macc[l] += oscores.attention_type_mass(rmass) / steps_in
        np.testing.assert_allclose(host(sched.mass_buf), macc, rtol=1e-4, atol=1e-6)
        ended = sched.end_step(f)
        if f == F - 1 or not (f == 0 or f % 3 == 0):
            assert not ended
            continue
        assert ended
        for l in range(L):
            per_type = {a: [] for a in cand}
            for b in range(B):
                mc = float(macc[l, b, cand].sum())
                if c == 0:
                    m0[l, b] = mc
                    r = rho_init
                else:
                    r = opol.retention_schedule(rho[l, b], rho_init, rho_min, mc, m0[l, b])
                rho[l, b] = r
                budget = opol.allocate_budget(macc[l, b, cand], prev[l][b], r * S[cand].sum())
                prev[l][b] = budget
                for i, a in enumerate(cand):
                    per_type[a].append(opol.budget_to_policy(types[a].policy, budget[i], types[a].n))
            for a in cand:
                new = _oracle_config(types[a].policy, types[a].n, per_type[a])
                if new == ocfg[l][a]:
                    continue
                kind, bits, keep = new
                if kind != "full":
                    for b in range(B):
                        have = oseg_[l][a][b][0].n_kept
                        kb = have if kind == "quant" else min(keep[b], have)
                        oseg_[l][a][b] = [oseg.recompress(oseg_[l][a][b][j], sc[l][b, j, begin[a]:], kind, kb,
                                                          bits) for j in range(HKV)]
                        keep[b] = kb
                    recompressions += 1
                ocfg[l][a] = (kind, bits, keep)
        macc[:] = 0.0
    assert recompressions >= 2          # the schedule did shrink something
    np.testing.assert_allclose(sched.rho, rho, rtol=1e-5)
    for l in range(L):
        for a in cand:
            seg = sched.segs[l][a]
            if seg.c.kind == uc.KIND_FULL:
                continue
            for b in range(B):
                for j in range(HKV):
                    if seg.c.bits < 16:
                        _check_quant_block(seg, b, j, oseg_[l][a][b][j])
                    else:
                        r = oseg_[l][a][b][j]
                        idx = seg.tensor("kept_idx").view(B * HKV, -1)[b * HKV + j, :r.n_kept].cpu().numpy()
                        np.testing.assert_array_equal(idx, r.kept_idx)
                        kk = host(seg.tensor("k").view(B * HKV, seg.c.cap, 128)[b * HKV + j, :r.n_kept])
                        np.testing.assert_array_equal(kk, r.k_kept)
