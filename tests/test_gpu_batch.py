"""Several decode-shaped attention calls in one launch (uc_attend_batch).

Each call of a batch must match the oracle exactly as a separate uc_attend
call does (same tolerance), and agree with that separate call up to the
summation order of the split-K merge. The calls differ in batch size, KV
heads, segment kinds and lengths.
"""
import numpy as np
import pytest
import torch

import synth
from oracle import attention as oattn
from tests import _packed
from tests.test_gpu_kernels import MIXES, _build_mix, dev, host

pytestmark = pytest.mark.gpu

uc = pytest.importorskip("paper_2609_32831_gb300")
DEV = "cuda"


def _call(mix, seed, B, hkv, hq, T):
    sizes, kinds, keeps, bits = MIXES[mix]
    if mix == "ragged_batch":
        keeps = [k[:B] if hasattr(k, "__len__") else k for k in keeps]
    gsegs, osegs = _build_mix(seed, B, hkv, sizes, kinds, keeps, bits)
    q = synth.make_q(seed + 1, B, hq, T)
    quant = [kd in ("quant", "evict_quant") for kd in kinds]
    return q, gsegs, osegs, quant


@pytest.mark.parametrize("T,shapes", [
    (1, [("four_kinds", 2, 4, 28), ("bf16_only", 1, 4, 28), ("ragged_batch", 3, 4, 28),
         ("quant_only_tail", 2, 8, 56)]),
    (2, [("text_full+vit_evict_int4", 2, 4, 28), ("four_kinds", 1, 2, 14)]),
    (1, [("text_full+vit_evict_int4", 1, 4, 28)]),
])
def test_attend_batch_matches_oracle_and_single_calls(T, shapes):
    calls = [_call(mix, 40 + 7 * i, B, hkv, hq, T) for i, (mix, B, hkv, hq) in enumerate(shapes)]
    ws = uc.Workspace(DEV)
    for rep in range(2):                    # the counters re-arm between launches
        res = uc.attend_batch([(dev(q), g) for q, g, _, _ in calls], ws=ws)
        for (q, g, o, quant), (O, lse, mass) in zip(calls, res):
            hkv = g[0].c.n_kv_heads
            rO, rl, rm = oattn.attend(q, o, hkv)
            assert _packed.attention_error(host(O), rO) <= _packed.ATTN_RTOL
            bound = _packed.logit_error_bound(q, o, hkv, quant)
            assert (np.abs(host(lse) - rl) <= bound).all()
            assert (np.abs(host(mass) - rm) <= 2 * bound[..., None]).all()
            O1, l1, m1 = uc.attend(dev(q), g)
            np.testing.assert_allclose(host(O), host(O1), rtol=0, atol=2e-2 * float(np.abs(host(O1)).max()))
            np.testing.assert_allclose(host(lse), host(l1), rtol=1e-5, atol=1e-5)
    assert ws.status() == 0


def test_attend_batch_rejects_mixed_tiles_and_dense_calls():
    qa, ga, _, _ = _call("four_kinds", 3, 2, 4, 28, 1)       # 7 rows: one tile of 8
    qb, gb, _, _ = _call("four_kinds", 5, 2, 4, 28, 2)       # 14 rows: two tiles
    with pytest.raises(uc.UniCacheError):
        uc.attend_batch([(dev(qa), ga), (dev(qb), gb)])
    qd, gd, _, _ = _call("bf16_only", 9, 1, 4, 28, 64)
    with pytest.raises(uc.UniCacheError):
        uc.attend_batch([(dev(qd), gd)])
    with pytest.raises(uc.UniCacheError):
        uc.attend_batch([(dev(qa), ga)] * 9)


def test_attend_batch_eight_calls_max_params():
    # UC_MAX_CALLS calls: the launch's parameter block holds eight calls
    calls = [_call(mix, 90 + 5 * i, 1 + i % 3, 4, 28, 1)
             for i, mix in enumerate(["four_kinds", "bf16_only", "quant_only_tail", "text_full+vit_evict_int4"] * 2)]
    res = uc.attend_batch([(dev(q), g) for q, g, _, _ in calls])
    for (q, g, o, quant), (O, lse, mass) in zip(calls, res):
        rO, rl, rm = oattn.attend(q, o, 4)
        assert _packed.attention_error(host(O), rO) <= _packed.ATTN_RTOL
        bound = _packed.logit_error_bound(q, o, 4, quant)
        assert (np.abs(host(lse) - rl) <= bound).all()
