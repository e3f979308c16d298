"""Library-owned segments (uc_compress_budget / uc_segment_free) on the GPU:
per-sequence budget tables (§3.3 Eq. 2 via uc_allocate_budget) become one
segment per cache type whose configuration, keep counts and stored content
match the caller-owned path, and attention over them matches the oracle
(§3.4, App. E). Storage comes from the default stream-ordered allocator or
from a caller's hooks, and every allocation is returned."""
import numpy as np
import pytest
import torch

import synth
from oracle import attention as oattn
from oracle import segment as oseg
from tests import _packed

pytestmark = pytest.mark.gpu
uc = pytest.importorskip("paper_2609_32831_gb300")
from paper_2609_32831_gb300 import _lib, api  # noqa: E402

DEV = torch.device("cuda")
NAMES = {_lib.KIND_FULL: "full", _lib.KIND_EVICT: "evict", _lib.KIND_QUANT: "quant",
         _lib.KIND_EVICT_QUANT: "evict_quant"}


def _dev(x):
    return torch.from_numpy(np.ascontiguousarray(x, np.float32)).to(torch.bfloat16).to(DEV)


class TorchHooks:
    """uc_allocator over torch's caching allocator, counting its calls."""

    def __init__(self):
        self.live, self.n_alloc, self.n_free = {}, 0, 0
        self._a = _lib.ALLOC_FN(self._alloc)
        self._f = _lib.FREE_FN(self._free)
        self.c = _lib.UcAllocator(self._a, self._f, None)

    def _alloc(self, nbytes, stream, ctx):
        p = torch.cuda.caching_allocator_alloc(int(nbytes), DEV.index or 0)
        self.live[p] = nbytes
        self.n_alloc += 1
        return p

    def _free(self, p, stream, ctx):
        torch.cuda.caching_allocator_delete(p)
        del self.live[p]
        self.n_free += 1


def _case(seed=5, B=2, hkv=4):
    n = [256, 768, 384]                      # text (protected), image, generated text
    begin = [0, 256, 1024]
    N = sum(n)
    k, v = synth.make_kv(seed, B, hkv, N)
    kd, vd = _dev(k), _dev(v)
    qwin = synth.make_q(seed + 1, B, 28, 32)
    scores = uc.score_accumulate(_dev(qwin), kd)
    torch.cuda.synchronize()
    tables = []
    for b in range(B):
        t = uc.SegmentTable(n, [False, True, True])
        t.c.policy[1], t.c.policy[2] = uc.POLICY_EVICT, uc.POLICY_QUANT
        # per-sequence Eq. 1 masses: the sequences get different budgets
        t.c.mass[0], t.c.mass[1], t.c.mass[2] = 0.2, 0.5 + 0.2 * b, 0.3 - 0.1 * b
        uc.allocate_budget(t, 0.25)
        tables.append(t)
    return k, v, kd, vd, scores, tables, n, begin


def _oracle_segments(k, v, scores_np, tables, n, begin, B, hkv):
    out = []
    for a in range(len(n)):
        kind, bits, full_view, keep = api.plan_batch(tables, a)
        name = "full" if full_view else NAMES[kind]
        per_b = []
        for b in range(B):
            row = []
            for j in range(hkv):
                ks = k[b, j, begin[a]:begin[a] + n[a]]
                vs = v[b, j, begin[a]:begin[a] + n[a]]
                if name == "full":
                    row.append(oattn.Plain(ks, vs))
                else:
                    sc = scores_np[b, j, begin[a]:begin[a] + n[a]]
                    row.append(oseg.compress(ks, vs, sc, name, keep[b], bits))
            per_b.append(row)
        out.append(per_b)
    return out


@pytest.mark.parametrize("hooks", [False, True])
def test_compress_budget_matches_plan_and_oracle(hooks):
    B, hkv = 2, 4
    k, v, kd, vd, scores, tables, n, begin = _case(B=B, hkv=hkv)
    alloc = TorchHooks() if hooks else None
    segs = [uc.compress_budget(kd, vd, tables, a, begin=begin[a], scores=scores,
                               allocator=None if alloc is None else alloc.c) for a in range(3)]
    kinds = []
    for a, seg in enumerate(segs):
        kind, bits, full_view, keep = api.plan_batch(tables, a)
        assert seg.kind == (_lib.KIND_FULL if full_view else kind)
        assert seg.bits == (16 if full_view else bits)
        assert seg.n_kept() == keep
        assert seg.tensor("n_kept").cpu().tolist() == keep
        kinds.append(NAMES[seg.kind])
    assert kinds[0] == "full" and kinds[1] == "evict" and kinds[2] in ("quant", "evict_quant")
    assert segs[1].n_kept()[0] != segs[1].n_kept()[1]      # per-sequence budgets
    scores_np = scores.cpu().numpy()
    osegs = _oracle_segments(k, v, scores_np, tables, n, begin, B, hkv)
    # kept indices of the evicted type: bit-exact with the oracle's selection
    idx = segs[1].tensor("kept_idx").view(B, hkv, segs[1].cap).cpu().numpy()
    for b in range(B):
        for j in range(hkv):
            kb = segs[1].n_kept()[b]
            np.testing.assert_array_equal(idx[b, j, :kb], osegs[1][b][j].kept_idx)
    q = synth.make_q(9, B, 28, 1)
    O, lse, mass = uc.attend(_dev(q), segs)
    rO, rl, rm = oattn.attend(q, osegs, hkv)
    assert _packed.attention_error(O.double().cpu().numpy(), rO) <= _packed.ATTN_RTOL
    bound = _packed.logit_error_bound(q, osegs, hkv, [False, False, True])
    assert (np.abs(lse.cpu().numpy() - rl) <= bound).all()
    torch.cuda.synchronize()
    for s in segs:
        s.free()
    torch.cuda.synchronize()
    if alloc is not None:
        assert alloc.n_alloc > 0 and alloc.n_alloc == alloc.n_free and not alloc.live


def test_compress_budget_releases_on_error():
    """A NaN score is the kernels' UC_ERR_RANGE: nothing is returned and the
    storage taken so far goes back to the allocator."""
    B, hkv = 2, 4
    k, v, kd, vd, scores, tables, n, begin = _case(seed=7, B=B, hkv=hkv)
    scores[0, 1, begin[1] + 5] = float("nan")
    alloc = TorchHooks()
    with pytest.raises(uc.UniCacheError) as e:
        uc.compress_budget(kd, vd, tables, 1, begin=begin[1], scores=scores, allocator=alloc.c)
    assert e.value.code == _lib.UC_ERR_RANGE
    torch.cuda.synchronize()
    assert alloc.n_alloc > 0 and alloc.n_alloc == alloc.n_free and not alloc.live
