"""The C-ABI library on the CPU: it loads, exports every declared symbol, its
struct layouts match what a C compiler makes of the header, argument checks
reject bad calls before any launch, and the host policy (no device work)
matches the oracle."""
import ctypes as C
import os
import re
import subprocess
import tempfile

import numpy as np
import pytest

from oracle import policy as opolicy
from paper_2609_32831_gb300 import _lib, api

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "unicache.h")


def _declared():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(uc_[a-z0-9_]+)\s*\(", text)))


def test_library_exports_every_declared_symbol():
    h = _lib.lib()
    names = _declared()
    assert len(names) >= 15
    for n in names:
        assert hasattr(h, n), n
    assert api.version() == 1


def test_dense_issue_order_option_round_trips():
    h = _lib.lib()
    assert h.uc_set_dense_serial_pv(0) == 1      # serial order is the default
    assert h.uc_set_dense_serial_pv(7) == 0
    assert h.uc_set_dense_serial_pv(1) == 1
    assert h.uc_set_dense_serial_pv(1) == 1


def test_struct_layout_matches_c_compiler():
    src = r"""
#include <stdio.h>
#include <stddef.h>
#include "unicache.h"
int main(void) {
  printf("%zu %zu %zu %zu %zu %zu\n", sizeof(uc_segment), offsetof(uc_segment, n_kept),
         offsetof(uc_segment, row_stride), offsetof(uc_segment, cache), sizeof(uc_segment_table),
         offsetof(uc_segment_table, kind));
  printf("%zu\n", sizeof(uc_segment_sizes));
  printf("%zu %zu\n", sizeof(uc_allocator), offsetof(uc_allocator, ctx));
  return 0;
}
"""
    with tempfile.TemporaryDirectory() as d:
        c = os.path.join(d, "t.c")
        exe = os.path.join(d, "t")
        open(c, "w").write(src)
        subprocess.run(["gcc", "-I", os.path.dirname(HEADER), c, "-o", exe], check=True)
        out = subprocess.run([exe], capture_output=True, text=True, check=True).stdout.split()
    got = [C.sizeof(_lib.UcSegment), _lib.UcSegment.n_kept.offset, _lib.UcSegment.row_stride.offset,
           _lib.UcSegment.cache.offset, C.sizeof(_lib.UcSegmentTable), _lib.UcSegmentTable.kind.offset,
           C.sizeof(_lib.UcSegmentSizes), C.sizeof(_lib.UcAllocator), _lib.UcAllocator.ctx.offset]
    assert [int(x) for x in out] == got


def test_argument_checks_reject_without_launch():
    h = _lib.lib()
    n0 = h.uc_launch_count()
    assert h.uc_attend(None, 28, 1, None, 1, None, None, None, None, 0, None) == _lib.UC_ERR_ARG
    seg = _lib.UcSegment()
    seg.kind, seg.bits, seg.batch, seg.n_kv_heads, seg.head_dim = 9, 16, 1, 4, 128
    assert h.uc_compress_segment(None, None, 0, 0, None, 0, 0, 0, C.byref(seg), None, 0, None) \
        == _lib.UC_ERR_ARG
    seg.kind, seg.head_dim = _lib.KIND_EVICT, 64
    fake = C.c_void_p(1 << 20)
    assert h.uc_compress_segment(fake, fake, 10, 0, fake, 10, 0, 0, C.byref(seg), fake, 4096, None) \
        == _lib.UC_ERR_SHAPE
    assert b"head_dim" in h.uc_last_error() or b"shape" in h.uc_last_error()
    assert h.uc_score_accumulate(fake, fake, 1, 28, 4, 64, 100, 100, fake, fake, 1 << 20, None) \
        == _lib.UC_ERR_SHAPE          # 7 * 64 rows > 256
    assert h.uc_launch_count() == n0


def test_compress_budget_rejects_before_allocating():
    """uc_compress_budget checks its arguments and the tables before its
    allocator is called; uc_segment_free ignores NULL and segments the
    library did not hand out."""
    h = _lib.lib()
    calls = []
    alloc = _lib.ALLOC_FN(lambda n, s, ctx: calls.append(("alloc", n)) or None)
    free = _lib.FREE_FN(lambda p, s, ctx: calls.append(("free", p)))
    hooks = _lib.UcAllocator(alloc, free, None)
    half = _lib.UcAllocator(alloc, _lib.FREE_FN(), None)
    t = api.SegmentTable([256, 768], [False, True])
    t.c.budget[1] = 1e9
    api.allocate_budget(t, 0.2)                    # keep and bits for type 1
    tables = (_lib.UcSegmentTable * 2)(t.c, t.c)
    fake = C.c_void_p(1 << 20)
    out = C.POINTER(_lib.UcSegment)()
    n0 = h.uc_launch_count()
    args = lambda **kw: dict(dict(k=fake, v=fake, B=2, hkv=4, n=768, stride=1024, off=256, scores=fake, sstride=1024,
                                  soff=256, recent=0, tables=tables, type=1, alloc=C.byref(hooks)), **kw)

    def call(**kw):
        a = args(**kw)
        return h.uc_compress_budget(a["k"], a["v"], a["B"], a["hkv"], a["n"], a["stride"], a["off"], a["scores"],
                                    a["sstride"], a["soff"], a["recent"], a["tables"], a["type"], a["alloc"], None,
                                    C.byref(out))
    assert h.uc_compress_budget(fake, fake, 2, 4, 768, 1024, 256, fake, 1024, 256, 0, tables, 1, None, None,
                                None) == _lib.UC_ERR_ARG
    assert call(k=None) == _lib.UC_ERR_ARG
    assert call(tables=None) == _lib.UC_ERR_ARG
    assert call(alloc=C.byref(half)) == _lib.UC_ERR_ARG
    assert call(type=2) == _lib.UC_ERR_ARG
    assert call(n=700) == _lib.UC_ERR_SHAPE           # the tables describe 768 tokens
    assert call(B=0) == _lib.UC_ERR_SHAPE
    assert call(stride=900) == _lib.UC_ERR_SHAPE      # rows [256, 1024) do not fit
    assert not out
    assert calls == [] and h.uc_launch_count() == n0
    h.uc_segment_free(None)
    seg = _lib.UcSegment()
    h.uc_segment_free(C.cast(C.pointer(seg), C.c_void_p))
    assert b"did not hand out" in h.uc_last_error() or b"not a segment" in h.uc_last_error()
    assert calls == []


def test_freed_owned_segment_is_refused():
    """After free() an OwnedSegment no longer points at the structure the
    library released: it holds an empty one, which calls refuse."""
    seg = _lib.UcSegment()
    seg.kind, seg.bits, seg.batch, seg.n_kv_heads, seg.head_dim, seg.cap = _lib.KIND_QUANT, 2, 2, 4, 128, 64
    for b in range(2):
        seg.n_kept_host[b] = 64
    owned = api.OwnedSegment(C.pointer(seg), "cpu")
    assert api.attend_plan([owned], 28, 1, 456)["items_per_bh"] >= 1
    owned.free()                                  # not the library's: uc_segment_free leaves it
    assert owned.c.batch == 0 and owned.tensor("n_kept") is None
    with pytest.raises(RuntimeError):
        api.attend_plan([owned], 28, 1, 456)
    owned.free()                                  # twice is harmless


def test_segment_sizes_of():
    seg = _lib.UcSegment()
    seg.kind, seg.bits, seg.batch, seg.n_kv_heads, seg.head_dim, seg.cap = _lib.KIND_EVICT_QUANT, 4, 2, 4, 128, 192
    sz = _lib.UcSegmentSizes()
    _lib.check("sizes", _lib.lib().uc_segment_sizes_of(C.byref(seg), C.byref(sz)))
    assert sz.k_codes == 8 * 192 * 128 * 4 // 8
    assert sz.k_params == 8 * (192 // 32) * 512
    assert sz.v_params == 8 * 192 * 16
    assert sz.k == 8 * 32 * 128 * 2
    seg.cap = 100
    assert _lib.lib().uc_segment_sizes_of(C.byref(seg), C.byref(sz)) == _lib.UC_ERR_SHAPE


# ------------------------------------------------------------- host policy

def test_concentration_matches_oracle():
    rng = np.random.default_rng(0)
    for n in (1, 7, 10, 768, 5000):
        m = rng.exponential(size=n).astype(np.float32) ** 3
        assert api.concentration(m) == pytest.approx(opolicy.concentration(m), rel=1e-12)


def test_allocate_budget_matches_oracle():
    rng = np.random.default_rng(1)
    for trial in range(200):
        n = int(rng.integers(1, 7))
        ntok = rng.integers(1, 5000, size=n)
        cand = rng.random(n) > 0.2
        t = api.SegmentTable(ntok, cand)
        mass = rng.random(n) * (rng.random(n) > 0.15)
        first = trial % 3 == 0
        prev = ntok * 512.0 * (1.0 if first else rng.uniform(0.2, 1.0, size=n))
        pol = rng.integers(0, 2, size=n)
        for a in range(n):
            t.c.mass[a] = mass[a]
            t.c.budget[a] = -1.0 if first else prev[a]
            if cand[a]:
                t.c.policy[a] = int(pol[a])
        rho = float(rng.uniform(0.05, 1.0))
        total = rho * float((ntok * 512.0)[cand].sum())
        api.allocate_budget(t, rho, first_chunk=first)
        mc = np.where(cand, mass, 0.0)
        ref = opolicy.allocate_budget(mc, np.where(cand, prev, 0.0), total)
        for a in range(n):
            if not cand[a]:
                assert t.c.kind[a] == _lib.KIND_FULL and t.c.keep[a] == ntok[a]
                continue
            assert t.c.budget[a] == pytest.approx(ref[a], rel=1e-9, abs=1e-6)
            keep, bits = opolicy.budget_to_policy("evict" if pol[a] == 0 else "quant", t.c.budget[a],
                                                  int(ntok[a]))
            assert (t.c.keep[a], t.c.bits[a]) == (keep, bits)


def test_calibrate_policy_matches_oracle():
    rng = np.random.default_rng(2)
    ntok = [50, 300, 40]
    t = api.SegmentTable(ntok, [True, True, False])
    examples = []
    for e in range(10):
        examples.append([rng.exponential(size=ntok[0]) ** 6,       # concentrated
                         rng.uniform(0.9, 1.1, size=ntok[1]),      # flat
                         rng.random(ntok[2])])
    api.calibrate_policy(t, examples)
    for a in range(2):
        ref = [opolicy.concentration(np.float32(ex[a])) for ex in examples]
        assert t.c.concentration[a] == pytest.approx(np.mean(ref), rel=1e-9)
    assert t.field("policy") == [_lib.POLICY_EVICT, _lib.POLICY_QUANT, _lib.POLICY_PROTECTED]


def test_retention_schedule_matches_oracle():
    for args in [(0.4, 0.4, 0.1, 1.5, 2.0), (0.3, 0.4, 0.1, 0.4, 2.0), (1.0, 1.0, 0.25, 0.6, 1.0)]:
        assert api.retention_schedule(*args) == opolicy.retention_schedule(*args)
    with pytest.raises(api.UniCacheError):
        api.retention_schedule(0.5, 0.4, 0.5, 1.0, 1.0)


# --------------------------------------------- batch configuration (§3.4)

KIND_OF = {"full": _lib.KIND_FULL, "evict": _lib.KIND_EVICT, "quant": _lib.KIND_QUANT,
           "evict_quant": _lib.KIND_EVICT_QUANT}


def test_plan_batch_matches_oracle():
    """Per-sequence Eq. 2 budgets -> §3.4 configurations (oracle:
    allocate_budget + budget_to_policy per sequence) -> one segment
    configuration per type for the batch (oracle plan_batch), against
    uc_allocate_budget + uc_plan_batch over random tables."""
    rng = np.random.default_rng(11)
    for trial in range(300):
        n = int(rng.integers(1, 6))
        B = int(rng.integers(1, 7))
        ntok = rng.integers(1, 4000, size=n)
        cand = rng.random(n) > 0.25
        pol = rng.integers(0, 2, size=n)
        rho = float(rng.uniform(0.05, 1.0))
        sizes = ntok * 512.0
        total = rho * float(sizes[cand].sum())
        tables, ref = [], []
        for b in range(B):
            t = api.SegmentTable(ntok, cand)
            mass = rng.random(n) * (rng.random(n) > 0.1)
            for a in range(n):
                t.c.mass[a] = mass[a]
                if cand[a]:
                    t.c.policy[a] = int(pol[a])
            api.allocate_budget(t, rho, first_chunk=True)
            tables.append(t)
            bud = opolicy.allocate_budget(np.where(cand, mass, 0.0), np.where(cand, sizes, 0.0), total)
            ref.append(bud)
        for a in range(n):
            if not cand[a]:
                kind, bits, view, keep = api.plan_batch(tables, a)
                assert view and kind == _lib.KIND_FULL and keep == [int(ntok[a])] * B
                continue
            p = "evict" if pol[a] == 0 else "quant"
            configs = []
            for b in range(B):
                keep, bits = opolicy.budget_to_policy(p, tables[b].c.budget[a], int(ntok[a]))
                assert tables[b].c.budget[a] == pytest.approx(ref[b][a], rel=1e-9, abs=1e-6)
                configs.append((opolicy.config_kind(p, keep, bits, int(ntok[a])), keep, bits))
            rk, rb, rv, rkeep = opolicy.plan_batch(configs, int(ntok[a]))
            kind, bits, view, keep = api.plan_batch(tables, a)
            assert (kind, bits, view, keep) == (KIND_OF[rk], rb, rv, rkeep), (trial, a)


def test_plan_batch_rejects_inconsistent_tables():
    t1 = api.SegmentTable([100, 50], [True, True])
    t2 = api.SegmentTable([100, 60], [True, True])
    for t in (t1, t2):
        t.c.policy[0] = t.c.policy[1] = _lib.POLICY_QUANT
        t.c.mass[0] = t.c.mass[1] = 1.0
        api.allocate_budget(t, 0.3)
    with pytest.raises(api.UniCacheError):
        api.plan_batch([t1, t2], 1)
    with pytest.raises(api.UniCacheError):
        api.plan_batch([t1], 2)


def test_keep_count_matches_oracle():
    for n in (0, 1, 2, 7, 768, 7168, 29492):
        for f in (0.01, 0.1, 0.2, 0.3, 1 / 3, 0.5, 0.999, 1.0):
            assert api.keep_count(n, f) == opolicy.keep_count(n, f), (n, f)
    assert api.keep_count(768, 0.2) == 153 and api.keep_count(7168, 0.3) == 2150
    with pytest.raises(api.UniCacheError):
        api.keep_count(10, 0.0)


def test_retention_step_matches_oracle():
    """M^(c) = sum of candidate masses, then Eq. 3 (chunk 0: M^(0), rho_init)."""
    rng = np.random.default_rng(12)
    for trial in range(100):
        n = int(rng.integers(1, 6))
        cand = rng.random(n) > 0.3
        t = api.SegmentTable(rng.integers(1, 100, size=n), cand)
        m0_mass = rng.random(n)
        for a in range(n):
            t.c.mass[a] = m0_mass[a]
        rho_init = float(rng.uniform(0.3, 1.0))
        rho_min = float(rng.uniform(0.05, rho_init))
        rho, m0 = api.retention_step(t, True, 1.0, rho_init, rho_min)
        assert rho == rho_init and m0 == pytest.approx(opolicy.chunk_mass(m0_mass, cand), rel=1e-15)
        mc_mass = rng.random(n) * rng.uniform(0.2, 2.0)
        for a in range(n):
            t.c.mass[a] = mc_mass[a]
        rho_prev = float(rng.uniform(rho_min, rho_init))
        rho2, m0b = api.retention_step(t, False, rho_prev, rho_init, rho_min, m0)
        mc = opolicy.chunk_mass(mc_mass, cand)
        ref = opolicy.retention_schedule(rho_prev, rho_init, rho_min, mc, m0) if m0 > 0 else rho_prev
        assert m0b == m0 and rho2 == pytest.approx(ref, rel=1e-14)


def test_wait_limit_setting_round_trips():
    """Host-side setting of the decode kernels' bounded-wait limit."""
    prev = api.set_wait_limit(123_456_789)
    try:
        assert api.set_wait_limit(0) == 123_456_789      # 0 restores the default
        assert api.set_wait_limit(prev) == 2_000_000_000
    finally:
        api.set_wait_limit(prev)
