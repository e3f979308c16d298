"""The decode planner on the CPU (uc_attend_plan with an explicit CTA-slot
count, so no device is touched): how a decode-shaped call is split into
split-K work items (App. E), hand-worked for the long-context shapes and
checked for its invariants over seeded random segment mixes."""
import ctypes as C

import numpy as np
import pytest

from paper_2609_32831_gb300 import _lib, api

SLOTS = 3 * 152          # single-tile calls: three CTAs on each of 152 SMs


def _seg(kind, bits, kept, hkv=4):
    s = _lib.UcSegment()
    s.kind, s.bits, s.batch, s.n_kv_heads, s.head_dim = kind, bits, len(kept), hkv, 128
    s.cap = max(max(kept), 1)
    for b, n in enumerate(kept):
        s.n_kept_host[b] = n
    return s


def _tiles(kind, bits, n):
    """(heavy tiles, tail tile) of a segment holding n tokens: 64-row bf16
    tiles, or packed tiles of 8 (int2) / 4 (int4) groups of 32 plus a bf16
    tail of n mod 32 tokens."""
    if kind in (_lib.KIND_FULL, _lib.KIND_EVICT):
        return -(-n // 64), 0
    g = n // 32
    per = 8 if bits == 2 else 4
    return -(-g // per), int(n % 32 > 0)


def test_long_context_32k_hand_worked():
    # batch 16: 3276 text + 29492 image tokens, both int2, 128 generated bf16
    text = _seg(_lib.KIND_QUANT, 2, [3276] * 16)
    vit = _seg(_lib.KIND_QUANT, 2, [29492] * 16)
    gen = _seg(_lib.KIND_EVICT, 16, [128] * 16)
    p = api.attend_plan([text, vit, gen], 28, 1, SLOTS)
    # heavy tiles: text ceil(102 / 8) = 13, image ceil(921 / 8) = 116 (24 KB
    # each); generated 2 bf16 tiles (64 KB) < half of the 3.2 MB / 7 average
    # item -> light. 7 heavy items fill 64 * 7 = 448 of 456 slots (>= 90 %);
    # split so the largest item is smallest: text 1 (13 tiles), image 6
    # (20 tiles; 5 would give 24). Light: both int2 tails and the bf16 segment.
    assert _tiles(_lib.KIND_QUANT, 2, 3276) == (13, 1)
    assert _tiles(_lib.KIND_QUANT, 2, 29492) == (116, 1)
    assert p["n_heavy"] == 7 and p["n_light"] == 3 and p["items_per_bh"] == 10
    assert p["n_chunks"] == [2, 7, 1]
    assert p["light"] == [False, False, True]
    assert p["grid"] == SLOTS and not p["merge_kernel"]


def test_understanding_8k_hand_worked():
    # batch 8 x 4 KV heads = 32 (sequence, KV head) pairs: 512 text bf16 rows
    # (8 tiles of 64 rows, 32 KB each), 2150 kept image tokens int4 (67
    # groups: 17 tiles of 4 groups, 20 KB each, + a 6-token tail), 512
    # generated tokens int2 (16 groups: 2 tiles of 8 groups, 24 KB each).
    text = _seg(_lib.KIND_FULL, 16, [512] * 8)
    vit = _seg(_lib.KIND_EVICT_QUANT, 4, [2150] * 8)
    gen = _seg(_lib.KIND_QUANT, 2, [512] * 8)
    assert _tiles(_lib.KIND_FULL, 16, 512) == (8, 0)
    assert _tiles(_lib.KIND_EVICT_QUANT, 4, 2150) == (17, 1)
    assert _tiles(_lib.KIND_QUANT, 2, 512) == (2, 0)
    p = api.attend_plan([text, vit, gen], 28, 1, SLOTS)
    # 13 heavy items would fill 416 of 456 slots (>= 90 %), but with the two
    # packed tails that is 15 > 14 items, more than one merge stages whole;
    # 12 still fill 384 (84 % >= 80 %). Largest item smallest, one item at a
    # time: image 6 items (3 tiles, 60 KB), text 5 (2 tiles, 64 KB),
    # generated 1 (48 KB). The fifth text item leaves the largest text item
    # at 2 tiles, so it is dropped: text 4, image 6 + tail, generated 1 +
    # tail (empty here) = 13 items, 11 of them heavy.
    assert p["n_chunks"] == [4, 7, 2]
    assert p["n_heavy"] == 11 and p["n_light"] == 2 and p["items_per_bh"] == 13
    assert p["grid"] == 13 * 32 and not p["merge_kernel"]


def test_no_item_leaves_a_segments_largest_item_as_it_was():
    # merged inside the launch, a segment of 8 tiles takes 4 items of 2 rather
    # than 5 of 1-2, whatever count the slot fill asked for
    for tiles, kind, bits, n in [(8, _lib.KIND_FULL, 16, 512), (17, _lib.KIND_QUANT, 4, 2144)]:
        seg = _seg(kind, bits, [n] * 2, hkv=1)
        for slots in (4, 6, 10, 12, 20, 30, 40):
            p = api.attend_plan([seg], 7, 1, slots)
            heavy = p["n_chunks"][0] - (1 if kind == _lib.KIND_QUANT else 0)
            per = -(-tiles // heavy)
            assert heavy == -(-tiles // per), (tiles, slots, heavy)


def test_long_context_128k_uses_the_merge_kernel():
    # batch 2: 8 (sequence, KV head) pairs need ~56 items each to fill 456 slots
    text = _seg(_lib.KIND_QUANT, 2, [13107] * 2)
    vit = _seg(_lib.KIND_QUANT, 2, [117965] * 2)
    p = api.attend_plan([text, vit], 28, 1, SLOTS)
    assert p["n_heavy"] * 8 >= 0.9 * SLOTS and p["n_heavy"] <= 56
    assert p["items_per_bh"] == p["n_heavy"] + 2 > 32
    assert p["merge_kernel"] and p["light"] == [False, False]


def test_a_short_segment_keeps_its_own_item_when_comparable():
    # two halves of equal size: neither is light, the items split evenly
    a = _seg(_lib.KIND_QUANT, 4, [8192] * 16)
    b = _seg(_lib.KIND_QUANT, 4, [8192] * 16)
    p = api.attend_plan([a, b], 28, 1, SLOTS)
    assert p["light"] == [False, False]
    assert abs(p["n_chunks"][0] - p["n_chunks"][1]) <= 1


def test_empty_segment_is_one_light_item():
    full = _seg(_lib.KIND_EVICT, 16, [4000] * 4)
    empty = _seg(_lib.KIND_EVICT, 16, [0] * 4)
    p = api.attend_plan([full, empty], 28, 1, SLOTS)
    assert p["light"] == [False, True] and p["n_chunks"][1] == 1


@pytest.mark.parametrize("seed", range(40))
def test_plan_invariants_random_mixes(seed):
    rng = np.random.default_rng(seed)
    nseg = int(rng.integers(1, 9))
    B = int(rng.choice([1, 2, 3, 8, 16, 64]))
    hkv = int(rng.choice([1, 2, 4, 8]))
    kinds = [int(k) for k in rng.integers(0, 4, nseg)]
    segs = []
    for k in kinds:
        bits = 16 if k in (_lib.KIND_FULL, _lib.KIND_EVICT) else int(rng.choice([2, 4]))
        top = int(rng.choice([1, 40, 700, 9000, 60000]))
        segs.append(_seg(k, bits, [int(x) for x in rng.integers(0, top + 1, B)], hkv))
    T = int(rng.integers(1, 9))
    slots = int(rng.choice([152, 456]))
    p = api.attend_plan(segs, 7 * hkv, T, slots)
    nbh = B * hkv
    assert 1 <= p["items_per_bh"] <= 64
    assert p["n_heavy"] + p["n_light"] == p["items_per_bh"] == sum(p["n_chunks"])
    assert p["n_heavy"] <= 56 and p["n_light"] <= 2 * nseg
    assert all(c >= 1 for c in p["n_chunks"])
    assert p["grid"] == min(p["items_per_bh"] * nbh, slots)
    assert p["merge_kernel"] == (p["items_per_bh"] > 32)
    for s, seg in zip(range(nseg), segs):
        packed = seg.kind in (_lib.KIND_QUANT, _lib.KIND_EVICT_QUANT)
        if p["light"][s]:
            # a light segment is one item, or its packed tiles and its tail
            assert p["n_chunks"][s] <= (2 if packed else 1)
        else:
            # a heavy packed segment ends with its (light) tail item
            assert p["n_chunks"][s] >= (2 if packed else 1)
            # and, where the launch merges its own partials, takes no item
            # that leaves its largest item as large
            tiles = _tiles(seg.kind, seg.bits, max(seg.n_kept_host[b] for b in range(B)))[0]
            hc = p["n_chunks"][s] - (1 if packed else 0)
            per = -(-tiles // hc)
            if not p["merge_kernel"]:
                assert hc == -(-tiles // per)


def test_plan_rejects_bad_calls():
    h = _lib.lib()
    seg = _seg(_lib.KIND_QUANT, 2, [64])
    arr = (C.POINTER(_lib.UcSegment) * 1)(C.pointer(seg))
    info = _lib.UcAttendPlanInfo()
    n0 = h.uc_launch_count()
    assert h.uc_attend_plan(None, 1, 28, 1, SLOTS, C.byref(info)) == _lib.UC_ERR_ARG
    assert h.uc_attend_plan(C.cast(arr, C.c_void_p), 1, 28, 9, SLOTS, C.byref(info)) == _lib.UC_ERR_SHAPE
    assert h.uc_attend_plan(C.cast(arr, C.c_void_p), 1, 30, 1, SLOTS, C.byref(info)) == _lib.UC_ERR_SHAPE
    seg.bits = 3
    assert h.uc_attend_plan(C.cast(arr, C.c_void_p), 1, 28, 1, SLOTS, C.byref(info)) == _lib.UC_ERR_SHAPE
    assert h.uc_launch_count() == n0
