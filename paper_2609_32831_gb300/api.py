"""Python binding of the UniCache C ABI (same names, minus the ``uc_`` prefix).

Torch supplies device memory and the current stream; every computation runs
in the CUDA library. Each function marshals its arguments and calls one C
entry point; nothing here computes any part of the method.
"""
from __future__ import annotations

import ctypes as C
from typing import List, Optional, Sequence, Tuple

import torch

from . import _lib
from ._lib import (GROUP, HEAD_DIM, KIND_EVICT, KIND_EVICT_QUANT, KIND_FULL, KIND_QUANT,
                   MAX_BATCH, MAX_SEGMENTS, POLICY_EVICT, POLICY_PROTECTED, POLICY_QUANT,
                   UcSegment, UcSegmentSizes, UcSegmentTable, UniCacheError, check, lib)

KIND_NAMES = {"full": KIND_FULL, "evict": KIND_EVICT, "quant": KIND_QUANT, "evict_quant": KIND_EVICT_QUANT}


def _stream(stream=None) -> C.c_void_p:
    s = stream if stream is not None else torch.cuda.current_stream()
    return C.c_void_p(s.cuda_stream)


def _ptr(t: Optional[torch.Tensor]) -> Optional[int]:
    return None if t is None else t.data_ptr()


class Workspace:
    """Zero-filled device scratch, grown on demand and reused across calls.

    ``uc_attend`` and ``uc_attend_batch`` keep self-resetting merge counters
    in their workspaces, so each gets a buffer of its own ("attend",
    "attend_batch"); every other entry point shares the "scratch" buffer."""

    def __init__(self, device=None):
        self.device = torch.device(device or "cuda")
        self.bufs = {}

    def get(self, nbytes: int, kind: str = "scratch") -> Tuple[int, int]:
        nbytes = max(256, int(nbytes))
        buf = self.bufs.get(kind)
        if buf is None or buf.numel() < nbytes:
            buf = torch.zeros(nbytes, dtype=torch.uint8, device=self.device)
            self.bufs[kind] = buf
        return buf.data_ptr(), buf.numel()

    def status(self, stream=None) -> int:
        """Synchronise and read (then clear) the device status words."""
        code = 0
        for buf in self.bufs.values():
            c = lib().uc_workspace_status(C.c_void_p(buf.data_ptr()), _stream(stream))
            code = code or c
        return code


_default_ws = {}


def default_workspace(device) -> Workspace:
    key = torch.device(device).index or 0
    if key not in _default_ws:
        _default_ws[key] = Workspace(device)
    return _default_ws[key]


class Segment:
    """One cache type of one layer for B sequences and Hkv KV heads, with its
    storage in torch device tensors (see ``uc_segment`` in unicache.h)."""

    def __init__(self, kind, bits: int, batch: int, n_kv_heads: int, n_src: int, cap: int,
                 device="cuda", label: int = 0):
        kind = KIND_NAMES.get(kind, kind)
        if kind == KIND_FULL:
            raise ValueError("use Segment.view() for full-precision segments")
        if kind in (KIND_QUANT, KIND_EVICT_QUANT):
            cap = (cap + 63) // 64 * 64
        else:
            bits = 16
        self.device = torch.device(device)
        c = UcSegment()
        c.kind, c.bits, c.batch, c.n_kv_heads = kind, bits, batch, n_kv_heads
        c.head_dim, c.n_src, c.cap, c.label = HEAD_DIM, n_src, cap, label
        sz = UcSegmentSizes()
        check("uc_segment_sizes_of", lib().uc_segment_sizes_of(C.byref(c), C.byref(sz)))
        self._t = {}

        def alloc(name, nbytes, dtype=torch.uint8):
            if nbytes == 0:
                return None
            el = torch.tensor([], dtype=dtype).element_size()
            t = torch.zeros(int(nbytes) // el, dtype=dtype, device=self.device)
            self._t[name] = t
            return t.data_ptr()

        c.n_kept = alloc("n_kept", sz.n_kept, torch.int32)
        c.kept_idx = alloc("kept_idx", sz.kept_idx, torch.int32)
        c.k = alloc("k", sz.k, torch.bfloat16)
        c.v = alloc("v", sz.v, torch.bfloat16)
        c.k_codes = alloc("k_codes", sz.k_codes)
        c.k_params = alloc("k_params", sz.k_params)
        c.v_codes = alloc("v_codes", sz.v_codes)
        c.v_params = alloc("v_params", sz.v_params)
        nbh = batch * n_kv_heads
        if kind in (KIND_QUANT, KIND_EVICT_QUANT):
            c.row_stride, c.row_offset, c.rows_total = GROUP, 0, nbh * GROUP
        else:
            c.row_stride, c.row_offset, c.rows_total = cap, 0, nbh * cap
        self.c = c

    @classmethod
    def view(cls, k: torch.Tensor, v: torch.Tensor, begin: int, n: int, label: int = 0) -> "Segment":
        """A full-precision segment over tokens [begin, begin + n) of caller
        tensors k, v [B, Hkv, N, 128] (bf16, contiguous). Borrowed, not copied."""
        assert k.dtype == torch.bfloat16 and k.is_contiguous() and v.is_contiguous()
        B, hkv, N, d = k.shape
        self = cls.__new__(cls)
        self.device = k.device
        c = UcSegment()
        c.kind, c.bits, c.batch, c.n_kv_heads = KIND_FULL, 16, B, hkv
        c.head_dim, c.n_src, c.cap, c.label = d, n, n, label
        for b in range(B):
            c.n_kept_host[b] = n
        nk = torch.full((B,), n, dtype=torch.int32, device=k.device)
        self._t = {"n_kept": nk, "k": k, "v": v}
        c.n_kept = nk.data_ptr()
        c.kept_idx = None
        c.k, c.v = k.data_ptr(), v.data_ptr()
        c.row_stride, c.row_offset, c.rows_total = N, begin, B * hkv * N
        self.c = c
        return self

    # -------------------------------------------------------------- views
    @property
    def kind(self) -> int:
        return self.c.kind

    @property
    def bits(self) -> int:
        return self.c.bits

    @property
    def batch(self) -> int:
        return self.c.batch

    @property
    def n_kv_heads(self) -> int:
        return self.c.n_kv_heads

    @property
    def cap(self) -> int:
        return self.c.cap

    def n_kept(self) -> List[int]:
        return [int(self.c.n_kept_host[b]) for b in range(self.c.batch)]

    def sync_host(self) -> None:
        """Copy the device kept counts into the host mirror (after appends
        that only advance the device counts, e.g. replayed graphs)."""
        counts = self._t["n_kept"].cpu().tolist()
        for b, n in enumerate(counts):
            self.c.n_kept_host[b] = int(n)

    def set_keep(self, keep: Sequence[int]) -> None:
        """Number of tokens to keep per sequence (before compress_segment)."""
        for b in range(self.c.batch):
            self.c.n_kept_host[b] = int(keep[b] if hasattr(keep, "__len__") else keep)

    def tensor(self, name: str) -> Optional[torch.Tensor]:
        return self._t.get(name)

    def stored_bytes(self, with_index: bool = False) -> int:
        """Bytes the stored tokens occupy in the packed layout (K + V)."""
        tot = 0
        for n in self.n_kept():
            per_head = 0
            if self.c.bits == 16:
                per_head = n * 4 * HEAD_DIM
            else:
                ng = n // GROUP
                per_head = (2 * GROUP * ng * HEAD_DIM * self.c.bits // 8 + ng * HEAD_DIM * 4 +
                            GROUP * ng * 16 + (n - GROUP * ng) * 4 * HEAD_DIM)
            if with_index and self.c.kind != KIND_FULL:
                per_head += 4 * n
            tot += per_head * self.c.n_kv_heads
        return tot


# ---------------------------------------------------------------- host policy

def concentration(mass, top_frac: float = 0.1) -> float:
    import numpy as np
    m = np.ascontiguousarray(mass, dtype=np.float32)
    out = C.c_double()
    check("uc_concentration", lib().uc_concentration(
        m.ctypes.data_as(C.c_void_p), m.size, top_frac, C.byref(out)))
    return out.value


class SegmentTable:
    """uc_segment_table: per-type candidates, sizes, policies and budgets."""

    def __init__(self, n_tokens: Sequence[int], candidate: Sequence[bool]):
        t = UcSegmentTable()
        t.n_types = len(n_tokens)
        for a, (n, c) in enumerate(zip(n_tokens, candidate)):
            t.n_tokens[a] = int(n)
            t.candidate[a] = 1 if c else 0
            t.policy[a] = POLICY_PROTECTED if not c else POLICY_EVICT
        self.c = t

    def field(self, name):
        arr = getattr(self.c, name)
        return [arr[a] for a in range(self.c.n_types)]


def calibrate_policy(table: SegmentTable, mass_vectors, top_frac: float = 0.1,
                     threshold: float = 0.5) -> None:
    """mass_vectors[e][a]: per-token mass (host array) of type a in example e."""
    import numpy as np
    n_ex = len(mass_vectors)
    nt = table.c.n_types
    keep_alive = []
    ptrs = (C.c_void_p * (n_ex * nt))()
    for e in range(n_ex):
        for a in range(nt):
            m = np.ascontiguousarray(mass_vectors[e][a], dtype=np.float32)
            if m.size != table.c.n_tokens[a]:
                raise ValueError(f"example {e} type {a}: {m.size} != {table.c.n_tokens[a]}")
            keep_alive.append(m)
            ptrs[e * nt + a] = m.ctypes.data_as(C.c_void_p)
    check("uc_calibrate_policy", lib().uc_calibrate_policy(
        C.byref(table.c), C.cast(ptrs, C.c_void_p), n_ex, top_frac, threshold))


def allocate_budget(table: SegmentTable, rho: float, first_chunk: bool = True) -> None:
    """Eq. 2 with B = rho * sum_a S_a; previous budgets are table.budget (or S
    on the first chunk). Fills table budget / keep / bits / kind."""
    check("uc_allocate_budget", lib().uc_allocate_budget(C.byref(table.c), float(rho), int(first_chunk)))


def retention_schedule(rho_prev, rho_init, rho_min, m_c, m_0) -> float:
    out = C.c_double()
    check("uc_retention_schedule", lib().uc_retention_schedule(
        float(rho_prev), float(rho_init), float(rho_min), float(m_c), float(m_0), C.byref(out)))
    return out.value


def retention_step(table: "SegmentTable", first_chunk: bool, rho_prev: float, rho_init: float, rho_min: float,
                   m_0: float = 0.0):
    """Eq. 3 for one (sequence, layer chunk) with M^(c) formed from the
    table's candidate masses; returns (rho, m_0) (see unicache.h)."""
    m0 = C.c_double(m_0)
    rho = C.c_double()
    check("uc_retention_step", lib().uc_retention_step(C.byref(table.c), int(first_chunk), float(rho_prev),
                                                       float(rho_init), float(rho_min), C.byref(m0),
                                                       C.byref(rho)))
    return rho.value, m0.value


def plan_batch(tables, type_index: int):
    """One segment configuration of type ``type_index`` for a batch of
    per-sequence tables (after allocate_budget): returns (kind, bits,
    full_view, keep list)."""
    from ._lib import UcTypeConfig
    n = len(tables)
    arr = (UcSegmentTable * n)(*[t.c for t in tables])
    keep = (C.c_int32 * n)()
    cfg = UcTypeConfig()
    check("uc_plan_batch", lib().uc_plan_batch(arr, n, int(type_index), keep, C.byref(cfg)))
    return int(cfg.kind), int(cfg.bits), bool(cfg.full_view), [int(x) for x in keep]


def keep_count(n: int, keep_frac: float) -> int:
    """Tokens a fixed keep fraction retains (see unicache.h)."""
    out = C.c_int32()
    check("uc_keep_count", lib().uc_keep_count(int(n), float(keep_frac), C.byref(out)))
    return int(out.value)


# ---------------------------------------------------------------- device calls

def score_accumulate(qwin: torch.Tensor, k: torch.Tensor, n_ctx: Optional[int] = None,
                     out: Optional[torch.Tensor] = None, ws: Optional[Workspace] = None,
                     stream=None) -> torch.Tensor:
    """qwin [B, Hq, W, 128], k [B, Hkv, N, 128] (bf16) -> scores [B, Hkv, n_ctx] fp32."""
    B, hq, W, d = qwin.shape
    _, hkv, N, _ = k.shape
    n_ctx = N if n_ctx is None else n_ctx
    if out is None:
        out = torch.empty((B, hkv, n_ctx), dtype=torch.float32, device=k.device)
    ws = ws or default_workspace(k.device)
    need = lib().uc_score_workspace_size(B, hq, hkv, W, n_ctx)
    wp, wn = ws.get(need)
    check("uc_score_accumulate", lib().uc_score_accumulate(
        _ptr(qwin), _ptr(k), B, hq, hkv, W, n_ctx, N, _ptr(out), wp, wn, _stream(stream)))
    return out


def segment_mass(scores: torch.Tensor, ranges: Sequence[Tuple[int, int]], n_q_heads: int,
                 window: int, out: Optional[torch.Tensor] = None, weight: float = 1.0,
                 accumulate: bool = False, stream=None) -> torch.Tensor:
    """Eq. 1 term per (sequence, type) from observation scores -> [B, n_seg]
    fp32; with accumulate=True adds weight * term into ``out``."""
    B, hkv, n_ctx = scores.shape
    ns = len(ranges)
    if out is None:
        out = torch.zeros((B, ns), dtype=torch.float32, device=scores.device)
    beg = (C.c_int32 * ns)(*[r[0] for r in ranges])
    end = (C.c_int32 * ns)(*[r[1] for r in ranges])
    check("uc_segment_mass", lib().uc_segment_mass(
        _ptr(scores), B, hkv, n_ctx, C.cast(beg, C.c_void_p), C.cast(end, C.c_void_p), ns,
        n_q_heads, window, float(weight), int(accumulate), _ptr(out), _stream(stream)))
    return out


def compress_segment(k_src: torch.Tensor, v_src: torch.Tensor, seg: Segment, begin: int = 0,
                     scores: Optional[torch.Tensor] = None, scores_begin: Optional[int] = None,
                     n_recent: int = 0, ws: Optional[Workspace] = None, stream=None) -> Segment:
    """Compress tokens [begin, begin + n_src) of k_src, v_src [B, Hkv, N, 128]
    into ``seg`` (keep counts set with ``seg.set_keep``). scores [B, Hkv, Ns]."""
    B, hkv, N, d = k_src.shape
    ws = ws or default_workspace(k_src.device)
    wp, wn = ws.get(lib().uc_compress_workspace_size(C.byref(seg.c)))
    s_stride = scores.shape[-1] if scores is not None else 0
    s_off = (begin if scores_begin is None else scores_begin) if scores is not None else 0
    check("uc_compress_segment", lib().uc_compress_segment(
        _ptr(k_src), _ptr(v_src), N, begin, _ptr(scores), s_stride, s_off, n_recent,
        C.byref(seg.c), wp, wn, _stream(stream)))
    return seg


class _CudaArray:
    """Device memory described by __cuda_array_interface__ (a view for torch)."""

    def __init__(self, iface):
        self.__cuda_array_interface__ = iface


class OwnedSegment(Segment):
    """A segment whose storage the library allocated (uc_compress_budget);
    its storage goes back to the allocator with uc_segment_free when this
    object is released (or on free())."""

    def __init__(self, ptr, device, keepalive=()):
        self._ptr = ptr
        self.c = ptr.contents
        self.device = torch.device(device)
        self._t = {}
        self._keep = keepalive   # the source rows a full view reads, the allocator's callbacks

    def sync_host(self) -> None:
        counts = self.tensor("n_kept").cpu().tolist()
        for b, n in enumerate(counts):
            self.c.n_kept_host[b] = int(n)

    def tensor(self, name: str) -> Optional[torch.Tensor]:
        """A view (no copy) of one of the segment's device arrays; valid while
        the segment lives."""
        if not self._ptr:
            return None
        sz = UcSegmentSizes()
        check("uc_segment_sizes_of", lib().uc_segment_sizes_of(C.byref(self.c), C.byref(sz)))
        dtypes = {"n_kept": ("<i4", 4), "kept_idx": ("<i4", 4), "k": ("<u2", 2), "v": ("<u2", 2),
                  "k_codes": ("|u1", 1), "k_params": ("|u1", 1), "v_codes": ("|u1", 1), "v_params": ("|u1", 1)}
        ptr = getattr(self.c, name)
        if name not in dtypes or not ptr:
            return None
        typestr, el = dtypes[name]
        nbytes = int(getattr(sz, name))
        if self.c.kind == KIND_FULL and name in ("k", "v"):
            nbytes = int(self.c.rows_total) * HEAD_DIM * 2
        iface = {"shape": (nbytes // el,), "typestr": typestr, "data": (int(ptr), False), "version": 3,
                 "strides": None}
        t = torch.as_tensor(_CudaArray(iface), device=self.device)
        return t.view(torch.bfloat16) if name in ("k", "v") else t

    def free(self) -> None:
        """Return the storage (uc_segment_free). The structure the library
        handed out goes with it, so this object keeps an empty one: a call
        that is given a freed segment fails its argument checks."""
        if self._ptr:
            self.c = UcSegment()
            lib().uc_segment_free(C.cast(self._ptr, C.c_void_p))
            self._ptr = None

    def __del__(self):
        try:
            self.free()
        except Exception:
            pass


def compress_budget(k_src: torch.Tensor, v_src: torch.Tensor, tables, type_index: int, begin: int = 0,
                    scores: Optional[torch.Tensor] = None, scores_begin: Optional[int] = None,
                    n_recent: int = 0, allocator: Optional["_lib.UcAllocator"] = None,
                    stream=None) -> OwnedSegment:
    """The budget form of compression: type ``type_index`` of k_src, v_src
    [B, Hkv, N, 128] (tokens [begin, begin + n)) compressed as the
    per-sequence tables (after allocate_budget) configure it, into storage
    the library allocates (through ``allocator``, else cudaMallocAsync)."""
    B, hkv, N, d = k_src.shape
    n = int(tables[0].c.n_tokens[type_index])
    arr = (UcSegmentTable * len(tables))(*[t.c for t in tables])
    s_stride = scores.shape[-1] if scores is not None else 0
    s_off = (begin if scores_begin is None else scores_begin) if scores is not None else 0
    out = C.POINTER(UcSegment)()
    check("uc_compress_budget", lib().uc_compress_budget(
        _ptr(k_src), _ptr(v_src), B, hkv, n, N, begin, _ptr(scores), s_stride, s_off, n_recent,
        arr, int(type_index), None if allocator is None else C.byref(allocator), _stream(stream),
        C.byref(out)))
    keep = (k_src, v_src, allocator) if out.contents.kind == KIND_FULL else (allocator,)
    return OwnedSegment(out, k_src.device, keep)


def recompress_segment(src: Segment, dst: Segment, scores: Optional[torch.Tensor] = None,
                       scores_begin: int = 0, n_recent: int = 0, ws: Optional[Workspace] = None,
                       stream=None) -> Segment:
    """Compress the tokens ``src`` still holds further into ``dst`` (keep counts
    set with ``dst.set_keep``). scores [B, Hkv, Ns] fp32 indexed by logical
    token (position scores_begin + token index), needed when dst evicts."""
    ws = ws or default_workspace(src.device)
    wp, wn = ws.get(lib().uc_recompress_workspace_size(C.byref(src.c), C.byref(dst.c)))
    s_stride = scores.shape[-1] if scores is not None else 0
    check("uc_recompress_segment", lib().uc_recompress_segment(
        C.byref(src.c), _ptr(scores), s_stride, scores_begin, n_recent, C.byref(dst.c), wp, wn,
        _stream(stream)))
    return dst


def accumulate_scores(q: torch.Tensor, seg: Segment, lse: torch.Tensor, acc: torch.Tensor, acc_begin: int = 0,
                      ws: Optional[Workspace] = None, stream=None) -> torch.Tensor:
    """Add one decode call's probabilities on the stored tokens of the bf16
    segment ``seg`` into ``acc`` [B, Hkv, N] fp32 at logical index
    acc_begin + token (lse: that call's [B, Hq, T] output)."""
    B, hq, T, d = q.shape
    ws = ws or default_workspace(q.device)
    wp, wn = ws.get(256)
    check("uc_accumulate_scores", lib().uc_accumulate_scores(
        _ptr(q), hq, T, C.byref(seg.c), _ptr(lse), _ptr(acc), acc.shape[-1], acc_begin, wp, wn,
        _stream(stream)))
    return acc


def attention_mass(mass: torch.Tensor, out: Optional[torch.Tensor] = None, weight: float = 1.0,
                   accumulate: bool = False, stream=None) -> torch.Tensor:
    """Eq. 1 term per (sequence, segment) from attend's mass [B, Hq, T, n_seg]
    -> [B, n_seg] fp32; with accumulate=True adds weight * term into ``out``."""
    B, hq, T, ns = mass.shape
    if out is None:
        out = torch.zeros((B, ns), dtype=torch.float32, device=mass.device)
    check("uc_attention_mass", lib().uc_attention_mass(
        _ptr(mass), B, hq, T, ns, float(weight), int(accumulate), _ptr(out), _stream(stream)))
    return out


def attend(q: torch.Tensor, segs: Sequence[Segment], out: Optional[torch.Tensor] = None,
           lse: Optional[torch.Tensor] = None, mass: Optional[torch.Tensor] = None,
           want_lse: bool = True, want_mass: bool = True, ws: Optional[Workspace] = None,
           stream=None):
    """q [B, Hq, T, 128] bf16 -> (O bf16 [B, Hq, T, 128], lse fp32 [B, Hq, T],
    mass fp32 [B, Hq, T, n_seg])."""
    B, hq, T, d = q.shape
    ns = len(segs)
    arr = (C.POINTER(UcSegment) * ns)(*[C.pointer(s.c) for s in segs])
    if out is None:
        out = torch.empty_like(q)
    if want_lse and lse is None:
        lse = torch.empty((B, hq, T), dtype=torch.float32, device=q.device)
    if want_mass and mass is None:
        mass = torch.empty((B, hq, T, ns), dtype=torch.float32, device=q.device)
    ws = ws or default_workspace(q.device)
    wp, wn = ws.get(lib().uc_attend_workspace_size(C.cast(arr, C.c_void_p), ns, hq, T), "attend")
    check("uc_attend", lib().uc_attend(
        _ptr(q), hq, T, C.cast(arr, C.c_void_p), ns, _ptr(out), _ptr(lse), _ptr(mass), wp, wn,
        _stream(stream)))
    return out, lse, mass


def attend_plan(segs, n_q_heads: int, n_qtok: int, slots: int = 0) -> dict:
    """How ``attend`` splits a decode-shaped call into work items, for
    ``slots`` resident CTAs (0: this device's occupancy). Host only when
    slots > 0. ``segs``: Segment objects or raw UcSegment structures."""
    from ._lib import UcAttendPlanInfo
    raw = [s.c if hasattr(s, "c") else s for s in segs]
    sp = (C.POINTER(UcSegment) * len(raw))(*[C.pointer(r) for r in raw])
    info = UcAttendPlanInfo()
    check("uc_attend_plan", lib().uc_attend_plan(C.cast(sp, C.c_void_p), len(raw), n_q_heads, n_qtok, slots,
                                                 C.byref(info)))
    n = len(raw)
    return {"items_per_bh": info.items_per_bh, "n_heavy": info.n_heavy, "n_light": info.n_light,
            "grid": info.grid, "merge_kernel": bool(info.merge_kernel),
            "n_chunks": list(info.n_chunks)[:n], "light": [bool(x) for x in list(info.light)[:n]]}


def attend_batch(calls, ws: Optional[Workspace] = None, stream=None):
    """Several decode-shaped attention calls in one launch. ``calls``: a list
    of (q, segs) or (q, segs, out, lse, mass) with q [B, Hq, T, 128] bf16
    (T <= 8; every call the same number of 8-row query tiles). Returns the
    list of (O, lse, mass) per call."""
    from ._lib import UcAttendCall
    n = len(calls)
    arr = (UcAttendCall * n)()
    keep = []
    results = []
    for i, call in enumerate(calls):
        q, segs = call[0], call[1]
        out, lse, mass = (list(call[2:5]) + [None, None, None])[:3]
        B, hq, T, d = q.shape
        ns = len(segs)
        if out is None:
            out = torch.empty_like(q)
        if lse is None:
            lse = torch.empty((B, hq, T), dtype=torch.float32, device=q.device)
        if mass is None:
            mass = torch.empty((B, hq, T, ns), dtype=torch.float32, device=q.device)
        sp = (C.POINTER(UcSegment) * ns)(*[C.pointer(s.c) for s in segs])
        keep.append(sp)
        arr[i].q, arr[i].n_q_heads, arr[i].n_qtok = _ptr(q), hq, T
        arr[i].segs, arr[i].n_seg = C.cast(sp, C.c_void_p), ns
        arr[i].out, arr[i].lse, arr[i].mass = _ptr(out), _ptr(lse), _ptr(mass)
        results.append((out, lse, mass))
    ws = ws or default_workspace(calls[0][0].device)
    wp, wn = ws.get(lib().uc_attend_batch_workspace_size(C.cast(arr, C.c_void_p), n), "attend_batch")
    check("uc_attend_batch", lib().uc_attend_batch(C.cast(arr, C.c_void_p), n, wp, wn, _stream(stream)))
    return results


def attend_workspace_size(segs: Sequence[Segment], n_q_heads: int, n_qtok: int) -> int:
    ns = len(segs)
    arr = (C.POINTER(UcSegment) * ns)(*[C.pointer(s.c) for s in segs])
    return int(lib().uc_attend_workspace_size(C.cast(arr, C.c_void_p), ns, n_q_heads, n_qtok))


def append(seg: Segment, k_new: torch.Tensor, v_new: torch.Tensor, position: int,
           ws: Optional[Workspace] = None, stream=None) -> None:
    """Append one token per sequence: k_new, v_new [B, Hkv, 128] (or [B, Hkv, 1, 128])."""
    ws = ws or default_workspace(k_new.device)
    wp, wn = ws.get(256)
    check("uc_append", lib().uc_append(
        C.byref(seg.c), _ptr(k_new), _ptr(v_new), int(position), wp, wn, _stream(stream)))



def append_next(seg: Segment, k_new: torch.Tensor, v_new: torch.Tensor, base_position: int,
                ws: Optional[Workspace] = None, stream=None) -> None:
    """Like ``append`` with the logical index base_position + n_kept[b] taken on
    the device and no host-side state: capturable in a CUDA graph."""
    ws = ws or default_workspace(k_new.device)
    wp, wn = ws.get(256)
    check("uc_append_next", lib().uc_append_next(
        C.byref(seg.c), _ptr(k_new), _ptr(v_new), int(base_position), wp, wn, _stream(stream)))


def set_dense_serial_pv(serial: bool) -> bool:
    """Issue order of the dense attention kernel (see unicache.h); returns the
    previous setting."""
    return bool(lib().uc_set_dense_serial_pv(1 if serial else 0))


def set_wait_limit(ns: int) -> int:
    """Limit of the decode kernels' bounded waits in ns (0: the default,
    2 s); returns the previous value."""
    return int(lib().uc_set_wait_limit(int(ns)))


def set_programmatic_launch(on: bool) -> bool:
    """Programmatic dependent launch of the decode kernels (see
    unicache.h for the ordering it asks of the caller); returns the previous
    setting."""
    return bool(lib().uc_set_programmatic_launch(1 if on else 0))


def debug_withhold_tile(pos: int) -> None:
    """Test hook: the next decode attention call never copies the first tile
    of its work item at processing position ``pos`` (see unicache.h)."""
    lib().uc_debug_withhold_tile(int(pos))


def launch_count() -> int:
    return int(lib().uc_launch_count())


def version() -> int:
    return int(lib().uc_version())
