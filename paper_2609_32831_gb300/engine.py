"""Orchestration of the hot path for one batch of requests.

``RequestCache`` holds, per layer, the list of segments (cache types in
context order, §3.1) and drives the C-ABI calls:

* ``calibrate``: offline policy choice per candidate type (§3.2, App. B) from
  observation scores of calibration examples;
* ``prefill``: per layer, observation-window scores (uc_score_accumulate),
  the Eq. 1 chunk mass on the device (uc_segment_mass), one read of the
  masses, Eq. 2 budgets per (sequence, layer chunk) (uc_allocate_budget) and
  the per-segment compression (uc_compress_segment) — §3.3, §3.4;
* ``decode_step``: per layer, append the new token (uc_append) and attend
  over all segments with one shared softmax (uc_attend) — App. E; with
  ``stream_evict``, each step's probabilities on tracked bf16 types are
  accumulated (uc_accumulate_scores) and the types are periodically
  re-evicted to their budget, heavy hitters plus a recent window
  (uc_recompress_segment);
* ``TemporalSchedule``: for generation and editing, Eq. 1 statistics from the
  attention calls' own mass output per chunk of layers and steps, Eq. 3's
  retention ratio, Eq. 2's type budgets, and the progressive re-compression
  of every type whose configuration shrank (uc_recompress_segment);
* ``capture_decode`` / ``decode_step_graph``: the same step with the layout
  frozen (App. E "Cached metadata and execution plans"): the 28-layer step is
  captured once as a CUDA graph (uc_append_next takes the token's position
  from the device count) and replayed for every later decode step until the
  next prefill changes the layout.

Nothing here computes part of the method; it only sequences library calls
and moves their small host-side results (masses, budgets) around.
"""
from __future__ import annotations

import dataclasses
from typing import Dict, List, Optional, Sequence

import numpy as np
import torch

from . import api
from ._lib import KIND_EVICT, KIND_EVICT_QUANT, KIND_FULL, KIND_QUANT, POLICY_EVICT, POLICY_QUANT

POLICY_NAMES = {"evict": POLICY_EVICT, "quant": POLICY_QUANT}


@dataclasses.dataclass
class CacheType:
    """One cache type of the context (§3.1).

    policy: 'full' (kept in bf16; protected objects), 'auto' (policy from
    calibration, budget from Eq. 2), or a fixed configuration 'evict',
    'quant', 'evict_quant' with ``keep_frac`` / ``bits``.
    """
    name: str
    n: int
    policy: str = "auto"
    keep_frac: float = 1.0
    bits: int = 16
    headroom: int = 0      # capacity for decode tokens appended to this type

    @property
    def candidate(self) -> bool:
        return self.policy != "full"


@dataclasses.dataclass
class StreamEvict:
    """Decode-time heavy-hitter + recent-window eviction of one bf16 type
    (App. E's heavy-hitter and recent-token selection, applied as decode
    proceeds): every decode step adds the step's attention probabilities to
    the type's per-token scores; every ``interval`` steps a layer whose type
    holds more than ``budget`` tokens is re-evicted to ``budget``: the
    ``window`` most recent stored tokens plus the highest-scoring others.
    ``name`` is a cache type or "gen" (the generated-token segment)."""
    name: str
    budget: int
    window: int = 32
    interval: int = 16


def fixed_keep(n: int, frac: float) -> int:
    """Tokens a fixed keep fraction retains (workload configuration; uc_keep_count)."""
    return api.keep_count(n, frac)


class RequestCache:
    def __init__(self, types: Sequence[CacheType], n_layers: int, batch: int, device,
                 n_q_heads: int = 28, n_kv_heads: int = 4, window: int = 32, rho: float = 0.2,
                 layer_chunk: int = 4, gen_capacity: int = 0, append_to: Optional[str] = None,
                 stream_evict: Sequence[StreamEvict] = ()):
        self.types = list(types)
        self.L, self.B = n_layers, batch
        self.device = torch.device(device)
        self.hq, self.hkv, self.W = n_q_heads, n_kv_heads, window
        self.rho, self.layer_chunk = rho, layer_chunk
        self.gen_capacity = gen_capacity
        self.append_to = append_to
        self.n_ctx = sum(t.n for t in self.types)
        self.begin = np.cumsum([0] + [t.n for t in self.types])[:-1].tolist()
        self.policy: Dict[str, int] = {}
        self.concentration: Dict[str, float] = {}
        self.layers: List[List[api.Segment]] = [[] for _ in range(n_layers)]
        self.gen: List[Optional[api.Segment]] = [None] * n_layers
        self.plans: List[Optional[api.SegmentTable]] = []
        self._pool: Dict[tuple, api.Segment] = {}
        self.ws = api.Workspace(self.device)
        self.score_buf: Optional[torch.Tensor] = None
        self.mass_buf: Optional[torch.Tensor] = None
        self.n_pos = self.n_ctx
        self._views: Dict[tuple, List[api.Segment]] = {}
        self.graph = None
        self.graphs: List = []
        self._graph_sig = None
        # captured decode steps by layout signature (a prefill into another
        # set of input buffers changes the views' addresses; each layout is
        # captured once and replayed when it comes back)
        self._captures: Dict[tuple, dict] = {}
        self.stream_evict = list(stream_evict)
        self.acc: Dict[tuple, torch.Tensor] = {}
        self._lse: Optional[torch.Tensor] = None
        self._steps = 0
        self.evictions = 0

    # ------------------------------------------------------------ calibration
    def calibrate(self, examples, top_frac: float = 0.1, threshold: float = 0.5) -> None:
        """``examples`` yields (k, qwin) with k [L, 1, Hkv, N, 128] or an
        iterable over layers of [1, Hkv, N, 128], qwin likewise. Concentration
        is averaged over examples, layers and KV heads (each head's mass vector
        is where eviction acts)."""
        auto = [i for i, t in enumerate(self.types) if t.policy == "auto"]
        if not auto:
            return
        vectors = []
        for k_layers, q_layers in examples:
            for k, qw in zip(k_layers, q_layers):
                s = api.score_accumulate(qw, k, ws=self.ws).cpu().numpy()
                for b in range(s.shape[0]):
                    for j in range(s.shape[1]):
                        vectors.append([s[b, j, self.begin[a]:self.begin[a] + self.types[a].n]
                                        for a in range(len(self.types))])
        table = api.SegmentTable([t.n for t in self.types], [t.candidate for t in self.types])
        api.calibrate_policy(table, vectors, top_frac, threshold)
        for a in auto:
            self.policy[self.types[a].name] = table.c.policy[a]
            self.concentration[self.types[a].name] = table.c.concentration[a]

    # ----------------------------------------------------------------- prefill
    def _view(self, key: tuple, k: torch.Tensor, v: torch.Tensor, begin: int, n: int) -> api.Segment:
        """A full-precision view, reused whenever it describes the same
        tensors (so a layout keeps its signature, and the device count a
        captured decode graph reads stays alive); the views of the last few
        input buffers are kept per key."""
        views = self._views.setdefault(key, [])
        for i, seg in enumerate(views):
            if seg.c.k == k.data_ptr() and seg.c.v == v.data_ptr() and seg.c.row_offset == begin \
                    and seg.c.n_src == n and seg.c.row_stride == k.shape[2]:
                views.insert(0, views.pop(i))
                return seg
        seg = api.Segment.view(k, v, begin, n)
        views.insert(0, seg)
        del views[self.MAX_CAPTURES:]
        return seg

    def _segment(self, key: tuple, kind: int, bits: int, n_src: int, cap: int) -> api.Segment:
        seg = self._pool.get(key)
        if seg is None or seg.kind != kind or seg.bits != (bits if kind in (KIND_QUANT, KIND_EVICT_QUANT) else 16) \
                or seg.cap < cap:
            seg = api.Segment(kind, bits, self.B, self.hkv, n_src, cap, self.device)
            self._pool[key] = seg
        return seg

    def _budgets(self, scores_fn) -> List[api.SegmentTable]:
        """Eq. 1 chunk masses on the device, then Eq. 2 per (sequence, chunk)."""
        n_chunks = (self.L + self.layer_chunk - 1) // self.layer_chunk
        ns = len(self.types)
        if self.mass_buf is None or self.mass_buf.shape != (n_chunks, self.B, ns):
            self.mass_buf = torch.zeros((n_chunks, self.B, ns), dtype=torch.float32, device=self.device)
        ranges = [(self.begin[a], self.begin[a] + t.n) for a, t in enumerate(self.types)]
        for l in range(self.L):
            c = l // self.layer_chunk
            size = min(self.layer_chunk, self.L - c * self.layer_chunk)
            api.segment_mass(scores_fn(l), ranges, self.hq, self.W, out=self.mass_buf[c],
                             weight=1.0 / size, accumulate=(l % self.layer_chunk) != 0)
        masses = self.mass_buf.cpu().numpy()
        tables = []
        for c in range(n_chunks):
            for b in range(self.B):
                t = api.SegmentTable([ty.n for ty in self.types], [ty.candidate for ty in self.types])
                for a, ty in enumerate(self.types):
                    t.c.mass[a] = float(masses[c, b, a])
                    if ty.policy == "auto":
                        t.c.policy[a] = self.policy[ty.name]
                api.allocate_budget(t, self.rho, first_chunk=True)
                tables.append(t)
        return tables

    def prefill(self, k, v, qwin, scores_out: Optional[List[torch.Tensor]] = None) -> None:
        """k, v: per layer [B, Hkv, N, 128] bf16 (a tensor [L, ...] or a list);
        qwin: per layer [B, Hq, W, 128]."""
        auto = any(t.policy == "auto" for t in self.types)
        evict_any = any(t.policy in ("auto", "evict", "evict_quant") for t in self.types)
        scores: List[Optional[torch.Tensor]] = [None] * self.L
        if evict_any:
            if self.score_buf is None or self.score_buf.shape != (self.L, self.B, self.hkv, self.n_ctx):
                self.score_buf = torch.empty((self.L, self.B, self.hkv, self.n_ctx), dtype=torch.float32,
                                             device=self.device)
            for l in range(self.L):
                scores[l] = api.score_accumulate(qwin[l], k[l], out=self.score_buf[l], ws=self.ws)
            if scores_out is not None:
                scores_out[:] = scores
        tables = self._budgets(lambda l: scores[l]) if auto else None
        for l in range(self.L):
            segs = []
            for a, ty in enumerate(self.types):
                if ty.policy == "full":
                    segs.append(self._view((l, a), k[l], v[l], self.begin[a], ty.n))
                    continue
                if ty.policy == "auto":
                    c = l // self.layer_chunk
                    kind, bits, full_view, keep = api.plan_batch(tables[c * self.B:(c + 1) * self.B], a)
                    if full_view:
                        segs.append(self._view((l, a), k[l], v[l], self.begin[a], ty.n))
                        continue
                else:
                    kind = api.KIND_NAMES[ty.policy]
                    bits = ty.bits if kind in (KIND_QUANT, KIND_EVICT_QUANT) else 16
                    keep = [ty.n if kind == KIND_QUANT else fixed_keep(ty.n, ty.keep_frac)] * self.B
                seg = self._segment((l, a), kind, bits, ty.n, max(keep) + ty.headroom)
                seg.set_keep(keep)
                api.compress_segment(k[l], v[l], seg, begin=self.begin[a], scores=scores[l], ws=self.ws)
                segs.append(seg)
            if self.gen_capacity:
                g = self._segment((l, "gen"), KIND_EVICT, 16, 0, self.gen_capacity)
                g.set_keep([0] * self.B)
                g.tensor("n_kept").zero_()
                self.gen[l] = g
                segs.append(g)
            elif self.append_to is not None:
                names = [t.name for t in self.types]
                self.gen[l] = segs[names.index(self.append_to)]
            self.layers[l] = segs
        self.plans = tables or []
        self.n_pos = self.n_ctx
        self._init_stream_scores(scores)
        if self.graph is not None:
            sig = self._layout_signature()
            if sig != self._graph_sig:
                # the layout changed: a capture of the new layout is reused,
                # else the next graphed step recaptures
                self.graph = None
                cap = self._captures.get(sig)
                if cap is not None:
                    self._restore_capture(sig, cap)

    # ------------------------------------------------- streaming re-eviction
    def _tracked(self, l: int):
        """(StreamEvict, type index or -1 for gen, segment) of layer l."""
        names = [t.name for t in self.types]
        for se in self.stream_evict:
            if se.name == "gen":
                if self.gen_capacity and self.gen[l] is not None:
                    yield se, -1, self.gen[l]
            else:
                a = names.index(se.name)
                seg = self.layers[l][a]
                if seg.c.kind in (KIND_EVICT, KIND_FULL):
                    yield se, a, seg

    def _init_stream_scores(self, scores) -> None:
        """Per (layer, tracked type) score accumulator by logical index: a
        context type starts from its prefill observation scores, the
        generated-token segment from zero (indices are absolute positions)."""
        self.acc = {}
        self._steps = 0
        self.evictions = 0
        self._parity: Dict[tuple, int] = {}
        for l in range(self.L):
            for se, a, seg in self._tracked(l):
                if a < 0:
                    n = self.n_ctx + max(self.gen_capacity, 1)
                    acc = torch.zeros((self.B, self.hkv, n), dtype=torch.float32, device=self.device)
                else:
                    n = self.types[a].n
                    acc = torch.zeros((self.B, self.hkv, n), dtype=torch.float32, device=self.device)
                    if scores[l] is not None:
                        acc.copy_(scores[l][:, :, self.begin[a]:self.begin[a] + n])
                self.acc[(l, se.name)] = acc

    def _stream_step(self, l: int, q, lse) -> None:
        for se, a, seg in self._tracked(l):
            api.accumulate_scores(q, seg, lse, self.acc[(l, se.name)], ws=self.ws)

    def _stream_evict(self) -> None:
        """Re-evict every tracked (layer, type) above its budget."""
        for l in range(self.L):
            for se, a, seg in list(self._tracked(l)):
                if self._steps % se.interval or max(seg.n_kept()) <= se.budget:
                    continue
                keep = [min(se.budget, n) for n in seg.n_kept()]
                cap = self.gen_capacity if a < 0 else max(keep)
                n_src = seg.c.n_src
                parity = self._parity.get((l, se.name), 0) ^ 1   # never the buffer it reads
                self._parity[(l, se.name)] = parity
                dst = self._segment(("stream", l, se.name, parity), KIND_EVICT, 16, n_src, cap)
                dst.set_keep(keep)
                api.recompress_segment(seg, dst, scores=self.acc[(l, se.name)], n_recent=se.window, ws=self.ws)
                if a < 0:
                    self.gen[l] = dst
                    self.layers[l][-1] = dst
                else:
                    self.layers[l][a] = dst
                self.evictions += 1

    def _layout_signature(self):
        return tuple((s.c.kind, s.c.bits, s.c.k, s.c.k_codes, s.c.n_kept, s.c.cap, tuple(s.n_kept()))
                     for segs in self.layers for s in segs)

    # ------------------------------------------------------------------ decode
    def decode_step(self, q, k_new=None, v_new=None, out=None, lse=None, mass=None, events=None):
        """q: per layer [B, Hq, T, 128]; k_new / v_new: per layer [B, Hkv, 128]
        appended first (to the generated-token segment or the ``append_to`` type).
        ``events``: optional list of (start, end) CUDA event pairs, one per
        layer, recorded around each attention launch."""
        outs = []
        track = bool(self.stream_evict)
        if track and lse is None:
            B, hq, T = q[0].shape[:3]
            if self._lse is None or self._lse.shape != (B, hq, T):
                self._lse = torch.empty((B, hq, T), dtype=torch.float32, device=self.device)
        for l in range(self.L):
            if k_new is not None:
                api.append(self.gen[l], k_new[l], v_new[l], self.n_pos, ws=self.ws)
            if events is not None:
                events[l][0].record()
            lse_l = lse[l] if lse is not None else (self._lse if track else None)
            o = api.attend(q[l], self.layers[l], out=None if out is None else out[l],
                           lse=lse_l, mass=None if mass is None else mass[l],
                           want_lse=lse_l is not None, want_mass=mass is not None, ws=self.ws)
            if events is not None:
                events[l][1].record()
            if track:
                self._stream_step(l, q[l], o[1])
            outs.append(o[0])
        if k_new is not None:
            self.n_pos += 1
        if track:
            self._steps += 1
            self._stream_evict()
        return outs

    def capture_decode(self, n_qtok: int = 1, want_lse: bool = False, want_mass: bool = False,
                       events: bool = False, copies: int = 1, event_layers: Optional[Sequence[int]] = None,
                       programmatic: bool = True) -> None:
        """Capture one decode step of every layer (append + attend) as a CUDA
        graph over static buffers, right after a prefill (App. E cached
        execution plans). ``events``: also capture a (start, end) pair of
        external CUDA events around each attention launch (``event_layers``:
        only around those layers' launches, fewer graph nodes). ``copies``: graphs
        of the same step with their own events, replayed in turn, so that one
        copy's timings can be read while the next step runs. ``programmatic``:
        the kernels launch with programmatic dependent launch, so the append
        and attention of layer l + 1 start while layer l's attention is
        finishing (each layer's attention has a workspace of its own)."""
        if not self.gen_capacity:
            raise ValueError("graphed decode needs the generated-token segment (gen_capacity > 0)")
        if self.stream_evict:
            raise ValueError("streaming re-eviction changes the layout between steps: no graphed decode")
        L, B, dev = self.L, self.B, self.device
        bf = torch.bfloat16
        self.g_q = torch.zeros((L, B, self.hq, n_qtok, 128), dtype=bf, device=dev)
        self.g_k = torch.zeros((L, B, self.hkv, 128), dtype=bf, device=dev)
        self.g_v = torch.zeros_like(self.g_k)
        self.g_out = torch.empty_like(self.g_q)
        self.g_lse = torch.empty((L, B, self.hq, n_qtok), dtype=torch.float32, device=dev) if want_lse else None
        ns = len(self.layers[0])
        self.g_mass = (torch.empty((L, B, self.hq, n_qtok, ns), dtype=torch.float32, device=dev)
                       if want_mass else None)
        # workspaces before capture (nothing may allocate inside it): one per
        # layer's attention, so that consecutive layers' launches may overlap
        self.g_ws = [api.Workspace(dev) for _ in range(L)]
        for l in range(L):
            self.g_ws[l].get(api.attend_workspace_size(self.layers[l], self.hq, n_qtok), "attend")
        self.ws.get(256)
        timed = list(range(L)) if event_layers is None else sorted(set(event_layers))
        self.g_events = [({l: (torch.cuda.Event(enable_timing=True, external=True),
                               torch.cuda.Event(enable_timing=True, external=True)) for l in timed}
                          if events else None) for _ in range(copies)]
        torch.cuda.synchronize(dev)
        self.graphs = []
        n0 = api.launch_count()
        prev = api.set_programmatic_launch(programmatic and L >= 2)
        try:
            for c in range(copies):
                g = torch.cuda.CUDAGraph()
                ev = self.g_events[c]
                with torch.cuda.graph(g):
                    for l in range(L):
                        api.append_next(self.gen[l], self.g_k[l], self.g_v[l], self.n_ctx, ws=self.ws)
                        if ev is not None and l in ev:
                            ev[l][0].record()
                        api.attend(self.g_q[l], self.layers[l], out=self.g_out[l],
                                   lse=None if self.g_lse is None else self.g_lse[l],
                                   mass=None if self.g_mass is None else self.g_mass[l],
                                   want_lse=want_lse, want_mass=want_mass, ws=self.g_ws[l])
                        if ev is not None and l in ev:
                            ev[l][1].record()
                self.graphs.append(g)
        finally:
            api.set_programmatic_launch(prev)
        self.graph = self.graphs[0]
        self.graph_kernels = (api.launch_count() - n0) // copies  # library kernels per replayed step
        self._graph_sig = self._layout_signature()
        if len(self._captures) >= self.MAX_CAPTURES:
            self._captures.pop(next(iter(self._captures)))
        self._captures[self._graph_sig] = {name: getattr(self, name) for name in self._CAPTURE_STATE}
        # the segments the graph reads (views and their device counts) live as long as the capture
        self._captures[self._graph_sig]["_capture_layers"] = [list(segs) for segs in self.layers]

    # a capture's own state (graphs, their events, static buffers, workspaces)
    _CAPTURE_STATE = ("graphs", "g_events", "g_q", "g_k", "g_v", "g_out", "g_lse", "g_mass", "g_ws",
                      "graph_kernels")
    MAX_CAPTURES = 4

    def _restore_capture(self, sig, cap: dict) -> None:
        for name in self._CAPTURE_STATE:
            setattr(self, name, cap[name])
        self.graph = self.graphs[0]
        self._graph_sig = sig

    def decode_step_graph(self, q, k_new, v_new, copy: int = 0):
        """One decode step through the captured graph (copy ``copy``): q [L, B,
        Hq, T, 128], k_new / v_new [L, B, Hkv, 128]; returns the static output
        [L, B, Hq, T, 128] (overwritten by the next step)."""
        if self.graph is None:
            raise RuntimeError("capture_decode() first (after the prefill)")
        self.g_q.copy_(q, non_blocking=True)
        self.g_k.copy_(k_new, non_blocking=True)
        self.g_v.copy_(v_new, non_blocking=True)
        self.graphs[copy].replay()
        self.n_pos += 1
        return self.g_out

    def graph_attention_ms(self, copy: int) -> List[float]:
        """Waits for the last replay of graph copy ``copy`` and returns the
        attention times (ms) of its timed layers from the captured events."""
        ev = self.g_events[copy]
        last = max(ev)
        ev[last][1].synchronize()
        return [ev[l][0].elapsed_time(ev[l][1]) for l in sorted(ev)]

    def sync_host_counts(self) -> None:
        """Refresh the host copies of the generated-token counts after graphed
        steps (uc_append_next advances only the device counts)."""
        for g in self.gen:
            if g is not None:
                g.sync_host()

    # --------------------------------------------------------------- reporting
    def stored_bytes(self, with_index: bool = False) -> int:
        return sum(s.stored_bytes(with_index) for segs in self.layers for s in segs)

    def cache_bytes(self, layer: int, include_generated: bool = True) -> int:
        """Bytes one decode attention call over this layer reads (K + V)."""
        return sum(s.stored_bytes() for s in self.layers[layer]
                   if include_generated or s is not self.gen[layer] or self.gen_capacity == 0)

    def full_bytes(self) -> int:
        return self.L * self.B * self.hkv * self.n_ctx * 4 * 128


# ------------------------------------------------------------ Eq. 3 schedule

@dataclasses.dataclass
class ScheduleConfig:
    """Constants of §3.3's temporal schedule: Eq. 3's initial and minimum
    retention ratios (0 < rho_min <= rho_init <= 1) and the chunking of
    Eq. 1's statistics (layers per layer chunk, denoising steps per step
    chunk)."""
    rho_init: float = 0.5
    rho_min: float = 0.2
    layer_chunk: int = 4
    step_chunk: int = 5


class TemporalSchedule:
    """Task-aware temporal budget over the denoising steps of one generation
    (§3.3 Eq. 1-3, §3.4).

    Chunk 0 is the first denoising step, attended with the full KV; its
    attention mass gives m_a^(0) and M^(0) per (layer chunk, sequence). Every
    later chunk spans ``step_chunk`` steps; at its end the chunk's Eq. 1
    statistics m_a^(c) (the mean over the chunk's layer-step pairs of the
    mass each attention call reports on the type's retained keys) give
    M^(c) = sum_a m_a^(c), Eq. 3 gives rho^(c+1), Eq. 2 the type budgets
    (capped by the previous ones) and §3.4 each type's configuration. A type
    whose configuration shrank is re-compressed from what it still holds
    (eviction is irreversible); a ``fresh`` type, whose bf16 rows the caller
    rewrites every step, is compressed from those rows every step at its
    current configuration instead.

    types: the context's cache types in context order, policy 'full'
    (protected) or the candidate's calibrated policy 'evict' / 'quant'.
    The context K/V of layer l is one tensor [B, Hkv, N_ctx, 128] holding
    the types' rows in that order; eviction scores are observation-window
    scores over it, taken once at ``start`` (the eviction policy's state).
    """

    def __init__(self, types: Sequence[CacheType], n_layers: int, batch: int, device,
                 cfg: Optional[ScheduleConfig] = None, n_q_heads: int = 28, n_kv_heads: int = 4,
                 fresh: Sequence[str] = (), ws: Optional[api.Workspace] = None):
        self.types = list(types)
        for t in self.types:
            if t.policy not in ("full", "evict", "quant"):
                raise ValueError(f"type {t.name}: policy must be full, evict or quant")
        self.cfg = cfg or ScheduleConfig()
        self.L, self.B = n_layers, batch
        self.device = torch.device(device)
        self.hq, self.hkv = n_q_heads, n_kv_heads
        self.fresh = set(fresh)
        self.ws = ws or api.Workspace(self.device)
        self.n_ctx = sum(t.n for t in self.types)
        self.begin = np.cumsum([0] + [t.n for t in self.types])[:-1].tolist()
        self.n_lc = (n_layers + self.cfg.layer_chunk - 1) // self.cfg.layer_chunk
        self.cand = [a for a, t in enumerate(self.types) if t.candidate]
        self.scores = None
        self.mass_buf = None
        self._pool: Dict[tuple, api.Segment] = {}
        self._slot: Dict[tuple, int] = {}
        self.trace: List[dict] = []

    # ------------------------------------------------------------ helpers
    def _lc(self, l: int) -> int:
        return l // self.cfg.layer_chunk

    def _layers_of(self, lc: int) -> range:
        c = self.cfg.layer_chunk
        return range(lc * c, min(self.L, (lc + 1) * c))

    def _chunk_of(self, step: int) -> int:
        return 0 if step == 0 else 1 + (step - 1) // self.cfg.step_chunk

    def _steps_in_chunk(self, c: int) -> int:
        if c == 0:
            return 1
        first = 1 + (c - 1) * self.cfg.step_chunk
        return max(1, min(self.cfg.step_chunk, self.n_steps - first))

    def _is_chunk_end(self, step: int) -> bool:
        return step == 0 or step % self.cfg.step_chunk == 0 or step == self.n_steps - 1

    def _new_segment(self, l: int, a: int, kind: int, bits: int, cap: int) -> api.Segment:
        """A segment from a two-slot pool per (layer, type): the new
        configuration never shares storage with the one it is built from."""
        slot = self._slot.get((l, a), 0) ^ 1
        self._slot[(l, a)] = slot
        key = (l, a, kind, bits, cap, slot)
        seg = self._pool.get(key)
        if seg is None:
            seg = api.Segment(kind, bits, self.B, self.hkv, self.types[a].n, cap, self.device)
            self._pool[key] = seg
        return seg

    def _config(self, tables, a: int):
        """§3.4 for one type of one layer chunk (uc_plan_batch): per-sequence
        keep counts, one kind and bit width for the batch."""
        kind, bits, full_view, keep = api.plan_batch(tables, a)
        return (KIND_FULL if full_view else kind, bits, tuple(keep))

    # ------------------------------------------------------------ public
    def start(self, k, v, qwin, n_steps: int, scores: Optional[torch.Tensor] = None) -> None:
        """k, v: per layer the context [B, Hkv, N_ctx, 128] bf16; qwin: per
        layer the observation window [B, Hq, W, 128]; n_steps: denoising
        steps of this generation. Chunk 0 (step 0) attends the full KV.
        ``scores`` [L, B, Hkv, N_ctx] fp32: eviction scores supplied by the
        caller instead of the observation-window scores of ``qwin``."""
        self.k, self.v, self.n_steps = k, v, n_steps
        L, B = self.L, self.B
        if scores is not None:
            self.scores = scores
        else:
            if self.scores is None or self.scores.shape != (L, B, self.hkv, self.n_ctx):
                self.scores = torch.empty((L, B, self.hkv, self.n_ctx), dtype=torch.float32, device=self.device)
            for l in range(L):
                api.score_accumulate(qwin[l], k[l], out=self.scores[l], ws=self.ws)
        self.config = [[(KIND_FULL, 16, tuple([t.n] * B)) for t in self.types] for _ in range(self.n_lc)]
        self.segs = [[api.Segment.view(k[l], v[l], self.begin[a], t.n) for a, t in enumerate(self.types)]
                     for l in range(L)]
        self.tables = [[None] * B for _ in range(self.n_lc)]
        self.rho = np.full((self.n_lc, B), self.cfg.rho_init)
        self.m0 = np.zeros((self.n_lc, B))
        self._fresh_step = [-1] * L
        self._obs = [0] * self.n_lc
        self.trace = []

    def segments(self, l: int, step: int) -> List[api.Segment]:
        """Layer l's context segments at ``step`` (fresh types compressed
        from their current rows, once per step)."""
        if self.fresh and self._fresh_step[l] != step:
            self._fresh_step[l] = step
            for a, t in enumerate(self.types):
                seg = self.segs[l][a]
                if t.name in self.fresh and seg.c.kind != KIND_FULL:
                    api.compress_segment(self.k[l], self.v[l], seg, begin=self.begin[a], scores=self.scores[l],
                                         ws=self.ws)
        return self.segs[l]

    def observe(self, l: int, step: int, mass: torch.Tensor) -> None:
        """Accumulate Eq. 1 from layer l's attention at ``step``: mass
        [B, Hq, T, n_seg] as uc_attend wrote it, the context types first."""
        lc = self._lc(l)
        ns = mass.shape[-1]
        if self.mass_buf is None or self.mass_buf.shape != (self.n_lc, self.B, ns):
            self.mass_buf = torch.zeros((self.n_lc, self.B, ns), dtype=torch.float32, device=self.device)
        w = 1.0 / (len(self._layers_of(lc)) * self._steps_in_chunk(self._chunk_of(step)))
        api.attention_mass(mass, out=self.mass_buf[lc], weight=w, accumulate=self._obs[lc] > 0)
        self._obs[lc] += 1

    def end_step(self, step: int) -> bool:
        """After every layer attended at ``step``: at the end of a chunk,
        Eq. 3 and Eq. 2 for the next chunk and the re-compressions they call
        for. Returns True if a chunk ended."""
        if not self._is_chunk_end(step) or step == self.n_steps - 1:
            return False
        c = self._chunk_of(step)
        m = self.mass_buf.cpu().numpy().astype(np.float64)      # one read per chunk
        self._obs = [0] * self.n_lc
        changed = 0
        for lc in range(self.n_lc):
            for b in range(self.B):
                if c == 0:
                    t = api.SegmentTable([ty.n for ty in self.types], [ty.candidate for ty in self.types])
                    for a, ty in enumerate(self.types):
                        if ty.candidate:
                            t.c.policy[a] = POLICY_NAMES[ty.policy]
                    self.tables[lc][b] = t
                t = self.tables[lc][b]
                for a in range(len(self.types)):
                    t.c.mass[a] = float(m[lc, b, a])
                # M^(c) over the candidates, Eq. 3 (chunk 0: M^(0) and rho_init)
                rho, self.m0[lc, b] = api.retention_step(t, c == 0, self.rho[lc, b], self.cfg.rho_init,
                                                         self.cfg.rho_min, self.m0[lc, b])
                api.allocate_budget(t, rho, first_chunk=(c == 0))
                self.rho[lc, b] = rho
            for a in self.cand:
                new = self._config(self.tables[lc], a)
                old = self.config[lc][a]
                if new == old:
                    continue
                kind, bits, keep = new
                for l in self._layers_of(lc):
                    src = self.segs[l][a]
                    keep_l = [min(x, y) for x, y in zip(keep, src.n_kept())]
                    if kind == KIND_FULL:
                        continue
                    if kind == KIND_QUANT:
                        keep_l = src.n_kept()
                    dst = self._new_segment(l, a, kind, bits, max(1, max(keep_l)))
                    dst.set_keep(keep_l)
                    if self.types[a].name not in self.fresh:
                        api.recompress_segment(src, dst, scores=self.scores[l], scores_begin=self.begin[a],
                                               ws=self.ws)
                    self.segs[l][a] = dst
                    changed += 1
                self.config[lc][a] = new
        self.trace.append({"chunk": c, "step": step, "rho": self.rho.mean(axis=1).round(4).tolist(),
                           "recompressed": changed})
        return True

    def stored_bytes(self) -> int:
        """Bytes the context types occupy now (K + V, packed layout)."""
        return sum(s.stored_bytes() for segs in self.segs for s in segs)
