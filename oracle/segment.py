"""Compress one segment and append decode tokens (oracle; test infrastructure).

§3.4: each candidate segment is compressed by its own policy, independently;
the result is reassembled in original token order. App. E: eviction stores the
retained entries and their logical indices; quantization stores packed codes,
scales, minima and a bf16 residual tail; protected segments stay as they are.

Kinds: 'full' (stored as is), 'evict' (top-k kept, bf16), 'quant' (all tokens,
quantized) and 'evict_quant' (top-k kept, then the kept tokens quantized in
ascending index order — the composite reading for the measured workloads).

Appending decode tokens extends the kept sequence; quantized groups are the
consecutive runs of 32 kept tokens counted from the first one, so a segment
that grows by appends equals a segment compressed from the whole sequence at
once (a property the tests check).

``recompress`` compresses an already compressed slice further (progressive
re-eviction and re-quantization when a later chunk's budget is lower).

Pinned through ``select`` and ``quant``, by the append / one-shot
equivalence, by nested re-eviction equalling one-shot eviction, and by
re-quantization of on-grid data reproducing it exactly.
"""
import dataclasses
from typing import Optional

import numpy as np

from . import quant, select

GROUP = 32


@dataclasses.dataclass
class Seg:
    """One (sequence, KV head) slice of a compressed segment."""
    kind: str
    bits: int
    kept_idx: np.ndarray          # ascending logical indices
    k_kept: np.ndarray            # [n_kept, d] bf16 values of the kept keys
    v_kept: np.ndarray
    k_codes: Optional[np.ndarray] = None   # [32 g, d]
    k_scale: Optional[np.ndarray] = None   # [g, d] f16
    k_zero: Optional[np.ndarray] = None
    v_codes: Optional[np.ndarray] = None   # [32 g, d]
    v_scale: Optional[np.ndarray] = None   # [32 g, d/32] f16
    v_zero: Optional[np.ndarray] = None

    @property
    def n_kept(self) -> int:
        return int(self.kept_idx.shape[0])

    @property
    def n_groups(self) -> int:
        return self.n_kept // GROUP if self.bits < 16 else 0

    @property
    def tail(self) -> int:
        return self.n_kept - GROUP * self.n_groups if self.bits < 16 else 0

    def kv(self):
        """Keys and values attention sees, fp64 [n_kept, d] each."""
        if self.bits == 16:
            return self.k_kept.astype(np.float64), self.v_kept.astype(np.float64)
        ng = GROUP * self.n_groups
        k = np.concatenate([quant.dequantize_k(self.k_codes, self.k_scale, self.k_zero),
                            self.k_kept[ng:].astype(np.float64)])
        v = np.concatenate([quant.dequantize_v(self.v_codes, self.v_scale, self.v_zero),
                            self.v_kept[ng:].astype(np.float64)])
        return k, v


def _build(kind: str, bits: int, kept: np.ndarray, k_kept, v_kept) -> Seg:
    seg = Seg(kind, bits, kept, np.asarray(k_kept, np.float32), np.asarray(v_kept, np.float32))
    if bits < 16:
        ng = GROUP * (kept.shape[0] // GROUP)
        seg.k_codes, seg.k_scale, seg.k_zero = quant.quantize_k(seg.k_kept[:ng], bits)
        seg.v_codes, seg.v_scale, seg.v_zero = quant.quantize_v(seg.v_kept[:ng], bits)
    return seg


def compress(k: np.ndarray, v: np.ndarray, scores: Optional[np.ndarray],
             kind: str, keep: int, bits: int, n_recent: int = 0) -> Seg:
    """k, v [n, d] for one (sequence, KV head); scores [n] or None."""
    n = k.shape[0]
    if kind in ("full", "quant"):
        kept = np.arange(n, dtype=np.int64)
    elif kind in ("evict", "evict_quant"):
        kept = select.topk_keep(scores, keep, n_recent)
    else:
        raise ValueError(kind)
    if kind in ("full", "evict"):
        bits = 16
    return _build(kind, bits, kept, k[kept], v[kept])


def append(seg: Seg, k_new: np.ndarray, v_new: np.ndarray, first_index: int) -> Seg:
    """Append rows k_new, v_new [m, d] with logical indices first_index.."""
    m = k_new.shape[0]
    kept = np.concatenate([seg.kept_idx, first_index + np.arange(m, dtype=np.int64)])
    return _build(seg.kind, seg.bits, kept,
                  np.concatenate([seg.k_kept, k_new]), np.concatenate([seg.v_kept, v_new]))


def stored_rows(seg: Seg):
    """The stored tokens of ``seg`` as bf16 rows (float32 values) [n_kept, d]:
    bf16 rows as stored, packed groups rebuilt through ``quant.rebuild_bf16``,
    the residual tail as stored."""
    if seg.bits == 16:
        return seg.k_kept.copy(), seg.v_kept.copy()
    ng = GROUP * seg.n_groups
    k = np.concatenate([quant.rebuild_bf16(quant.dequantize_k(seg.k_codes, seg.k_scale, seg.k_zero)),
                        seg.k_kept[ng:]])
    v = np.concatenate([quant.rebuild_bf16(quant.dequantize_v(seg.v_codes, seg.v_scale, seg.v_zero)),
                        seg.v_kept[ng:]])
    return k.astype(np.float32), v.astype(np.float32)


def recompress(seg: Seg, scores: Optional[np.ndarray], kind: str, keep: int, bits: int,
               n_recent: int = 0) -> Seg:
    """Compress what ``seg`` still stores into a smaller configuration.

    §3.3 lowers a type's budget from chunk to chunk (Eq. 2 caps b_a^(c+1) by
    b_a^(c), Eq. 3 never raises rho) and notes that eviction is irreversible;
    §3.4 turns the new budget into the policy's configuration. Readings: the
    candidates are the tokens ``seg`` holds, as the bf16 rows of
    ``stored_rows``; an evicting kind scores them by their logical token
    (``scores`` is indexed by logical index, the eviction policy's state)
    and keeps ``keep`` of them with ``select.topk_keep`` (the ``n_recent``
    most recent stored tokens always); 'quant' keeps them all. The kept rows
    are then compressed as ``compress`` does, keeping their logical indices.
    """
    k_rows, v_rows = stored_rows(seg)
    n = seg.n_kept
    if kind == "quant":
        if keep != n:
            raise ValueError("quant keeps every stored token")
        rows = np.arange(n, dtype=np.int64)
    elif kind in ("evict", "evict_quant"):
        rows = select.topk_keep(np.asarray(scores)[seg.kept_idx], keep, n_recent)
    else:
        raise ValueError(kind)
    if kind == "evict":
        bits = 16
    return _build(kind, bits, seg.kept_idx[rows], k_rows[rows], v_rows[rows])


def stored_bytes(seg: Seg, d: int = 128, with_index: bool = False) -> int:
    """Bytes this slice occupies in the packed layout (per KV head)."""
    if seg.bits == 16:
        b = seg.n_kept * 4 * d
    else:
        ng = seg.n_groups
        codes = 2 * GROUP * ng * d * seg.bits // 8
        params = ng * d * 4 + GROUP * ng * (d // GROUP) * 4
        b = codes + params + seg.tail * 4 * d
    if with_index and seg.kind != "full":
        b += 4 * seg.n_kept
    return b
