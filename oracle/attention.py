"""Shared-softmax attention over heterogeneous segments (oracle; test infra).

App. E ("Attention over heterogeneous cache segments"): all segments of one
(sequence, KV head) are combined under one softmax normalisation; chunks
computed separately merge by log-sum-exp. This is the plain definition with
no split: concatenate every segment's keys and values (dequantized, fp64),
take one softmax per query row, and report

    O[b, h, t]       = softmax(q K^T / sqrt(d)) V
    lse[b, h, t]     = log sum_k exp(q . k / sqrt(d))       (natural log)
    mass[b, h, t, s] = sum of the probabilities on segment s

``mass`` is the per-(layer, step) term inside Eq. 1. Query head h reads KV
head h // (Hq / Hkv). Readings: no mask (every cached token is visible to
decode queries; denoising latents attend bidirectionally); positions are
already encoded in the cached keys, so kept indices are metadata only.

``token_probabilities`` gives the same probabilities per token (summed over
the heads of a KV head and the query tokens), the per-step term of decode-time
heavy-hitter scores.

Pinned by tests against: torch scaled_dot_product_attention in fp64 for
uncompressed segments (ratio 1) and for exactly the kept subset (eviction),
probabilities summing to 1 (masses sum to 1), and the log-sum-exp merge of
separately computed parts equalling the unsplit result; token_probabilities
against observation scores of the same queries (a separately written route)
and against the per-segment mass of ``attend``.
"""
import numpy as np


def attend(q: np.ndarray, segs, hkv: int):
    """q [B, Hq, T, d]; segs[s][b][j] -> object with ``kv()`` giving fp64
    (K, V) [n, d] for sequence b and KV head j.

    Returns O [B, Hq, T, d], lse [B, Hq, T], mass [B, Hq, T, n_seg] (fp64)."""
    B, hq, T, d = q.shape
    g = hq // hkv
    nseg = len(segs)
    O = np.zeros((B, hq, T, d))
    lse = np.zeros((B, hq, T))
    mass = np.zeros((B, hq, T, nseg))
    for b in range(B):
        for j in range(hkv):
            ks, vs, owner = [], [], []
            for s, seg in enumerate(segs):
                k, v = seg[b][j].kv()
                ks.append(k)
                vs.append(v)
                owner.append(np.full(k.shape[0], s))
            K = np.concatenate(ks)
            V = np.concatenate(vs)
            own = np.concatenate(owner)
            if K.shape[0] == 0:
                raise ValueError("attention over an empty key set")
            rows = q[b, j * g:(j + 1) * g].reshape(g * T, d).astype(np.float64)
            logits = rows @ K.T / np.sqrt(d)
            m = logits.max(axis=1, keepdims=True)
            e = np.exp(logits - m)
            l = e.sum(axis=1, keepdims=True)
            p = e / l
            O[b, j * g:(j + 1) * g] = (p @ V).reshape(g, T, d)
            lse[b, j * g:(j + 1) * g] = (m[:, 0] + np.log(l[:, 0])).reshape(g, T)
            for s in range(nseg):
                mass[b, j * g:(j + 1) * g, :, s] = p[:, own == s].sum(axis=1).reshape(g, T)
    return O, lse, mass


def token_probabilities(q: np.ndarray, segs, hkv: int):
    """Heavy-hitter statistics of one attention call: for every segment s,
    an array [B, Hkv, n_s] holding, for each of its tokens, the softmax
    probability it receives summed over the query heads of its KV head and
    over the T query tokens (the same shared softmax as ``attend``). The
    accumulation of these per decode step is the heavy-hitter score of
    App. E's selection applied during decode."""
    B, hq, T, d = q.shape
    g = hq // hkv
    out = [np.zeros((B, hkv, seg[0][0].kv()[0].shape[0])) for seg in segs]
    for b in range(B):
        for j in range(hkv):
            ks = [seg[b][j].kv()[0] for seg in segs]
            K = np.concatenate(ks)
            rows = q[b, j * g:(j + 1) * g].reshape(g * T, d).astype(np.float64)
            logits = rows @ K.T / np.sqrt(d)
            m = logits.max(axis=1, keepdims=True)
            e = np.exp(logits - m)
            p = e / e.sum(axis=1, keepdims=True)
            col = p.sum(axis=0)
            off = 0
            for s, kk in enumerate(ks):
                n = kk.shape[0]
                if out[s].shape[2] != n:
                    raise ValueError("token_probabilities: ragged batches need one call per sequence")
                out[s][b, j] = col[off:off + n]
                off += n
    return out


class Plain:
    """A bf16 (uncompressed) slice given directly as K, V arrays."""

    def __init__(self, k, v):
        self.k = np.asarray(k)
        self.v = np.asarray(v)

    def kv(self):
        return self.k.astype(np.float64), self.v.astype(np.float64)
