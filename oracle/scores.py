"""Observation-window attention scores (oracle; test infrastructure only).

Follows §3.3 (Eq. 1: P_{h,q,k} is the attention probability of query q in head
h on key k) and App. E ("Batched GQA token selection": scores are summed over
the query heads that share one KV head).

Reading used where the paper is silent: the window queries are W extra query
vectors that attend, without a causal mask, to all N context keys; each row's
softmax runs over the whole context (protected tokens included); a token's
score is the sum of its probabilities over the g query heads of its KV head
and over the W window queries. Query head h reads KV head h // g.

Pinned by tests against: the closed form sum_t score = g * W, a one-key
context (score = g * W exactly), and column sums of a library attention
(torch scaled_dot_product_attention in fp64 with V = identity).
``attention_type_mass`` is pinned to ``type_mass`` of the observation scores
of the same queries (two separately written routes to Eq. 1's inner term).
"""
import numpy as np


def observation_scores(qwin: np.ndarray, k: np.ndarray) -> np.ndarray:
    """qwin [B, Hq, W, d], k [B, Hkv, N, d]  ->  scores [B, Hkv, N] (fp64)."""
    B, hq, W, d = qwin.shape
    hkv, N = k.shape[1], k.shape[2]
    g = hq // hkv
    out = np.zeros((B, hkv, N), dtype=np.float64)
    for b in range(B):
        for j in range(hkv):
            rows = qwin[b, j * g:(j + 1) * g].reshape(g * W, d).astype(np.float64)
            keys = k[b, j].astype(np.float64)
            logits = rows @ keys.T / np.sqrt(d)
            logits = logits - logits.max(axis=1, keepdims=True)
            p = np.exp(logits)
            p = p / p.sum(axis=1, keepdims=True)
            out[b, j] = p.sum(axis=0)
    return out


def type_mass(scores_bt: np.ndarray, lo: int, hi: int, hq: int, window: int) -> float:
    """Eq. 1 inner term for one sequence and one (layer, step) pair:
    Mean over heads h and queries q of the probability mass on keys [lo, hi).

    ``scores_bt`` is [Hkv, N] for one sequence (already summed over the heads
    of each KV head and over the window queries)."""
    return float(scores_bt[:, lo:hi].sum() / (hq * window))


def attention_type_mass(mass: np.ndarray) -> np.ndarray:
    """Eq. 1 inner term per (sequence, type) for one (layer, step) pair, from
    the attention probabilities themselves: ``mass`` [B, Hq, T, n_types] holds
    each query's probability on each type's retained keys (as
    ``attention.attend`` reports it); the term is its mean over heads and
    queries -> [B, n_types] (fp64)."""
    m = np.asarray(mass, dtype=np.float64)
    return m.mean(axis=(1, 2))


def chunk_mass(per_pair_masses) -> float:
    """Eq. 1 outer average: mean over the (layer, step) pairs of a chunk."""
    v = np.asarray(per_pair_masses, dtype=np.float64)
    return float(v.mean())
