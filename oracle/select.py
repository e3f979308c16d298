"""Per-KV-head token selection (oracle; test infrastructure only).

App. E ("Batched GQA token selection"): heavy-hitter plus recent-token
selection, independently for each KV head, on scores summed over the query
heads of that KV head.

Readings: exactly k tokens are kept; the ``n_recent`` most recent tokens are
always kept (0 in every measured configuration) and the rest are the largest
scores among the older tokens; equal scores go to the lower token index;
-0.0 equals +0.0; NaN is an error. The kept indices are returned ascending,
which is the original token order the paper reassembles (§3.4).

Pinned by tests against brute force over all k-subsets on small n (forced
ties, all-equal scores, k = n, k = 1).
"""
import numpy as np


def topk_keep(scores: np.ndarray, k: int, n_recent: int = 0) -> np.ndarray:
    s = np.asarray(scores)
    n = s.shape[0]
    if np.isnan(s).any():
        raise ValueError("NaN score")
    k = min(int(k), n)
    r = min(int(n_recent), k)
    old = n - r
    idx = np.arange(old)
    # full sort by (score descending, index ascending)
    order = np.lexsort((idx, -s[:old].astype(np.float64)))
    chosen = np.concatenate([order[:k - r], np.arange(old, n)])
    return np.sort(chosen).astype(np.int64)
