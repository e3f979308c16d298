"""Host policy of UniCache (oracle; test infrastructure only).

* ``concentration`` / ``assign_policy`` — App. B (Calibration Setting): the
  share of within-type attention mass held by the top 10 % of tokens,
  averaged over calibration examples; eviction if >= 0.5, else quantization.
* ``allocate_budget`` — §3.3 Eq. 2 plus its redistribution rule: a type's
  new budget is min(previous allocation, mass share x shared budget); budget
  left by capped types goes to uncapped types with positive mass in proportion
  to their mass. Types with zero mass receive nothing.
* ``retention_schedule`` — §3.3 Eq. 3.
* ``budget_to_policy`` — §3.4 (eviction sets the number of kept tokens,
  quantization sets the precision); the byte model is the packed layout's.
* ``chunk_mass`` — M^(c) of Eq. 3: the Eq. 1 masses summed over candidate
  types.
* ``plan_batch`` — §3.4 for a batch held in one segment per (layer, type):
  one kind and bit width for all sequences, keep counts per sequence.

Readings (the paper is silent): the top-10 % count is ceil(0.1 n); an
eviction budget keeps floor(budget / 512 B) tokens per KV head; a quantization
budget takes the widest of int4 / int2 that fits, and if int2 does not fit it
evicts down to floor(budget / int2 cost) tokens before quantizing. A batch's
segment for one type takes the lowest bit width any sequence's budget allows;
it is a plain view when every sequence keeps every token in bf16, quantized
whole when every sequence keeps every token, otherwise evicted (then
quantized for a quantization policy) with per-sequence keep counts.

Pinned by tests against: hand-worked Eq. 2 / Eq. 3 cases (tests/golden), an
independent water-level solution of Eq. 2 by bisection, invariants (sum <=
budget, caps respected, equal budget/mass ratios among uncapped types), and
closed forms of the concentration (uniform -> ceil(0.1 n)/n, one-hot -> 1).
"""
import math

import numpy as np

HEAD_DIM = 128
GROUP = 32


def topk_count(n: int, frac: float) -> int:
    """ceil(frac * n), guarded against binary rounding of frac * n."""
    return int(math.ceil(frac * n - 1e-9))


def concentration(mass: np.ndarray, top_frac: float = 0.1) -> float:
    mass = np.asarray(mass, dtype=np.float64)
    total = mass.sum()
    if total <= 0:
        return 0.0
    k = max(1, topk_count(mass.size, top_frac))
    top = np.sort(mass)[::-1][:k].sum()
    return float(top / total)


def assign_policy(concentrations, threshold: float = 0.5) -> str:
    """Average the per-example concentrations and choose the policy."""
    c = float(np.mean(np.asarray(concentrations, dtype=np.float64)))
    return "evict" if c >= threshold else "quant"


def allocate_budget(mass, prev, total: float, tol: float = 1e-12) -> np.ndarray:
    """Eq. 2 with redistribution. mass, prev: per-type arrays; total: B^(c+1)."""
    m = np.asarray(mass, dtype=np.float64)
    cap = np.asarray(prev, dtype=np.float64)
    b = np.zeros_like(m)
    s = m.sum()
    if s <= 0 or total <= 0:
        return b
    b = np.minimum(cap, m / s * total)
    for _ in range(len(m) + 1):
        rest = total - b.sum()
        open_ = (b < cap) & (m > 0)
        if rest <= tol * max(total, 1.0) or not open_.any():
            break
        share = rest * m[open_] / m[open_].sum()
        b[open_] = np.minimum(cap[open_], b[open_] + share)
    return b


def retention_schedule(rho_prev: float, rho_init: float, rho_min: float,
                       m_c: float, m_0: float) -> float:
    """Eq. 3: rho^(c+1) = min(rho^(c), max(rho_min, rho_init * M^(c) / M^(0)))."""
    return min(rho_prev, max(rho_min, rho_init * m_c / m_0))


def bytes_per_token(bits: int, d: int = HEAD_DIM) -> float:
    """Per-token, per-KV-head bytes of K + V in the packed layout.

    bf16: 2 * d * 2. Quantized: K and V codes (d * bits / 8 each), the V
    per-token (scale, zero) fp16 pairs for d / 32 channel groups, and the K
    per-channel (scale, zero) fp16 pairs amortised over 32 tokens."""
    if bits == 16:
        return 4.0 * d
    codes = 2 * d * bits / 8
    v_params = (d // GROUP) * 4
    k_params = d * 4 / GROUP
    return codes + v_params + k_params


def budget_to_policy(policy: str, budget: float, n: int, d: int = HEAD_DIM):
    """Map a byte budget (per KV head) to (keep, bits)."""
    if n <= 0:
        return 0, 16
    if policy == "evict":
        keep = int(math.floor(budget / bytes_per_token(16, d) + 1e-9))
        return max(1, min(n, keep)), 16
    for bits in (4, 2):
        if n * bytes_per_token(bits, d) <= budget * (1 + 1e-12):
            return n, bits
    keep = int(math.floor(budget / bytes_per_token(2, d) + 1e-9))
    return max(1, min(n, keep)), 2


def keep_count(n: int, keep_frac: float) -> int:
    """Number of tokens a fixed keep fraction retains: max(1, floor(f n))."""
    if n <= 0:
        return 0
    return max(1, min(n, int(math.floor(keep_frac * n + 1e-9))))


def chunk_mass(mass, candidate) -> float:
    """M^(c) = sum of m_a^(c) over the candidate types (Eq. 3's statistic)."""
    return float(sum(float(m) for m, c in zip(mass, candidate) if c))


def config_kind(policy: str, keep: int, bits: int, n: int) -> str:
    """§3.4 for one sequence: the segment kind its (keep, bits) amounts to."""
    if policy == "evict":
        return "full" if keep == n else "evict"
    return "quant" if keep == n else "evict_quant"


def plan_batch(configs, n: int):
    """configs: per sequence (kind, keep, bits) of one type, kind in 'full',
    'evict', 'quant', 'evict_quant' (as §3.4 chose for that sequence alone).
    Returns (kind, bits, full_view, keeps) of the batch's segment."""
    keeps = [int(k) for _, k, _ in configs]
    if all(kind == "full" for kind, _, _ in configs):
        return "full", 16, True, keeps
    bits = min(int(b) for _, _, b in configs)
    if bits == 16:
        return "evict", 16, False, keeps
    return ("quant" if all(k == n for k in keeps) else "evict_quant"), bits, False, keeps
