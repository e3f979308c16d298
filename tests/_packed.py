"""Test-side helpers: decode the packed segment layout of include/unicache.h
into logical arrays, and the attention tolerance check.

Decoding is layout bookkeeping (where each code sits), not the method's
arithmetic, so it lives with the tests rather than in the oracle.
"""
import numpy as np

GROUP = 32
D = 128


def _words(raw: np.ndarray) -> np.ndarray:
    return np.ascontiguousarray(raw).view(np.uint32)


def unpack_k_codes(raw: np.ndarray, n_groups: int, bits: int) -> np.ndarray:
    """raw: bytes of one (b, kvh) block -> codes [32 * n_groups, 128]."""
    mask = (1 << bits) - 1
    per_lane = bits * 4
    kpairs = 16 // bits
    out = np.zeros((32 * n_groups, D), dtype=np.uint8)
    w = _words(raw[: n_groups * 4 * 32 * per_lane]).reshape(n_groups * 4, 32, per_lane // 4)
    for lane in range(32):
        n, j = lane >> 2, lane & 3
        for q in range(per_lane // 4):
            word = w[:, lane, q]
            for p in range(kpairs):
                i = q * (kpairs // 2) + p // 2
                sub = p & 1
                ca = 16 * i + 2 * j + 8 * sub
                tok = np.arange(n_groups * 4) * 8 + n
                out[tok, ca] = (word >> (bits * p)) & mask
                out[tok, ca + 1] = (word >> (16 + bits * p)) & mask
    return out


def unpack_k_params(raw: np.ndarray, n_groups: int):
    """-> scale, zero [n_groups, 128] float16."""
    h = np.ascontiguousarray(raw[: n_groups * 512]).view(np.float16).reshape(n_groups, 8, 4, 8)
    s = np.zeros((n_groups, D), np.float16)
    z = np.zeros((n_groups, D), np.float16)
    for i in range(8):
        for j in range(4):
            c0 = 16 * i + 2 * j
            e = h[:, i, j]
            s[:, c0], s[:, c0 + 1], s[:, c0 + 8], s[:, c0 + 9] = e[:, 0], e[:, 1], e[:, 2], e[:, 3]
            z[:, c0], z[:, c0 + 1], z[:, c0 + 8], z[:, c0 + 9] = e[:, 4], e[:, 5], e[:, 6], e[:, 7]
    return s, z


def unpack_v_codes(raw: np.ndarray, n_groups: int, bits: int) -> np.ndarray:
    mask = (1 << bits) - 1
    per_lane = bits * 8
    kpairs = 16 // bits
    nt = 2 * n_groups
    out = np.zeros((16 * nt, D), dtype=np.uint8)
    w = _words(raw[: nt * 32 * per_lane]).reshape(nt, 32, per_lane // 4)
    for lane in range(32):
        gq, j = lane >> 2, lane & 3
        for q in range(per_lane // 4):
            word = w[:, lane, q]
            for p in range(kpairs):
                m = q * (kpairs // 2) + p // 2
                sub = p & 1
                ta = np.arange(nt) * 16 + 2 * j + 8 * sub
                c = 8 * m + gq
                out[ta, c] = (word >> (bits * p)) & mask
                out[ta + 1, c] = (word >> (16 + bits * p)) & mask
    return out


def unpack_v_params(raw: np.ndarray, n_groups: int):
    """-> scale, zero [32 * n_groups, 4] float16."""
    nt = 2 * n_groups
    h = np.ascontiguousarray(raw[: nt * 256]).view(np.float16).reshape(nt, 4, 4, 8)
    s = np.zeros((16 * nt, 4), np.float16)
    z = np.zeros((16 * nt, 4), np.float16)
    for g in range(4):
        for j in range(4):
            t0 = np.arange(nt) * 16 + 2 * j
            e = h[:, g, j]
            for k, off in enumerate((0, 1, 8, 9)):
                s[t0 + off, g] = e[:, k]
                z[t0 + off, g] = e[:, 4 + k]
    return s, z


def half_ulp_bf16(x: np.ndarray) -> np.ndarray:
    """Half a bf16 unit in the last place at |x| (0 for x = 0)."""
    ax = np.abs(np.asarray(x, np.float64))
    e = np.floor(np.log2(np.where(ax > 0, ax, 1.0)))
    return np.where(ax > 0, 2.0 ** (e - 8), 0.0)


def attention_error(o: np.ndarray, r: np.ndarray) -> float:
    """Largest per-row error of bf16 outputs o against the fp64 reference r,
    after allowing each element its own bf16 output rounding, relative to the
    row's max |r|. Rows are the last axis."""
    o = np.asarray(o, np.float64)
    r = np.asarray(r, np.float64)
    slack = half_ulp_bf16(np.maximum(np.abs(o), np.abs(r)))
    err = np.maximum(np.abs(o - r) - slack, 0.0).max(axis=-1)
    scale = np.abs(r).max(axis=-1)
    return float((err / np.where(scale > 0, scale, 1.0)).max())


ATTN_RTOL = 2e-3


def logit_error_bound(q: np.ndarray, segs, hkv: int, quantized) -> np.ndarray:
    """Per query row, a bound on the logit error of the GPU path: keys of a
    quantized segment are rebuilt in fp16 (relative error <= 2^-11 per
    element), bf16 keys enter exactly (fp32 accumulation, ~2^-20 here), so
    |d logit| <= eps * sum_c |q_c k_c| / sqrt(d). lse moves by at most the
    largest such error and a segment's mass by at most twice it."""
    B, hq, T, d = q.shape
    g = hq // hkv
    out = np.zeros((B, hq, T))
    for b in range(B):
        for j in range(hkv):
            rows = np.abs(q[b, j * g:(j + 1) * g].reshape(g * T, d).astype(np.float64))
            worst = np.zeros(g * T)
            for seg, qz in zip(segs, quantized):
                kk, _ = seg[b][j].kv()
                if kk.shape[0] == 0:
                    continue
                eps = 2.0 ** -11 if qz else 2.0 ** -20
                worst = np.maximum(worst, eps * (rows @ np.abs(kk).T).max(axis=1) / np.sqrt(d))
            out[b, j * g:(j + 1) * g] = worst.reshape(g, T)
    return out + 1e-6
