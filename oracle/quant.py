"""Low-bit group quantization (oracle; test infrastructure only).

App. E ("Physical, type-aware KV storage"): quantized segments hold packed
low-bit codes with scales and minima, plus a short bf16 residual tail.
Parameters not in the paper (bit widths 4 / 2, group 32, fp16 scale and
zero-point, keys grouped per channel over 32 consecutive kept tokens, values
grouped per token over 32 consecutive channels) come from the measured
workload definitions.

Exact arithmetic (reading; every operation is IEEE binary32 round-to-nearest-
even, fp16 storage rounds to nearest even):

    qmax = 2**bits - 1
    s    = fp16( fp32(mx - mn) / qmax + 0 )  z = fp16(mn + 0)
    code = clamp( rint_even( fp32(x - z) / s ), 0, qmax );   code = 0 if s == 0
    x_hat = code * s + z                      (dequantization, fp64 here)

A group minimum of zero is stored as +0: the sign of a zero minimum changes
neither x - z nor x_hat, and adding +0 (round to nearest: -0 + 0 = +0) makes
the stored bits independent of which signed zero a minimum search returns.
The same holds for a zero scale: a group of zeros of both signs gives
mx - mn = -0 when the maximum search returns -0 and the minimum +0; the
scale is stored as +0 either way (its codes are all 0).
An fp16 scale or zero-point that is infinite, or a non-finite input, is an
error. The last (n mod 32) kept tokens stay in bf16 for both K and V.

Pinned by tests against: the exactly nearest quantization level (computed in
fp64 from s and z) for every element whose exact quotient is not within
fp32 rounding of a half-way point, the bound |x - x_hat| <= s/2 for unclamped
elements (plus the fp16 rounding slack of s and z at the clamped ends), and
known fp16 roundings (65504, subnormals, ties to even). ``round_bf16`` is
pinned to torch's bf16 conversion and hand-worked ties; ``rebuild_bf16`` by a
case where rounding through fp32 and rounding once differ.
"""
import numpy as np

GROUP = 32


class RangeError(ValueError):
    """A scale or zero-point does not fit fp16, or the input is not finite."""


def _params(mn: np.ndarray, mx: np.ndarray, bits: int):
    qmax = np.float32(2 ** bits - 1)
    with np.errstate(over="ignore"):
        s16 = ((mx.astype(np.float32) - mn.astype(np.float32)) / qmax + np.float32(0.0)).astype(np.float16)
        z16 = (mn.astype(np.float32) + np.float32(0.0)).astype(np.float16)
    if not (np.isfinite(s16).all() and np.isfinite(z16).all()):
        raise RangeError("scale or zero-point overflows fp16")
    return s16, z16


def _codes(x: np.ndarray, s16: np.ndarray, z16: np.ndarray, bits: int) -> np.ndarray:
    qmax = np.float32(2 ** bits - 1)
    s = s16.astype(np.float32)
    z = z16.astype(np.float32)
    t = x.astype(np.float32) - z
    safe = np.where(s == 0, np.float32(1), s)
    q = np.rint(t / safe)
    q = np.where(s == 0, np.float32(0), q)
    return np.clip(q, 0, qmax).astype(np.uint8)


def quantize_k(x: np.ndarray, bits: int):
    """Keys, per channel. x [n, d] (bf16 values, n multiple of 32).
    Returns codes [n, d] uint8, scale [n/32, d] f16, zero [n/32, d] f16."""
    x = np.asarray(x, dtype=np.float32)
    if not np.isfinite(x).all():
        raise RangeError("non-finite key")
    n, d = x.shape
    ng = n // GROUP
    xg = x[:ng * GROUP].reshape(ng, GROUP, d)
    s16, z16 = _params(xg.min(axis=1), xg.max(axis=1), bits)
    codes = _codes(xg, s16[:, None, :], z16[:, None, :], bits)
    return codes.reshape(ng * GROUP, d), s16, z16


def quantize_v(x: np.ndarray, bits: int):
    """Values, per token. x [n, d]. Returns codes [n, d] uint8,
    scale [n, d/32] f16, zero [n, d/32] f16."""
    x = np.asarray(x, dtype=np.float32)
    if not np.isfinite(x).all():
        raise RangeError("non-finite value")
    n, d = x.shape
    xg = x.reshape(n, d // GROUP, GROUP)
    s16, z16 = _params(xg.min(axis=2), xg.max(axis=2), bits)
    codes = _codes(xg, s16[:, :, None], z16[:, :, None], bits)
    return codes.reshape(n, d), s16, z16


def round_bf16(x) -> np.ndarray:
    """fp32 -> nearest bf16 (ties to even), returned as float32 values.

    bf16 keeps the upper 16 bits of the binary32 pattern; rounding adds
    0x7FFF plus the lowest kept bit before truncating (round half to even
    on the dropped 16 bits). Inputs here are finite."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) & 0xFFFF0000
    return u.astype(np.uint32).view(np.float32)


def rebuild_bf16(x_hat: np.ndarray) -> np.ndarray:
    """Dequantized values (exact, fp64) as the bf16 rows a re-compression
    starts from: the value is first rounded to fp32 (as a fused multiply-add
    of code * s + z rounds it), then to bf16. code * s + z needs at most 44
    significant bits, so the fp64 x_hat is exact before these roundings."""
    return round_bf16(np.asarray(x_hat, np.float64).astype(np.float32))


def dequantize_k(codes, s16, z16) -> np.ndarray:
    n, d = codes.shape
    c = codes.reshape(n // GROUP, GROUP, d).astype(np.float64)
    out = c * s16.astype(np.float64)[:, None, :] + z16.astype(np.float64)[:, None, :]
    return out.reshape(n, d)


def dequantize_v(codes, s16, z16) -> np.ndarray:
    n, d = codes.shape
    c = codes.reshape(n, d // GROUP, GROUP).astype(np.float64)
    out = c * s16.astype(np.float64)[:, :, None] + z16.astype(np.float64)[:, :, None]
    return out.reshape(n, d)
