"""Seeded synthetic inputs shaped like the paper's BAGEL workloads.

This module is shared by the tests, the benchmark and the oracle-driven checks.
It holds no arithmetic of the method itself: it only draws random numbers,
rounds them to bf16 (the storage type of a KV cache) and describes workload
shapes.

Recipe (the paper's models and datasets are not available, so these stand in
for them; §4.1 and §4.4 name BAGEL-7B-MoT with 28 query / 4 KV heads, d = 128):

* K ~ N(0, 1) with ``n_outlier`` channels per layer scaled by ``outlier_scale``
  (which channels is drawn from the seed), V ~ N(0, 1), Q ~ N(0, 1).
* Every tensor is rounded to bf16 before use, so the CPU checker and the GPU
  path see bit-identical inputs.
* Observation-window queries (``qwin``) are drawn like Q.

Two generators exist: ``numpy`` (host, used for the small parity cases) and
``torch`` on a CUDA device (used at full size where host generation would be
slow). Both are deterministic per seed; they produce different streams, and a
test always feeds the checker the same values that the GPU path consumed.
"""
from __future__ import annotations

import dataclasses
from typing import List, Optional, Sequence, Tuple

import numpy as np

HQ = 28          # query heads
HKV = 4          # KV heads
HEAD_DIM = 128   # head dimension
GQA = HQ // HKV  # query heads per KV head
GROUP = 32       # quantization group (tokens for K, channels for V)


def bf16_round(x: np.ndarray) -> np.ndarray:
    """Round a float array to the nearest bf16 value (ties to even); float32 out."""
    import torch
    t = torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32))
    return t.to(torch.bfloat16).to(torch.float32).numpy()


def outlier_channels(seed: int, n_outlier: int = 4, d: int = HEAD_DIM) -> np.ndarray:
    rng = np.random.default_rng(seed + 7919)
    return np.sort(rng.choice(d, size=n_outlier, replace=False))


def make_kv(seed: int, B: int, hkv: int, n: int, d: int = HEAD_DIM,
            n_outlier: int = 4, outlier_scale: float = 10.0) -> Tuple[np.ndarray, np.ndarray]:
    """K, V of shape [B, hkv, n, d] as bf16-valued float32 arrays."""
    rng = np.random.default_rng(seed)
    k = rng.standard_normal((B, hkv, n, d), dtype=np.float32)
    v = rng.standard_normal((B, hkv, n, d), dtype=np.float32)
    if n_outlier:
        k[..., outlier_channels(seed, n_outlier, d)] *= np.float32(outlier_scale)
    return bf16_round(k), bf16_round(v)


def make_q(seed: int, B: int, hq: int, t: int, d: int = HEAD_DIM) -> np.ndarray:
    """Queries [B, hq, t, d] as bf16-valued float32."""
    rng = np.random.default_rng(seed + 104729)
    return bf16_round(rng.standard_normal((B, hq, t, d), dtype=np.float32))


def make_scores(seed: int, shape: Sequence[int], tie_frac: float = 0.0) -> np.ndarray:
    """Positive fp32 score arrays for top-k tests; ``tie_frac`` of entries are
    snapped to a few shared values so that ties are common."""
    rng = np.random.default_rng(seed + 15485863)
    s = rng.exponential(1.0, size=shape).astype(np.float32)
    if tie_frac > 0:
        mask = rng.random(shape) < tie_frac
        levels = np.array([0.5, 1.0, 2.0], dtype=np.float32)
        s[mask] = levels[rng.integers(0, 3, size=int(mask.sum()))]
    return s


# ---------------------------------------------------------------- torch (GPU)

def torch_kv(seed: int, B: int, hkv: int, n: int, device, d: int = HEAD_DIM,
             n_outlier: int = 4, outlier_scale: float = 10.0):
    """Device K, V [B, hkv, n, d] bf16, generated on ``device`` from ``seed``."""
    import torch
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    k = torch.randn((B, hkv, n, d), generator=g, device=device, dtype=torch.float32)
    v = torch.randn((B, hkv, n, d), generator=g, device=device, dtype=torch.float32)
    if n_outlier:
        idx = torch.as_tensor(outlier_channels(seed, n_outlier, d), device=device)
        k[..., idx] *= outlier_scale
    return k.to(torch.bfloat16), v.to(torch.bfloat16)


def torch_q(seed: int, B: int, hq: int, t: int, device, d: int = HEAD_DIM):
    import torch
    g = torch.Generator(device=device)
    g.manual_seed(int(seed) + 104729)
    return torch.randn((B, hq, t, d), generator=g, device=device,
                       dtype=torch.float32).to(torch.bfloat16)


# ------------------------------------------------------------- workload specs

@dataclasses.dataclass
class SegmentSpec:
    """One cache type of a workload (§3.1 segmentation).

    kind: 'full' (protected or kept full), 'evict', 'quant', 'evict_quant'
    or 'auto' (policy from calibration and budget from Eq. 2).
    """
    name: str
    n: int
    kind: str
    keep_frac: float = 1.0
    bits: int = 16
    candidate: bool = True


@dataclasses.dataclass
class Workload:
    name: str
    layers: int
    batch: int
    segments: List[SegmentSpec]
    window: int = 32
    decode_steps: int = 0
    q_tokens: int = 1
    retention: Optional[float] = None   # fixed rho for understanding tasks
    gen_capacity: int = 0               # bf16 generated-token segment size
    flow_steps: int = 0                 # denoising steps per generation (dense workloads)
    quant_steps: int = 0                # leading flow steps whose latent cache is int4

    @property
    def n_ctx(self) -> int:
        return sum(s.n for s in self.segments)


def workload(name: str) -> Workload:
    """Workload shapes of the measured configurations (§4.4 scale)."""
    if name == "single_layer_1k":
        return Workload(name, 1, 1, [
            SegmentSpec("text", 256, "full", candidate=False),
            SegmentSpec("vit", 768, "evict_quant", keep_frac=0.2, bits=4),
        ], window=32, decode_steps=1)
    if name == "understanding_decode_8k":
        return Workload(name, 28, 8, [
            SegmentSpec("text", 512, "full", candidate=False),
            SegmentSpec("vit", 4 * 1792, "evict_quant", keep_frac=0.3, bits=4),
            SegmentSpec("gen", 512, "quant", bits=2),
        ], window=32, decode_steps=128)
    if name == "long_context_32k":
        n = 32768
        return Workload(name, 28, 16, [
            SegmentSpec("text", n // 10, "auto"),
            SegmentSpec("vit", n - n // 10, "auto"),
        ], window=32, decode_steps=256, retention=0.2, gen_capacity=256)
    if name == "long_context_128k":
        n = 131072
        return Workload(name, 28, 2, [
            SegmentSpec("text", n // 10, "auto"),
            SegmentSpec("vit", n - n // 10, "auto"),
        ], window=32, decode_steps=256, retention=0.2, gen_capacity=256)
    if name == "denoise_4k":
        # text-to-image: 256 prompt tokens, a cached copy of the 4096 latent
        # tokens (int4 for the first 40 of 50 flow steps, bf16 for the last
        # 20 %), and the current latents, which the 4096 latent queries also
        # attend to (protected, bf16)
        return Workload(name, 28, 4, [
            SegmentSpec("text", 256, "full", candidate=False),
            SegmentSpec("latent_cache", 4096, "quant", bits=4),
            SegmentSpec("latent", 4096, "full", candidate=False),
        ], window=32, q_tokens=4096, flow_steps=50, quant_steps=40)
    if name == "edit_4k":
        # image editing: 128 instruction tokens (full), 4096 source VAE tokens
        # (int4), 1792 source ViT tokens evicted to 20 %, and the current
        # latents (protected, bf16)
        return Workload(name, 28, 4, [
            SegmentSpec("text", 128, "full", candidate=False),
            SegmentSpec("vae", 4096, "quant", bits=4),
            SegmentSpec("vit", 1792, "evict", keep_frac=0.2),
            SegmentSpec("latent", 4096, "full", candidate=False),
        ], window=32, q_tokens=4096, flow_steps=50)
    raise KeyError(name)
