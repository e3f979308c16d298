"""Benchmark of the compressed-KV hot path on GB300.

Workload (default ``long_context_32k``): 28 layers x (28 query / 4 KV heads,
d = 128), batch 16, 32768 cached tokens per sequence (10 % text, 90 % image
tokens), both types compression candidates with calibrated policies and
attention-guided budgets at a fixed 0.2 retention (5x), then 256 decode
steps of one query token. One step = the whole hot path over one batch:
observation-window scores, Eq. 1 masses, Eq. 2 budgets, per-segment top-k /
gather / quantization for every layer, then 256 decode steps (append +
shared-softmax attention over all segments, every layer). The metric is
generated tokens per second of the whole job (batch x decode steps / step
time). Inputs are synthetic (seeded Gaussian K/V with outlier key channels),
resident in HBM before the timed region and far larger than L2 (30 GB of
bf16 KV per step), so no L2 flush is needed.

Also reported: the roofline of the dominant kernel (decode attention,
HBM-bound; CUDA events around every attention launch of the timed steps),
an end-to-end figure through the public API with host<->device copies in the
timed region, and the CPU oracle on a bounded sample of the same workload.

Dense workloads (``--workload denoise_4k`` or ``edit_4k``): one step is one
whole generation of batch 4: the conditioning caches compressed once, then
50 flow steps of 28 layers, each attending 4096 latent queries to the
compressed cache and to the current latents on the tensor cores (the first
40 flow steps of ``denoise_4k`` re-quantize the latent cache to int4). The
metric is denoising steps per second; the roofline is the attention calls'
algorithmic FLOPs over their CUDA-event time against the sustained bf16 peak.

  python bench.py [--steps K] [--warmup W] [--gpus N] [--impl native|reference] [--workload NAME]
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time
from typing import List, Optional

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

import synth  # noqa: E402

METRIC = "compressed-KV decode tokens/s at 32K context (HBM-bound attention, frac of peak)"
UNIT = "tokens/s"



def rank_env():
    """(world size, rank, local rank) from the torchrun environment."""
    return (int(os.environ.get("WORLD_SIZE", "1")), int(os.environ.get("RANK", "0")),
            int(os.environ.get("LOCAL_RANK", "0")))


def max_over_ranks(x: float, world: int, device) -> float:
    """The largest x over all ranks of the process group (x itself for one
    process): the slowest rank's time is the job's time."""
    if world <= 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(units_per_rank: float, world: int, ms: float) -> float:
    """Units all ranks processed per second (weak scaling: every rank does
    the same work), timed by the slowest rank."""
    return units_per_rank * world / (ms / 1000.0)

def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


# ----------------------------------------------------------------- clocks
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id: str):
        self.gpu = gpu_id
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            for n, val in zip(names, f[5:9]):
                if val.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        loaded = [s for s in sm if s > 0.5 * max(sm)] or sm
        return {"sm_mhz": statistics.median(loaded), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


# --------------------------------------------------------------- workload
def make_types(wl):
    from paper_2609_32831_gb300.engine import CacheType
    return [CacheType(s.name, s.n, s.kind if s.kind != "auto" else "auto", s.keep_frac, s.bits)
            for s in wl.segments]


def layer_seed(layer: int) -> int:
    return 5000 + layer


def gen_inputs(wl, device, decode_steps, rank):
    """Resident synthetic inputs of one batch: per-layer K, V, window queries,
    decode queries and new decode-token K/V."""
    import torch
    L, B, N = wl.layers, wl.batch, wl.n_ctx
    K = torch.empty((L, B, 4, N, 128), dtype=torch.bfloat16, device=device)
    V = torch.empty_like(K)
    Qw = torch.empty((L, B, 28, wl.window, 128), dtype=torch.bfloat16, device=device)
    for l in range(L):
        k, v = synth.torch_kv(layer_seed(l) + 100000 * rank, B, 4, N, device)
        K[l].copy_(k)
        V[l].copy_(v)
        Qw[l].copy_(synth.torch_q(layer_seed(l) + 7 + 100000 * rank, B, 28, wl.window, device))
        del k, v
    g = torch.Generator(device=device)
    g.manual_seed(777 + rank)
    Qd = torch.randn((decode_steps, L, B, 28, 1, 128), generator=g, device=device).to(torch.bfloat16)
    Kn = torch.randn((decode_steps, L, B, 4, 128), generator=g, device=device).to(torch.bfloat16)
    Vn = torch.randn((decode_steps, L, B, 4, 128), generator=g, device=device).to(torch.bfloat16)
    return K, V, Qw, Qd, Kn, Vn


def calibration_examples(wl, device, n_examples=10):
    """10 calibration examples (App. B), one sequence each, per layer."""
    for e in range(n_examples):
        def ks():
            for l in range(wl.layers):
                yield synth.torch_kv(90000 + 100 * e + l, 1, 4, wl.n_ctx, device)[0]

        def qs():
            for l in range(wl.layers):
                yield synth.torch_q(95000 + 100 * e + l, 1, 28, wl.window, device)
        yield ks(), qs()


# ------------------------------------------------------------ CPU oracle
def oracle_sample(wl, decode_steps: int, policies: dict, seed_layer: int = 0, chosen: Optional[dict] = None,
                  realized: Optional[dict] = None):
    """One bounded sample of the workload on the CPU oracle: one layer, one
    sequence, the whole compression path and ``decode_steps`` decode steps.
    A calibrated type missing from ``policies`` takes the oracle's own
    calibration on the sample (App. B: mean top-10 % share of its heads'
    scores, evict at >= 0.5); ``chosen`` receives the policies used and
    ``realized`` the sample's concentration per type and compression ratio.
    Returns (seconds of the compression, seconds of the decode steps)."""
    from oracle import attention as oattn
    from oracle import policy as opol
    from oracle import scores as osc
    from oracle import segment as oseg
    N = wl.n_ctx
    rng = np.random.default_rng(123)
    k, v = synth.make_kv(layer_seed(seed_layer), 1, 4, N)
    qw = synth.make_q(layer_seed(seed_layer), 1, 28, wl.window)
    qd = synth.bf16_round(rng.standard_normal((decode_steps, 1, 28, 1, 128)).astype(np.float32))
    kn = synth.bf16_round(rng.standard_normal((decode_steps, 4, 128)).astype(np.float32))
    vn = synth.bf16_round(rng.standard_normal((decode_steps, 4, 128)).astype(np.float32))
    t0 = time.perf_counter()
    s = osc.observation_scores(qw, k)
    begins = np.cumsum([0] + [t.n for t in wl.segments])
    m = [osc.type_mass(s[0], begins[a], begins[a + 1], 28, wl.window) for a in range(len(wl.segments))]
    sizes = np.array([t.n * 512.0 for t in wl.segments])
    if wl.retention is not None:
        b = opol.allocate_budget(m, sizes, wl.retention * sizes.sum())
    segs = []
    for a, t in enumerate(wl.segments):
        if wl.retention is None:        # the workload's fixed policies
            kind, bits = t.kind, t.bits
            keep = t.n if kind in ("full", "quant") else synth_keep(t)
        else:
            pol = policies.get(t.name)
            if pol is None:
                pol = opol.assign_policy([opol.concentration(s[0, j, begins[a]:begins[a + 1]]) for j in range(4)])
            if chosen is not None:
                chosen[t.name] = pol
            keep, bits = opol.budget_to_policy(pol, b[a], t.n)
            kind = "evict" if bits == 16 else ("quant" if keep == t.n else "evict_quant")
        lo, hi = begins[a], begins[a + 1]
        segs.append([[oseg.compress(k[0, j, lo:hi], v[0, j, lo:hi], s[0, j, lo:hi], kind, keep, bits)
                      for j in range(4)]])
    t1 = time.perf_counter()
    gen = [[oattn.Plain(np.zeros((0, 128)), np.zeros((0, 128))) for j in range(4)]]
    for t in range(decode_steps):
        gen = [[oattn.Plain(np.concatenate([gen[0][j].k, kn[t, j:j + 1]]),
                            np.concatenate([gen[0][j].v, vn[t, j:j + 1]])) for j in range(4)]]
        oattn.attend(qd[t], segs + [gen], 4)
    t2 = time.perf_counter()
    if realized is not None:
        realized["concentration"] = {
            t.name: float(np.mean([opol.concentration(s[0, j, begins[a]:begins[a + 1]]) for j in range(4)]))
            for a, t in enumerate(wl.segments) if wl.retention is not None}
        stored = sum(oseg.stored_bytes(sg) for seg in segs for sg in seg[0])
        realized["compression_ratio"] = 4 * N * 512 / max(1, stored)
    return t1 - t0, t2 - t1


def oracle_rate(wl, t_compress: float, t_decode: float, measured_steps: int) -> float:
    """Decode tokens/s of the oracle for the workload's step (one compression
    amortised over wl.decode_steps decode steps), from a sample that timed
    the compression and ``measured_steps`` decode steps of one layer and one
    sequence: tokens/s = D / (layers x (t_compress + D x t_decode / measured))."""
    D = wl.decode_steps
    return D / (wl.layers * (t_compress + D * t_decode / measured_steps))


def oracle_sample_text(wl, steps: int) -> str:
    return (f"1 of {wl.layers} layers, 1 of {wl.batch} sequences: full {wl.n_ctx}-token compression + {steps} "
            f"decode steps timed, the decode time scaled to the workload's {wl.decode_steps} steps per "
            f"compression; tokens/s = {wl.decode_steps} / (layers x (compression + {wl.decode_steps} x decode "
            f"step)); numpy fp64 with its BLAS threads")


def cpu_baseline(wl, policies, decode_steps=32):
    tc, td = oracle_sample(wl, decode_steps, policies)
    value = oracle_rate(wl, tc, td, decode_steps)
    return {"value": value, "unit": UNIT, "cores": os.cpu_count(), "kind": "oracle",
            "sample": oracle_sample_text(wl, decode_steps) + f"; {tc + td:.1f} s"}


# ------------------------------------------------------------------ probe
def attend_probe(kind: str, iters: int):
    """One layer of the long-context 32K cache (batch 16, 3276 + 29492 tokens
    per KV head) stored as `kind` (int2 / int4: all tokens quantized; bf16:
    20 % of tokens kept) and one decode-attention call timed `iters` times.
    Used for single-kernel profiles."""
    import torch

    import paper_2609_32831_gb300 as uc
    dev = torch.device("cuda")
    B, hkv, N = 16, 4, 32768
    n_text = N // 10
    k, v = synth.torch_kv(1, B, hkv, N, dev)
    segs = []
    for lo, n in [(0, n_text), (n_text, N - n_text)]:
        if kind == "bf16":
            seg = uc.Segment("evict", 16, B, hkv, n, n // 5, dev)
            seg.set_keep([n // 5] * B)
            uc.compress_segment(k, v, seg, begin=lo, scores=torch.rand((B, hkv, N), device=dev))
        else:
            seg = uc.Segment("quant", 2 if kind == "int2" else 4, B, hkv, n, n, dev)
            seg.set_keep([n] * B)
            uc.compress_segment(k, v, seg, begin=lo)
        segs.append(seg)
    q = synth.torch_q(2, B, 28, 1, dev)
    out = torch.empty_like(q)
    ws = uc.Workspace(dev)
    for _ in range(3):
        uc.attend(q, segs, out=out, want_lse=False, want_mass=False, ws=ws)
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for _ in range(iters):
        uc.attend(q, segs, out=out, want_lse=False, want_mass=False, ws=ws)
    b.record()
    torch.cuda.synchronize()
    us = a.elapsed_time(b) * 1000 / iters
    byts = sum(s.stored_bytes() for s in segs)
    print(json.dumps({"probe": "attend", "kind": kind, "us_per_launch": us, "bytes": byts,
                      "GBps": byts / us / 1e3, "status": ws.status()}))


def score_probe(iters: int):
    """Observation-window scores of one layer of the long-context 32K cache
    (batch 16, 4 KV heads, 32768 tokens, 28 heads x 32 window queries) timed
    `iters` times. Used for single-kernel profiles."""
    import torch

    import paper_2609_32831_gb300 as uc
    dev = torch.device("cuda")
    B, N = 16, 32768
    k, _ = synth.torch_kv(1, B, 4, N, dev)
    q = synth.torch_q(2, B, 28, 32, dev)
    out = torch.empty((B, 4, N), dtype=torch.float32, device=dev)
    ws = uc.Workspace(dev)
    for _ in range(3):
        uc.score_accumulate(q, k, out=out, ws=ws)
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for _ in range(iters):
        uc.score_accumulate(q, k, out=out, ws=ws)
    b.record()
    torch.cuda.synchronize()
    us = a.elapsed_time(b) * 1000 / iters
    print(json.dumps({"probe": "score", "us_per_call": us, "GBps": 2 * B * 4 * N * 256 / us / 1e3,
                      "row_sum": float(out.sum(dim=2).mean()), "status": ws.status()}))


def eviction_path(device, iters: int = 10) -> dict:
    """The eviction kernels on one layer of the long-context 32K cache (batch
    16, 4 KV heads, 32768 tokens: 3276 text + 29492 image), which the
    calibrated 32K workload itself does not run (both of its types are
    quantized): observation-window scores (both tcgen05 passes) and the
    image segment evicted to 20 % (per-head top-k over 29492 candidates,
    then the gather of the kept bf16 rows), each timed with CUDA events over
    `iters` calls after 3 warm-up calls."""
    import torch

    import paper_2609_32831_gb300 as uc
    B, hkv, N = 16, 4, 32768
    n_text = N // 10
    n_img = N - n_text
    keep = n_img // 5
    k, v = synth.torch_kv(1, B, hkv, N, device)
    q = synth.torch_q(2, B, 28, 32, device)
    scores = torch.empty((B, hkv, N), dtype=torch.float32, device=device)
    seg = uc.Segment("evict", 16, B, hkv, n_img, keep, device)
    seg.set_keep([keep] * B)
    ws = uc.Workspace(device)

    def timed(fn):
        for _ in range(3):
            fn()
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        for _ in range(iters):
            fn()
        b.record()
        torch.cuda.synchronize()
        return a.elapsed_time(b) * 1000.0 / iters

    score_us = timed(lambda: uc.score_accumulate(q, k, out=scores, ws=ws))
    evict_us = timed(lambda: uc.compress_segment(k, v, seg, begin=n_text, scores=scores, ws=ws))
    if ws.status() != 0:
        raise RuntimeError(f"eviction path: workspace status {ws.status()}")
    kept = seg.n_kept()
    del k, v, q, scores, seg, ws
    return {"workload": f"one layer of the 32K cache: batch {B}, {hkv} KV heads, {N} tokens; "
                        f"the {n_img}-token image segment evicted to {keep} per (sequence, KV head)",
            "score_accumulate_us": score_us, "evict_compress_us": evict_us,
            "kept_per_bh": int(min(kept)), "calls_timed": iters,
            "kernels": "score_accumulate: two tcgen05 passes + merge; compress_segment: per-head top-k + gather"}


def quant_probe(bits: int, iters: int, B: int = 16):
    """Group quantization of one layer of the long-context 32K cache (batch
    B = 16, 4 KV heads, all 32768 tokens kept, int4 or int2) through
    compress_segment, timed `iters` times: bf16 K and V rows read, codes and
    scale / zero-point pairs written (the kept-index list and the 32-row bf16
    tail are a few MB beside them). Used for single-kernel profiles."""
    import torch

    import paper_2609_32831_gb300 as uc
    dev = torch.device("cuda")
    hkv, N = 4, 32768
    k, v = synth.torch_kv(1, B, hkv, N, dev)
    seg = uc.Segment("quant", bits, B, hkv, N, N, dev)
    seg.set_keep([N] * B)
    ws = uc.Workspace(dev)
    for _ in range(3):
        uc.compress_segment(k, v, seg, ws=ws)
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for _ in range(iters):
        uc.compress_segment(k, v, seg, ws=ws)
    b.record()
    torch.cuda.synchronize()
    us = a.elapsed_time(b) * 1000 / iters
    read = 2 * B * hkv * N * 256
    written = B * hkv * N * (2 * 128 * bits // 8 + 32)  # K and V codes, 16 + 16 bytes of parameters per token
    print(json.dumps({"probe": "quant", "bits": bits, "batch": B, "us_per_call": us, "bytes": read + written,
                      "GBps": (read + written) / us / 1e3, "status": ws.status()}))


def batch_probe(iters: int):
    """Serving-shaped decode: eight requests of one layer with their own cache
    layouts (32768 down to 256 cached tokens, 10 % int4 prompt + int2 rest,
    batch 1, 28 / 4 heads), attended as eight uc_attend launches and as one
    uc_attend_batch launch (each replayed from a CUDA graph). Prints both
    timings and the stored bytes read."""
    import torch

    import paper_2609_32831_gb300 as uc
    dev = torch.device("cuda")
    calls = []
    for i, N in enumerate([32768, 16384, 8192, 4096, 2048, 1024, 512, 256]):
        k, v = synth.torch_kv(10 + i, 1, 4, N, dev)
        segs = []
        n_text = N // 10
        for lo, n, bits in [(0, n_text, 4), (n_text, N - n_text, 2)]:
            seg = uc.Segment("quant", bits, 1, 4, n, n, dev)
            seg.set_keep([n])
            uc.compress_segment(k, v, seg, begin=lo)
            segs.append(seg)
        q = synth.torch_q(20 + i, 1, 28, 1, dev)
        calls.append((q, segs, torch.empty_like(q)))
    ws1, ws2 = uc.Workspace(dev), uc.Workspace(dev)

    def separate():
        for q, segs, out in calls:
            uc.attend(q, segs, out=out, want_lse=False, want_mass=False, ws=ws1)

    def batched():
        uc.attend_batch([(q, segs, out) for q, segs, out in calls], ws=ws2)

    # each variant is captured once as a CUDA graph and replayed, so the
    # timings are device time, not the host cost of issuing the calls
    res = {}
    for name, fn in (("separate", separate), ("batched", batched)):
        for _ in range(3):
            fn()
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            fn()
        for _ in range(3):
            g.replay()
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        for _ in range(iters):
            g.replay()
        b.record()
        torch.cuda.synchronize()
        res[name] = a.elapsed_time(b) * 1000 / iters
    byts = sum(s.stored_bytes() for _, segs, _ in calls for s in segs)
    print(json.dumps({"probe": "attend_batch", "calls": len(calls), "bytes": byts,
                      "us_separate": res["separate"], "us_batched": res["batched"],
                      "GBps_separate": byts / res["separate"] / 1e3, "GBps_batched": byts / res["batched"] / 1e3,
                      "status": ws1.status() or ws2.status()}))


def profiled_traffic_ratio():
    """DRAM traffic per algorithmic byte of the attention kernel from the
    committed ncu summary, if it was taken from the current kernel source."""
    import hashlib
    path = os.path.join(ROOT, "profiles", "attend_kernel_long_context_32k_int2.md")
    src = os.path.join(ROOT, "paper_2609_32831_gb300", "csrc", "attend.cu")
    try:
        fields = dict(line.split(": ", 1) for line in open(path).read().splitlines() if ": " in line
                      and line.split(": ", 1)[0] in ("traffic_ratio", "source_sha256_16"))
        sha = hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]
        if fields.get("source_sha256_16", "").strip() == sha:
            return float(fields["traffic_ratio"])
    except Exception:
        pass
    return None


# ------------------------------------------------------ dense workloads
DENSE_METRIC = "denoising steps/s (4096 latent queries x 28 layers, batch 4; tensor-core attention)"
DENSE_UNIT = "steps/s"


def _tensor_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["bf16_tflops_sustained"]), float(p["bf16_tflops"]), "measured"
    except Exception:
        return 1700.0, 1900.0, "fallback"


def dense_keys(wl) -> int:
    """Keys every latent query attends to (kept tokens of every segment)."""
    n = 0
    for s in wl.segments:
        n += s.n if s.kind in ("full", "quant") else synth_keep(s)
    return n


def synth_keep(s) -> int:
    return max(1, int(np.floor(s.keep_frac * s.n)))


class DenseJob:
    """Resident inputs and segments of one denoising / editing generation:
    per layer the conditioning K/V (compressed once per generation), the
    current-latent K/V and the 4096 latent queries (both standing in for the
    model's per-step projections), and the latent-cache segment that the
    early flow steps re-quantize."""

    def __init__(self, wl, device, rank):
        import torch

        import paper_2609_32831_gb300 as uc
        self.uc, self.wl, self.dev = uc, wl, device
        L, B, T = wl.layers, wl.batch, wl.q_tokens
        self.cond = [s for s in wl.segments if s.name not in ("latent", "latent_cache")]
        self.n_cond = sum(s.n for s in self.cond)
        self.has_cache = any(s.name == "latent_cache" for s in wl.segments)
        self.Kc = torch.empty((L, B, 4, self.n_cond, 128), dtype=torch.bfloat16, device=device)
        self.Vc = torch.empty_like(self.Kc)
        self.Kl = torch.empty((L, B, 4, T, 128), dtype=torch.bfloat16, device=device)
        self.Vl = torch.empty_like(self.Kl)
        self.Q = torch.empty((L, B, 28, T, 128), dtype=torch.bfloat16, device=device)
        for l in range(L):
            k, v = synth.torch_kv(layer_seed(l) + 100000 * rank, B, 4, self.n_cond, device)
            self.Kc[l].copy_(k)
            self.Vc[l].copy_(v)
            k, v = synth.torch_kv(layer_seed(l) + 50000 + 100000 * rank, B, 4, T, device)
            self.Kl[l].copy_(k)
            self.Vl[l].copy_(v)
            self.Q[l].copy_(synth.torch_q(layer_seed(l) + 7 + 100000 * rank, B, 28, T, device))
        self.ws = uc.Workspace(device)
        self.scores = torch.empty((B, 4, self.n_cond), dtype=torch.float32, device=device)
        self.layers = []
        for l in range(L):
            segs, off = [], 0
            for s in self.cond:
                if s.kind == "full":
                    segs.append(("view", uc.Segment.view(self.Kc[l], self.Vc[l], off, s.n), off))
                else:
                    keep = s.n if s.kind == "quant" else synth_keep(s)
                    g = uc.Segment(s.kind, s.bits, B, 4, s.n, keep, device)
                    g.set_keep([keep] * B)
                    segs.append(("compress", g, off))
                off += s.n
            cache_q = cache_full = None
            if self.has_cache:
                cache_q = uc.Segment("quant", 4, B, 4, T, T, device)
                cache_q.set_keep([T] * B)
                cache_full = uc.Segment.view(self.Kl[l], self.Vl[l], 0, T)
            latent = uc.Segment.view(self.Kl[l], self.Vl[l], 0, T)
            self.layers.append((segs, cache_q, cache_full, latent))

    def prepare(self, l):
        """Compress layer l's conditioning caches (once per generation); the
        eviction scores come from an observation window of 32 latent queries."""
        uc = self.uc
        segs = self.layers[l][0]
        if any(kind == "compress" and seg.c.kind in (uc.KIND_EVICT, uc.KIND_EVICT_QUANT)
               for kind, seg, _ in segs):
            uc.score_accumulate(self.Q[l][:, :, :self.wl.window].contiguous(), self.Kc[l], out=self.scores,
                                ws=self.ws)
        for kind, seg, off in segs:
            if kind == "compress":
                uc.compress_segment(self.Kc[l], self.Vc[l], seg, begin=off, scores=self.scores, ws=self.ws)

    def segments(self, l, f):
        """Segment list of layer l at flow step f (re-quantizes the latent
        cache in the int4 steps)."""
        segs, cache_q, cache_full, latent = self.layers[l]
        out = [seg for _, seg, _ in segs]
        if self.has_cache:
            if f < self.wl.quant_steps:
                self.uc.compress_segment(self.Kl[l], self.Vl[l], cache_q, ws=self.ws)
                out.append(cache_q)
            else:
                out.append(cache_full)
        out.append(latent)
        return out

    def generation(self, out, lse, mass, events=None, flow_steps=None):
        F = flow_steps or self.wl.flow_steps
        for l in range(self.wl.layers):
            self.prepare(l)
        for f in range(F):
            for l in range(self.wl.layers):
                segs = self.segments(l, f)
                m = mass[:, :, :, :len(segs)]
                if events is not None:
                    events[f][l][0].record()
                self.uc.attend(self.Q[l], segs, out=out, lse=lse, mass=m, ws=self.ws)
                if events is not None:
                    events[f][l][1].record()


class ScheduledDenseJob:
    """One denoising / editing generation under §3.3's temporal schedule
    (Eq. 1-3) instead of fixed per-type configurations: step 0 attends the
    full context, later chunks of steps re-allocate the budget from the
    attention calls' own mass and re-compress the types whose budget fell.
    The context is every segment but the current latents; a latent cache is
    a fresh type, compressed from its rows every step."""

    def __init__(self, wl, device, rank, cfg):
        import torch

        import paper_2609_32831_gb300 as uc
        from paper_2609_32831_gb300 import engine
        self.uc, self.wl, self.dev = uc, wl, device
        L, B, T = wl.layers, wl.batch, wl.q_tokens
        ctx = [s for s in wl.segments if s.name != "latent"]
        self.n_ctx = sum(s.n for s in ctx)
        types = [engine.CacheType(s.name, s.n, "full" if s.kind == "full" else
                                  ("evict" if s.kind == "evict" else "quant")) for s in ctx]
        fresh = [s.name for s in ctx if s.name == "latent_cache"]
        self.Kc = torch.empty((L, B, 4, self.n_ctx, 128), dtype=torch.bfloat16, device=device)
        self.Vc = torch.empty_like(self.Kc)
        self.Kl = torch.empty((L, B, 4, T, 128), dtype=torch.bfloat16, device=device)
        self.Vl = torch.empty_like(self.Kl)
        self.Q = torch.empty((L, B, 28, T, 128), dtype=torch.bfloat16, device=device)
        n_cond = sum(s.n for s in ctx if s.name != "latent_cache")
        for l in range(L):
            k, v = synth.torch_kv(layer_seed(l) + 100000 * rank, B, 4, n_cond, device)
            self.Kc[l, :, :, :n_cond].copy_(k)
            self.Vc[l, :, :, :n_cond].copy_(v)
            k, v = synth.torch_kv(layer_seed(l) + 50000 + 100000 * rank, B, 4, T, device)
            self.Kl[l].copy_(k)
            self.Vl[l].copy_(v)
            if fresh:   # the latent cache holds a copy of the latents
                self.Kc[l, :, :, n_cond:].copy_(k)
                self.Vc[l, :, :, n_cond:].copy_(v)
            self.Q[l].copy_(synth.torch_q(layer_seed(l) + 7 + 100000 * rank, B, 28, T, device))
        self.ws = uc.Workspace(device)
        self.sched = engine.TemporalSchedule(types, L, B, device, cfg, fresh=fresh, ws=self.ws)
        self.latent = [uc.Segment.view(self.Kl[l], self.Vl[l], 0, T) for l in range(L)]
        self.Qw = self.Q[:, :, :, :wl.window].contiguous()   # observation window: 32 latent queries
        self.keys = []

    def generation(self, out, lse, mass, events=None, flow_steps=None, count_keys=False):
        F = flow_steps or self.wl.flow_steps
        sched = self.sched
        sched.start(self.Kc, self.Vc, self.Qw, F)
        if count_keys:
            self.keys = []
        for f in range(F):
            for l in range(self.wl.layers):
                segs = list(sched.segments(l, f)) + [self.latent[l]]
                if count_keys:
                    self.keys.append(sum(sum(s.n_kept()) for s in segs))
                if events is not None:
                    events[f][l][0].record()
                self.uc.attend(self.Q[l], segs, out=out, lse=lse, mass=mass, ws=self.ws)
                if events is not None:
                    events[f][l][1].record()
                sched.observe(l, f, mass)
            sched.end_step(f)


def dense_oracle_sample(wl, n_q: int = 1024):
    """One bounded sample on the CPU oracle: one layer, one sequence, one KV
    head (7 query heads), n_q of the 4096 latent queries; the conditioning
    compression, the latent-cache quantization of one int4 flow step and the
    attention. Returns (seconds per flow step of that unit, description)."""
    from oracle import attention as oattn
    from oracle import scores as osc
    from oracle import segment as oseg
    T = wl.q_tokens
    cond = [s for s in wl.segments if s.name not in ("latent", "latent_cache")]
    n_cond = sum(s.n for s in cond)
    kc, vc = synth.make_kv(layer_seed(0), 1, 1, n_cond)
    kl, vl = synth.make_kv(layer_seed(0) + 50000, 1, 1, T)
    q = synth.make_q(layer_seed(0) + 7, 1, 7, T)
    t0 = time.perf_counter()
    sc = osc.observation_scores(q[:, :, :wl.window], kc)
    segs, off = [], 0
    for s in cond:
        kind = s.kind
        keep = s.n if kind in ("full", "quant") else synth_keep(s)
        segs.append([[oseg.compress(kc[0, 0, off:off + s.n], vc[0, 0, off:off + s.n], sc[0, 0, off:off + s.n],
                                    kind, keep, s.bits)]])
        off += s.n
    t_cond = time.perf_counter() - t0
    t0 = time.perf_counter()
    if any(s.name == "latent_cache" for s in wl.segments):
        segs.append([[oseg.compress(kl[0, 0], vl[0, 0], None, "quant", T, 4)]])
    t_quant = time.perf_counter() - t0
    segs.append([[oattn.Plain(kl[0, 0], vl[0, 0])]])
    t0 = time.perf_counter()
    oattn.attend(q[:, :, :n_q], segs, 1)
    t_att = time.perf_counter() - t0
    secs = t_att * (T / n_q) + t_quant + t_cond / wl.flow_steps
    desc = (f"1 of {wl.layers} layers, 1 of {wl.batch} sequences, 1 of 4 KV heads: attention of {n_q} of {T} "
            f"latent queries ({t_att:.1f} s, scaled x{T / n_q:g}), the latent-cache int4 quantization "
            f"({t_quant:.1f} s) and the conditioning compression ({t_cond:.1f} s, /{wl.flow_steps}); "
            f"numpy fp64 with its BLAS threads")
    return secs, desc


def dense_cpu_value(wl, secs):
    """Flow steps per second if every (layer, sequence, KV head) unit took
    ``secs`` on these cores, one after another."""
    return 1.0 / (secs * wl.layers * wl.batch * 4)


def profiled_dense_traffic(wl):
    """DRAM bytes per dense-kernel launch from the committed ncu summary, if
    it was taken from the current kernel source."""
    import hashlib
    path = os.path.join(ROOT, "profiles", f"dense_kernel_{wl.name}.md")
    src = os.path.join(ROOT, "paper_2609_32831_gb300", "csrc", "dense.cu")
    try:
        fields = dict(line.split(": ", 1) for line in open(path).read().splitlines() if ": " in line
                      and line.split(": ", 1)[0] in ("traffic_bytes_per_launch", "source_sha256_16"))
        sha = hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]
        if fields.get("source_sha256_16", "").strip() == sha:
            return float(fields["traffic_bytes_per_launch"])
    except Exception:
        pass
    return None


def run_dense_reference(args, wl):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    for _ in range(args.warmup):
        dense_oracle_sample(wl, args.ref_queries)
    runs = [dense_oracle_sample(wl, args.ref_queries) for _ in range(args.steps)]
    secs = [r[0] for r in runs]
    desc = runs[-1][1]
    avg = sum(secs) / len(secs)
    value = dense_cpu_value(wl, avg)
    line = {"metric": DENSE_METRIC, "value": value, "unit": DENSE_UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000.0 * wl.flow_steps / value,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "impl": "reference",
            "config": {"workload": wl.name, "layers": wl.layers, "batch": wl.batch, "latent_queries": wl.q_tokens,
                       "keys": dense_keys(wl), "flow_steps": wl.flow_steps},
            "cpu_baseline": {"value": value, "unit": DENSE_UNIT, "cores": os.cpu_count(), "kind": "oracle",
                             "sample": f"each step (flow step of one unit): {desc}; value = 1 / (seconds x "
                                       f"{wl.layers} layers x {wl.batch} sequences x 4 KV heads)"},
            "e2e": {"value": value, "unit": DENSE_UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def dense_main(args, wl):
    import torch
    import torch.distributed as dist

    import paper_2609_32831_gb300 as uc
    world, rank, local = rank_env()
    device = torch.device(f"cuda:{local}")
    torch.cuda.set_device(device)
    if world > 1:
        dist.init_process_group("nccl", device_id=device)

    def barrier():
        if world > 1:
            dist.barrier()

    F = args.flow_steps or wl.flow_steps
    cfg = None
    if args.schedule == "eq3":
        from paper_2609_32831_gb300 import engine
        cfg = engine.ScheduleConfig(args.rho_init, args.rho_min, args.layer_chunk, args.step_chunk)
        make_job = lambda: ScheduledDenseJob(wl, device, rank, cfg)
    else:
        make_job = lambda: DenseJob(wl, device, rank)
    job = make_job()
    B, T, L = wl.batch, wl.q_tokens, wl.layers
    out = torch.empty((B, 28, T, 128), dtype=torch.bfloat16, device=device)
    lse = torch.empty((B, 28, T), dtype=torch.float32, device=device)
    mass = torch.empty((B, 28, T, len(wl.segments)), dtype=torch.float32, device=device)
    for _ in range(args.warmup):
        job.generation(out, lse, mass, flow_steps=F)
    torch.cuda.synchronize()
    ev = [[[(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
            for _ in range(L)] for _ in range(F)] for _ in range(args.steps)]
    try:
        uuid = str(torch.cuda.get_device_properties(device).uuid)
        gpu_id = uuid if uuid.startswith("GPU-") else "GPU-" + uuid
    except Exception:
        gpu_id = str(local)
    clocks = ClockSampler(gpu_id)
    n_launch0 = uc.launch_count()
    barrier()
    torch.cuda.synchronize()
    clocks.start()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record()
    for s in range(args.steps):
        job.generation(out, lse, mass, events=ev[s], flow_steps=F)
    t1.record()
    torch.cuda.synchronize()
    clk = clocks.stop()
    barrier()
    launches = uc.launch_count() - n_launch0
    ms = max_over_ranks(t0.elapsed_time(t1) / args.steps, world, device)
    value = whole_job_rate(F, world, ms)   # denoising steps of a batch-4 generation per second, all GPUs

    att_ms = [e[0].elapsed_time(e[1]) for st in ev for row in st for e in row]
    att_avg = sum(att_ms) / len(att_ms)
    if cfg is not None:
        job.generation(out, lse, mass, flow_steps=F, count_keys=True)   # untimed: kept keys per call
        torch.cuda.synchronize()
        nkeys = sum(job.keys) / (len(job.keys) * B)
    else:
        nkeys = dense_keys(wl)
    flops = 4.0 * B * 28 * T * nkeys * 128
    sustained, burst, src = _tensor_peaks()
    achieved = flops / (att_avg / 1000.0) / 1e12
    traffic = profiled_dense_traffic(wl) if cfg is None else None
    if cfg is not None:
        stored = full = 0
    else:
        stored = sum(seg.stored_bytes() for seg in job.segments(0, 0)[:-1])
        full = B * 4 * (nkeys - T) * 512
    result = {
        "metric": DENSE_METRIC, "value": value, "unit": DENSE_UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16 in/out, fp16 MMA operands (packed keys as fp16 hi + lo), fp32 accumulate",
        "data": "synthetic",
        "config": {"workload": wl.name, "layers": L, "batch_per_gpu": B, "latent_queries": T, "keys": nkeys,
                   "flow_steps_per_generation": F, "int4_latent_cache_steps": min(F, wl.quant_steps) if cfg is None else None,
                   "segments": [s.name for s in wl.segments],
                   "conditioning_compression": (full / max(1, stored)
                                                if wl.quant_steps == 0 and cfg is None else None),
                   "l2": "inputs larger than L2 (3.3 GB of queries per flow step; no flush)"},
        "ms_per_flow_step": ms / F,
        **({"schedule": {"rule": "Eq. 3 retention + Eq. 2 budgets, progressive re-compression",
                         "rho_init": cfg.rho_init, "rho_min": cfg.rho_min, "layer_chunk": cfg.layer_chunk,
                         "step_chunk": cfg.step_chunk, "mean_keys_per_sequence": nkeys,
                         "chunks": job.sched.trace}} if cfg is not None else {}),
        "roofline": {"bound": "tensor", "achieved": achieved, "peak": sustained, "unit": "TFLOP/s",
                     "frac": achieved / sustained, "traffic": traffic, "kernel": "uc::dense_kernel",
                     "flops_per_launch": flops, "avg_launch_us": att_avg * 1000.0,
                     "peak_source": f"{src} bf16 sustained", "frac_of_burst_peak": achieved / burst,
                     "timed": "uc_attend calls (materialize + dense kernels) by CUDA events"},
        "gpu_launches": int(launches),
        "clocks": clk,
    }
    if not args.no_e2e:
        result["e2e"] = dense_e2e(args, wl, job, out, lse, mass, device, world, F, make_job)
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        secs, desc = dense_oracle_sample(wl, args.ref_queries)
        result["cpu_baseline"] = {"value": dense_cpu_value(wl, secs), "unit": DENSE_UNIT, "cores": os.cpu_count(),
                                  "kind": "oracle", "sample": desc}
    if rank == 0:
        print(json.dumps(result), flush=True)
    if world > 1:
        dist.destroy_process_group()


class HostStaging:
    """Pinned host copies of one device input set, copied onto one of two
    device sets per step. The copy is split into chunks over several copy
    streams, so that more than one copy engine moves it; each stream first
    waits for the step that last read the target set. Records whether the
    host memory is pinned and the copy rate of an untimed copy."""

    def __init__(self, srcs, targets, n_streams=4):
        import torch
        self.host = []
        for t in srcs:
            try:
                h = torch.empty(t.shape, dtype=t.dtype, pin_memory=True)
            except RuntimeError:
                h = torch.empty(t.shape, dtype=t.dtype)
            h.copy_(t)
            self.host.append(h)
        self.targets = targets
        self.bytes = sum(t.numel() * t.element_size() for t in srcs)
        self.pinned = all(h.is_pinned() for h in self.host)
        self.streams = [torch.cuda.Stream() for _ in range(max(1, n_streams))]
        self.copied = [[torch.cuda.Event() for _ in self.streams] for _ in targets]
        self.released = [None] * len(targets)
        # chunks of at most 256 MB, dealt round-robin to the streams
        self.chunks = []
        for k, t in enumerate(srcs):
            rows = t.shape[0]
            per = max(1, (256 << 20) // max(1, t[0].numel() * t.element_size())) if t.dim() > 0 else 1
            for r0 in range(0, rows, per):
                self.chunks.append((k, r0, min(rows, r0 + per)))

    def issue(self, i):
        import torch
        for j, st in enumerate(self.streams):
            with torch.cuda.stream(st):
                if self.released[i] is not None:
                    st.wait_event(self.released[i])
                for c, (k, r0, r1) in enumerate(self.chunks):
                    if c % len(self.streams) == j:
                        self.targets[i][k][r0:r1].copy_(self.host[k][r0:r1], non_blocking=True)
                self.copied[i][j].record(st)

    def wait(self, i, stream):
        for ev in self.copied[i]:
            stream.wait_event(ev)

    def release(self, i, stream):
        import torch
        ev = torch.cuda.Event()
        ev.record(stream)
        self.released[i] = ev

    def reset(self):
        self.released = [None] * len(self.targets)

    def rate_gbps(self):
        """Copy rate of one untimed copy into target set 0 (host clock)."""
        import time
        import torch
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        self.issue(0)
        for evs in self.copied[0]:
            evs.synchronize()
        return self.bytes / (time.perf_counter() - t0) / 1e9


def dense_e2e(args, wl, job, out, lse, mass, device, world, F, make_job):
    """Whole generations through the public API with the inputs of each
    generation (conditioning K/V, latent queries and latent K/V of every
    layer) copied from pinned host memory and the last layer's output read
    back. Two jobs (two device input sets) alternate: the next generation's
    inputs are copied on separate copy streams while the current one
    computes."""
    import torch
    import torch.distributed as dist
    jobs = [job, make_job()]
    srcs = [[j.Kc, j.Vc, j.Kl, j.Vl, j.Q] for j in jobs]
    stage = HostStaging(srcs[0], srcs, args.copy_streams)
    h2d = stage.bytes
    out_host = torch.empty(out.shape, dtype=out.dtype, pin_memory=True)
    d2h = out.numel() * out.element_size()
    main = torch.cuda.current_stream()

    def gen(s_, last):
        i = s_ % 2
        stage.wait(i, main)
        if not last:
            stage.issue(1 - i)
        jobs[i].generation(out, lse, mass, flow_steps=F)
        out_host.copy_(out, non_blocking=True)
        stage.release(i, main)

    for i in range(2):          # warm both jobs
        stage.issue(i)
        gen(i, True)
    torch.cuda.synchronize()
    stage.reset()
    rate = stage.rate_gbps()
    torch.cuda.synchronize()
    stage.reset()
    n = max(1, min(args.steps, 2))
    if world > 1:
        dist.barrier()
    a = torch.cuda.Event(enable_timing=True)
    b = torch.cuda.Event(enable_timing=True)
    a.record()
    stage.issue(0)
    for s_ in range(n):
        gen(s_, s_ == n - 1)
    b.record()
    torch.cuda.synchronize()
    ms = max_over_ranks(a.elapsed_time(b) / n, world, device)
    return {"value": whole_job_rate(F, world, ms), "unit": DENSE_UNIT, "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h, "ms_per_step": ms, "steps": n, "host_pinned": stage.pinned,
            "h2d_GBps": rate, "copy_streams": len(stage.streams),
            "copies": "every generation's inputs H2D from pinned host memory; the next generation's copy "
                      "overlaps this one's compute on separate copy streams (two jobs)"}


# ------------------------------------------------------------------ main
def run_reference(args, wl):
    """The reference arm: the CPU oracle (the paper ships no code) on the same
    bounded sample as cpu_baseline, each step one compression and
    --ref-decode-steps decode steps of one layer and one sequence, scaled to
    the workload's decode steps per compression; the same config keys as the
    native line."""
    import torch.distributed as dist  # noqa: F401
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    pol = {}
    chosen, realized = {}, {}
    steps, warm, m = args.steps, args.warmup, args.ref_decode_steps
    for _ in range(warm):
        oracle_sample(wl, m, pol)
    times = [oracle_sample(wl, m, pol, chosen=chosen, realized=realized) for _ in range(steps)]
    tc = sum(t[0] for t in times) / steps
    td = sum(t[1] for t in times) / steps
    value = oracle_rate(wl, tc, td, m)
    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus, "steps": steps,
            "warmup": warm, "ms_per_step": 1000 * (tc + td), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "impl": "reference",
            "config": workload_config(wl, wl.decode_steps, chosen),
            "realized": realized,
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": os.cpu_count(), "kind": "oracle",
                             "sample": "each step: " + oracle_sample_text(wl, m)},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def workload_config(wl, decode_steps, policies) -> dict:
    """The `config` object of both arms' lines (the workload definition)."""
    return {"workload": wl.name, "layers": wl.layers, "batch_per_gpu": wl.batch, "context": wl.n_ctx,
            "decode_steps": decode_steps, "retention": wl.retention, "policies": dict(sorted(policies.items())),
            "l2": "inputs larger than L2 (no flush)"}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="native", choices=["native", "reference"])
    ap.add_argument("--workload", default="long_context_32k")
    ap.add_argument("--decode-steps", type=int, default=None)
    ap.add_argument("--ref-decode-steps", type=int, default=8,
                    help="reference arm: decode steps timed per step's sample (scaled to the workload's)")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--copy-streams", type=int, default=1,
                    help="copy streams that share each step's host-to-device input copy (end-to-end leg)")
    ap.add_argument("--eager", dest="decode_graph", action="store_false",
                    help="launch every decode kernel from Python instead of replaying the decode step as a "
                         "captured CUDA graph of the frozen layout (the default)")
    ap.add_argument("--decode-graph", dest="decode_graph", action="store_true", default=True,
                    help=argparse.SUPPRESS)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-eviction-path", action="store_true",
                    help="skip the one-layer timing of the eviction kernels (decode workloads that do not evict)")
    ap.add_argument("--no-pdl", dest="pdl", action="store_false",
                    help="captured decode step without programmatic dependent launch (each kernel waits for the "
                         "previous one to finish)")
    ap.add_argument("--attend-probe", choices=["int2", "int4", "bf16"], default=None,
                    help="time one decode-attention call of one layer instead of the bench")
    ap.add_argument("--iters", type=int, default=20)
    ap.add_argument("--stream-evict", default=None, metavar="BUDGET:WINDOW:INTERVAL",
                    help="decode workloads: heavy-hitter + recent-window re-eviction of the generated tokens")
    ap.add_argument("--quant-probe", type=int, choices=[2, 4], default=None,
                    help="time one layer's group quantization (int2 / int4) and exit")
    ap.add_argument("--probe-batch", type=int, default=16,
                    help="sequences of the --quant-probe layer (smaller for profiler captures)")
    ap.add_argument("--score-probe", action="store_true",
                    help="time the observation-window score kernels on one layer of the 32K cache")
    ap.add_argument("--batch-probe", action="store_true",
                    help="time eight serving-shaped decode calls separately and as one batched launch")
    ap.add_argument("--schedule", choices=["fixed", "eq3"], default="fixed",
                    help="dense workloads: fixed per-type configurations, or the Eq. 3 temporal schedule")
    ap.add_argument("--rho-init", type=float, default=0.5)
    ap.add_argument("--rho-min", type=float, default=0.2)
    ap.add_argument("--layer-chunk", type=int, default=4)
    ap.add_argument("--step-chunk", type=int, default=5)
    ap.add_argument("--flow-steps", type=int, default=None,
                    help="denoise / edit workloads: flow steps per generation (default: the workload's)")
    ap.add_argument("--layers", type=int, default=None,
                    help="fewer layers than the workload's (small cases for profiles only)")
    ap.add_argument("--ref-queries", type=int, default=1024,
                    help="denoise / edit workloads: latent queries in the oracle's bounded sample")
    args = ap.parse_args()
    if args.attend_probe:
        return attend_probe(args.attend_probe, args.iters)
    if args.batch_probe:
        return batch_probe(args.iters)
    if args.score_probe:
        return score_probe(args.iters)
    if args.quant_probe:
        return quant_probe(args.quant_probe, args.iters, args.probe_batch)
    wl = synth.workload(args.workload)
    if args.layers:
        wl.layers = args.layers
    if wl.q_tokens > 8:
        return run_dense_reference(args, wl) if args.impl == "reference" else dense_main(args, wl)
    if args.impl == "reference":
        return run_reference(args, wl)

    import torch
    import torch.distributed as dist

    import paper_2609_32831_gb300 as uc
    from paper_2609_32831_gb300.engine import RequestCache

    world, rank, local = rank_env()
    device = torch.device(f"cuda:{local}")
    torch.cuda.set_device(device)
    if world > 1:
        dist.init_process_group("nccl", device_id=device)

    def barrier():
        if world > 1:
            dist.barrier()

    D = args.decode_steps or wl.decode_steps
    stream = []
    if args.stream_evict:
        from paper_2609_32831_gb300.engine import StreamEvict
        budget, window, interval = (int(x) for x in args.stream_evict.split(":"))
        stream = [StreamEvict("gen", budget, window, interval)]
    cache = RequestCache(make_types(wl), wl.layers, wl.batch, device, rho=wl.retention or 0.2,
                         gen_capacity=D, stream_evict=stream)
    cache.calibrate(calibration_examples(wl, device))
    K, V, Qw, Qd, Kn, Vn = gen_inputs(wl, device, D, rank)
    torch.cuda.synchronize()

    graphed = args.decode_graph and not stream   # re-eviction changes the layout between steps

    def step(att_ms=None, events=None):
        cache.prefill(K, V, Qw)
        if not graphed:
            for t in range(D):
                cache.decode_step(Qd[t], Kn[t], Vn[t], events=None if events is None else events[t])
            return
        # frozen layout: the decode step replays a captured graph (two copies
        # in turn; the previous step's attention times are read meanwhile)
        if cache.graph is None:   # attention timed on two of the layers (few graph nodes)
            cache.capture_decode(events=True, copies=2, event_layers=(0, wl.layers // 2), programmatic=args.pdl)
        for t in range(D):
            cache.decode_step_graph(Qd[t], Kn[t], Vn[t], copy=t % 2)
            if att_ms is not None and t >= 1:
                att_ms.extend(cache.graph_attention_ms((t - 1) % 2))
        if att_ms is not None:
            att_ms.extend(cache.graph_attention_ms((D - 1) % 2))

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()

    # attention-launch timing inside the timed steps
    ev = None if graphed else [[[(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                                 for _ in range(wl.layers)] for _ in range(D)] for _ in range(args.steps)]
    att_ms: List[float] = []
    try:
        uuid = str(torch.cuda.get_device_properties(device).uuid)
        gpu_id = uuid if uuid.startswith("GPU-") else "GPU-" + uuid
    except Exception:
        gpu_id = str(local)
    clocks = ClockSampler(gpu_id)
    n_launch0 = uc.launch_count()
    barrier()
    torch.cuda.synchronize()
    clocks.start()
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    t_start.record()
    for s in range(args.steps):
        step(att_ms, None if ev is None else ev[s])
    t_end.record()
    torch.cuda.synchronize()
    clk = clocks.stop()
    barrier()
    launches = uc.launch_count() - n_launch0
    if graphed:  # kernels replayed from the captured decode step
        launches += args.steps * D * cache.graph_kernels
    ms = max_over_ranks(t_start.elapsed_time(t_end) / args.steps, world, device)
    value = whole_job_rate(wl.batch * D, world, ms)

    # roofline of the attention kernel: algorithmic bytes / event time
    if ev is not None:
        att_ms = [s_[0].elapsed_time(s_[1]) for st in ev for row in st for s_ in row]
    att_avg_ms = sum(att_ms) / len(att_ms)
    layer_bytes = [cache.cache_bytes(l, include_generated=False) for l in range(wl.layers)]
    per_launch_cache = sum(layer_bytes) / wl.layers
    gen_avg = (D + 1) / 2 * 512 * 4 * wl.batch            # generated tokens read on average
    qo_bytes = 2 * wl.batch * 28 * 128 * 2                 # Q in, O out (bf16)
    alg_bytes = per_launch_cache + gen_avg + qo_bytes
    peak, peak_kind = _peaks()
    achieved = alg_bytes / (att_avg_ms / 1000.0) / 1e9
    ratio = profiled_traffic_ratio()
    traffic = None if ratio is None else ratio * alg_bytes
    decode_ms = sum(att_ms) / args.steps

    result = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "fp16/bf16 MMA on int2/int4 codes and bf16 rows, fp32 accumulate", "data": "synthetic",
        "config": workload_config(wl, D, {k: ("evict" if p == 0 else "quant") for k, p in cache.policy.items()}),
        "realized": {"concentration": cache.concentration,
                     "compression_ratio": cache.full_bytes() / max(1, cache.stored_bytes())},
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak, "traffic": traffic, "kernel": "uc::attend_kernel",
                     "bytes_per_launch": alg_bytes, "avg_launch_us": att_avg_ms * 1000.0,
                     "peak_source": peak_kind},
        "attention_ms_per_step": decode_ms,
        "decode": "CUDA graph of the 28-layer step (frozen layout), replayed per token" if graphed
                  else "eager launches",
        **({"stream_evict": {"type": "generated tokens", "budget": stream[0].budget, "window": stream[0].window,
                             "interval": stream[0].interval, "evictions_per_step": cache.evictions}}
           if stream else {}),
        "gpu_launches": int(launches),
        "clocks": clk,
    }

    # end to end through the public API: inputs from pinned host memory
    if not args.no_e2e:
        result["e2e"] = e2e(args, wl, cache, (K, V, Qw, Qd, Kn, Vn), device, world)
    evicts = any(sp.kind in ("evict", "evict_quant") for sp in wl.segments) or any(
        p == 0 for p in cache.policy.values())
    if rank == 0 and not args.no_eviction_path and wl.decode_steps > 0 and not evicts:
        # the workload's own steps run no eviction kernel: time them on one layer
        try:
            result["eviction_path"] = eviction_path(device)
        except Exception as e:  # reported, never fatal to the bench line
            result["eviction_path"] = {"error": str(e)[:200]}
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        pols = {k: ("evict" if p == 0 else "quant") for k, p in cache.policy.items()}
        # a bounded sample: 32 decode steps at 32K context and below, fewer
        # beyond (the per-step oracle cost grows with the context)
        result["cpu_baseline"] = cpu_baseline(wl, pols, decode_steps=min(32, max(8, 32 * 32768 // wl.n_ctx)))
    if rank == 0:
        print(json.dumps(result), flush=True)
    if world > 1:
        dist.destroy_process_group()


def e2e(args, wl, cache, dev_inputs, device, world):
    """Whole steps through the public API with every step's inputs copied
    from pinned host memory and the last layer's outputs read back. Two
    device input sets alternate: the next step's copy runs on separate copy
    streams while the current step computes, so only the first copy of the
    timed run is exposed (a serving loop prefetching its next batch)."""
    import torch
    import torch.distributed as dist
    sets = [[torch.empty_like(t) for t in dev_inputs] for _ in range(2)]
    stage = HostStaging(list(dev_inputs), sets, args.copy_streams)
    h2d = stage.bytes
    D = dev_inputs[3].shape[0]
    L = wl.layers
    out_last = torch.empty((D, wl.batch, 28, 1, 128), dtype=torch.bfloat16, device=device)
    out_host = torch.empty(out_last.shape, dtype=out_last.dtype, pin_memory=True)
    d2h = out_last.numel() * out_last.element_size()
    main = torch.cuda.current_stream()
    graphed = args.decode_graph and not cache.stream_evict

    def step(s, last):
        i = s % 2
        stage.wait(i, main)
        if not last:
            stage.issue(1 - i)
        K, V, Qw, Qd, Kn, Vn = sets[i]
        cache.prefill(K, V, Qw)
        if graphed and cache.graph is None:   # recaptured only when the layout changed
            cache.capture_decode(events=True, copies=2, event_layers=(0, wl.layers // 2), programmatic=args.pdl)
        for t in range(D):
            if graphed:
                outs = cache.decode_step_graph(Qd[t], Kn[t], Vn[t], copy=t % 2)
            else:
                outs = cache.decode_step(Qd[t], Kn[t], Vn[t])
            out_last[t].copy_(outs[L - 1])
        out_host.copy_(out_last, non_blocking=True)
        stage.release(i, main)

    for i in range(2):          # warm both input sets (each layout's decode graph is captured here)
        stage.issue(i)
        step(i, True)
    torch.cuda.synchronize()
    stage.reset()
    rate = stage.rate_gbps()
    torch.cuda.synchronize()
    stage.reset()
    n = max(1, args.steps)
    if world > 1:
        dist.barrier()
    a = torch.cuda.Event(enable_timing=True)
    b = torch.cuda.Event(enable_timing=True)
    a.record()
    stage.issue(0)
    for s_ in range(n):
        step(s_, s_ == n - 1)
    b.record()
    torch.cuda.synchronize()
    ms = max_over_ranks(a.elapsed_time(b) / n, world, device)
    return {"value": whole_job_rate(wl.batch * D, world, ms), "unit": UNIT, "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h, "ms_per_step": ms, "steps": n, "host_pinned": stage.pinned,
            "h2d_GBps": rate, "copy_streams": len(stage.streams),
            "copies": "every step's inputs H2D from pinned host memory; the next step's copy overlaps "
                      "this step's compute on separate copy streams (two device input sets)"}


if __name__ == "__main__":
    main()
