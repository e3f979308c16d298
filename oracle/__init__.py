"""CPU oracle for UniCache's compressed-KV hot path (arxiv 2609.32831).

TEST INFRASTRUCTURE ONLY. This package is a plain, slow, readable restatement
of what the paper defines, used to check the CUDA path. Only ``tests/``,
``__graft_entry__.smoke()`` and the ``cpu_baseline`` / reference leg of
``bench.py`` may import it. The product path (the C-ABI library and its Python
binding) never imports, links or calls anything here, and nothing here imports
the product package. The two share no code; inputs come from ``synth``.

Precision: floating point is fp64 except where the method fixes another
precision. Group quantization is specified in fp32 round-to-nearest-even with
fp16 storage of scale and zero-point, so ``quant`` emulates exactly that with
numpy float32 / float16 arithmetic.

Modules and the passages they follow:

* ``scores``    — observation-window attention mass per token (§3.3 Eq. 1's
                  P, GQA aggregation of App. E "Batched GQA token selection").
* ``policy``    — concentration and policy choice (App. B), Eq. 2 budget
                  allocation with redistribution (§3.3), Eq. 3 temporal
                  retention schedule (§3.3), budget -> (keep, bits) mapping.
* ``select``    — per-KV-head heavy-hitter (+ recent) top-k (App. E).
* ``quant``     — int4 / int2 group quantization, keys per channel, values
                  per token, with a bf16 residual tail (App. E storage).
* ``segment``   — compress one segment (evict / quantize / both) and append
                  decode tokens (§3.4, App. E).
* ``attention`` — one shared softmax over all segments, with log-sum-exp and
                  per-segment attention mass (App. E, Eq. 1).

Parity status of each function is stated in its module docstring. The only
unpinned item is whether Gaussian synthetic attention resembles a trained
model's (no model weights or datasets exist here): "parity unpinned" for
workload realism, not for any function below.
"""
from . import scores, policy, select, quant, segment, attention  # noqa: F401
