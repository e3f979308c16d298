"""GB300-native UniCache compressed-KV hot path (arxiv 2609.32831).

The compute lives in ``lib/libunicache.so`` (CUDA for sm_103a, C ABI in
``include/unicache.h``); this package is its Python binding. Importing the
package does not load the library; the first call does, and fails loudly if
the library has not been built.
"""
from .api import (KIND_EVICT, KIND_EVICT_QUANT, KIND_FULL, KIND_QUANT, POLICY_EVICT,
                  POLICY_PROTECTED, POLICY_QUANT, Segment, SegmentTable, UniCacheError, Workspace,
                  accumulate_scores, allocate_budget, append, append_next, attend, attend_batch, attend_plan,
                  attend_workspace_size,
                  attention_mass, calibrate_policy, compress_budget, compress_segment, concentration, keep_count,
                  launch_count, OwnedSegment,
                  plan_batch, recompress_segment, retention_schedule, retention_step, score_accumulate,
                  segment_mass, set_dense_serial_pv, set_programmatic_launch, set_wait_limit,
                  debug_withhold_tile, version)

__all__ = [
    "Segment", "SegmentTable", "Workspace", "UniCacheError", "accumulate_scores", "allocate_budget", "append", "append_next",
    "attend", "attend_batch", "attend_plan", "attend_workspace_size", "attention_mass", "calibrate_policy",
    "compress_budget", "compress_segment", "OwnedSegment",
    "concentration", "keep_count", "launch_count", "plan_batch", "recompress_segment", "retention_schedule",
    "retention_step", "score_accumulate",
    "segment_mass", "set_dense_serial_pv", "set_programmatic_launch", "set_wait_limit", "debug_withhold_tile", "version", "KIND_FULL", "KIND_EVICT", "KIND_QUANT",
    "KIND_EVICT_QUANT", "POLICY_EVICT", "POLICY_QUANT", "POLICY_PROTECTED",
]
