"""fp64 CPU oracle (test infrastructure only; see pad_oracle.py)."""
from .pad_oracle import (bf16_to_f64, event_mask, video_attention, decode_step, event_rows,
                         lse_merge, simulate_append, bf16_round, rope_rotate, rope_bits,
                         rotated_workload, ground_segment_scores, ground_salient,
                         attention_aggregate, prefill_mask, prefill_attention, OK,
                         OUT_OF_PAGES, INVALID)

__all__ = ["bf16_to_f64", "event_mask", "video_attention", "decode_step", "event_rows",
           "lse_merge", "simulate_append", "bf16_round", "rope_rotate", "rope_bits",
           "rotated_workload", "ground_segment_scores", "ground_salient", "attention_aggregate",
           "prefill_mask", "prefill_attention", "OK", "OUT_OF_PAGES", "INVALID"]
