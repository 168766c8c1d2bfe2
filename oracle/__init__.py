"""fp64 CPU oracle of the TGV-KV eviction step -- test infrastructure only.

Importable by the tests, ``__graft_entry__.smoke()`` and the CPU-baseline arm
of ``bench.py``; never by the product path.
"""
from .tgvkv_oracle import (  # noqa: F401
    widen_bf16, causal_text_attention, twr_scores_tvb_stat, vision_budget_total,
    tvb_budgets, tpr_select, compact, compacted_kv_bytes, evict,
    text_scores_and_weights, all_budget_total, sink_positions, tpr_select_general,
    decode_attention, tt_statistic, tv_statistic_per_head, head_budget,
    prefill_attention, row_statistics,
)
