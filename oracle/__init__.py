"""CPU fp64 oracle (test infrastructure; never imported by the product path)."""
from .cover_oracle import (  # noqa: F401
    route_seeds, view_for_row, attention_row, override_attention_rows, override_attention,
    override_attention_closed_form, override_attention_window, corrected_weights_row, score_rows, topk_select, topk_margin,
    FLAG_SEED, attention_mass, decide_sequence, decide_step, seed_kv_gather, seed_kv_override,
)
