"""fp64 oracle of the classify path (test infrastructure only; see sp_oracle)."""
from .sp_oracle import (Layer, attention, attention_probs, attention_step, classify, rms_norm,
                        rope, sequence_kv, silu, softmax_rows, to_f64)

__all__ = ["Layer", "attention", "attention_probs", "attention_step", "classify", "rms_norm",
           "rope", "sequence_kv", "silu", "softmax_rows", "to_f64"]
