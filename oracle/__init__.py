"""CPU oracle for DARD's per-step hot path (test infrastructure only; see dard_oracle)."""
from .dard_oracle import *  # noqa: F401,F403
from .dard_oracle import (C, LAMBDA_DEFAULT, M, P0_DEFAULT, U, ScoreResult, SeqLayout,
                          attention_mask, confidence, masked_attention, mix_logits,
                          mixing_weight, next_state, position_states, score_block,
                          top2_gap)
