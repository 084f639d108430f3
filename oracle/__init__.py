"""fp64 CPU oracle of the JET candidate-scoring step (test infrastructure only)."""
from .jet_oracle import *  # noqa: F401,F403
from .jet_oracle import (ARGMAX, BINARY, ORDINAL, visible_keys, gated_delta_step,  # noqa: F401
                         gated_linear_step, row_logsumexp)
