"""CPU oracle of the TADM sampling loop (test infrastructure only)."""
from .tadm_oracle import *  # noqa: F401,F403
from .tadm_oracle import Oracle, confidence, select_topk, unmask_count, layer_cost  # noqa: F401
