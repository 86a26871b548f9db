"""fp64 CPU oracle of the SAO loss head (test infrastructure only; see sao_oracle)."""
from .sao_oracle import *  # noqa: F401,F403
