"""fp64 CPU oracle of the EAT MoE layer -- test infrastructure only (see eat_oracle.py)."""
from .eat_oracle import *  # noqa: F401,F403
