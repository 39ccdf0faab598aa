"""fp64 CPU oracle of the VaSE eviction step -- test infrastructure only (see vase_oracle)."""
from .vase_oracle import *  # noqa: F401,F403
