"""CPU oracle of the streaming action-decode step (test infrastructure only).

Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline legs import it;
the CUDA library never does.
"""
from .flashvla_oracle import *  # noqa: F401,F403
