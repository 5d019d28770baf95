"""fp64 CPU oracle of MemDecay (test infrastructure only).

Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline / reference
legs may import this package; the product path never does."""
from .memdecay_oracle import *  # noqa: F401,F403
from .memdecay_oracle import Oracle, OracleConfig  # noqa: F401
