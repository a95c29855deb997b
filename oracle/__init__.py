"""fp64 CPU oracle (test infrastructure).

Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline and
reference legs may import this package; the product path never does.
"""
from .frt_oracle import (OracleStream, attention, bf16_round, rope3d,  # noqa: F401
                         rope_angles, token_positions, window_index)
