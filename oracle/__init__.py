"""CPU oracle for the DFlow round (TEST INFRASTRUCTURE ONLY).

Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline leg may import
or run anything in this package.  The CUDA path never calls it and shares no
code with it; the two meet only in the seeded input generators of `synth`.

See oracle/dflow_oracle.py for what is computed and which passage of the paper
each function follows.
"""
from .dflow_oracle import (  # noqa: F401
    Oracle, State, RoundOut, rmsnorm, layernorm, silu, rope, attend, argmax_rows, top2_gap,
    log_softmax, gumbel_argmax, speculative_sample,
)
