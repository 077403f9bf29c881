"""CPU oracle for ML^2Tuner batched candidate screening (test infrastructure).

Only the test suite, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  The product library never calls it and
shares no code with it.
"""
from .oracle import (  # noqa: F401
    NODE_DTYPE,
    OP_DTYPE,
    build,
    decode,
    features,
    half_ensemble,
    margins,
    rerank,
    round_half,
    sa_step,
    screen,
    screen_rows,
    sigmoid,
    tau,
    topk,
    tree_leaf,
)
