"""Seeded synthetic inputs for the gradient-coding hot path.

This package is the ONLY thing the CUDA path and the fp64 oracle share: it
produces data (features X, labels y, the parameter vector w, the PS matrix R,
chunk gradients for the decode-only workload, and straggler state vectors psi)
and holds none of the protocol's arithmetic (no assignment, no coefficient
solve, no encode or decode).  Random numbers the protocol itself draws (the
Gaussian matrix R of Sec. II) are produced here and handed to both sides.
"""
from .configs import CONFIGS, Config, get  # noqa: F401
from .gen import (  # noqa: F401
    make_R,
    make_w,
    make_data,
    make_chunk_grads,
    make_patterns,
    all_patterns,
    random_regular_graph,
    second_eigenvalue,
    random_order,
    make_worker_times,
)
