"""RefAdapt-DiT CPU oracle (fp64) — TEST INFRASTRUCTURE.

Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline / reference
legs may import, call or build anything in this package. The product library
(paper_2609_32415_gb300) never imports it and it never imports the product.
Every function cites the passage of the paper it restates; see core.py.

The DiT block around the hot path (output projection, MLP, AdaLN, QK norm,
RoPE, the reference stream's hidden-state cache) is in ``oracle.dit``.

Parity pins: every function here is checked by the `-m "not gpu"` tests in
tests/test_oracle_pins.py and tests/test_oracle_dit_pins.py against brute
force, closed forms, library special cases and invariants; none is "parity
unpinned".
"""
from .core import (REUSE, BOUNDARY, COMPUTE, FULL, ROLES, Gate, adjacent_ref_mass_change, attention_flops,
                   bf16_to_f64, block_attention, closed_loop, default_threads, endpoint_drift, exposure,
                   head_mean_exposure, joint_attention, local_impact, q_change, reuse_score_fraction)

__all__ = ["REUSE", "BOUNDARY", "COMPUTE", "FULL", "ROLES", "Gate", "adjacent_ref_mass_change",
           "attention_flops", "bf16_to_f64", "block_attention", "closed_loop", "default_threads",
           "endpoint_drift", "exposure", "head_mean_exposure", "joint_attention", "local_impact", "q_change",
           "reuse_score_fraction"]
