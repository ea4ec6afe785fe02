"""RefAdapt-DiT hot path on GB300 (sm_103a).

librefadapt.so (C ABI, include/refadapt.h) holds every kernel: joint attention
with the reference mass on tcgen05 tensor cores, the target-Q change
reduction, the first-crossing gate and the reference-cache update, and the
layers of the DiT block around the attention (tcgen05 GEMM with fused
epilogues, modulated LayerNorm, RoPE table). This package is its thin binding
(``api``), Algorithm 1's host loop over the attention (``executor``) and over
a stack of DiT blocks (``dit``), and the seeded synthetic input generator
(``synth``). Calls fail loudly when
the library has not been built; nothing falls back to the CPU.
"""
from . import api, synth  # noqa: F401
from ._lib import (RA_MODE_BOUNDARY, RA_MODE_COMPUTE, RA_MODE_FULL, RA_MODE_REUSE,  # noqa: F401
                   RefAdaptError)
from .dit import DiTExecutor  # noqa: F401
from .executor import Executor, roles_from_joint  # noqa: F401

__version__ = "0.1.0"
