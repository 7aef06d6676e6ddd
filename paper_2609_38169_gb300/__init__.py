"""STEPQuant decode-step library for one NVIDIA GB300 (sm_103a).

The per-token gated Delta-rule decode step on a low-bit, mixed-precision,
dual-axis-scaled recurrent state (arxiv 2609.38169), as a C-ABI shared library
(`include/stepq.h`, built from `csrc/`) with this thin Python binding.
"""
from .api import *  # noqa: F401,F403
from .api import Config, Plan, CalibStats, calibrate, alloc_pool, version  # noqa: F401
