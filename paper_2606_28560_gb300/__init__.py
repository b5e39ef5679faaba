"""GB300 (sm_103a) library for depth-staggered scaled-Fibonacci sparse
attention (arXiv 2606.28560).  The compute path is the CUDA library built
from ``csrc/`` and exposed through the C ABI of ``include/fibattn.h``; this
package only marshals arguments to it.
"""
from .binding import (FibattnError, alpha_schedule, base, bwd, bwd_workspace_bytes, fwd,  # noqa: F401
                      fwd_workspace_bytes, lib, library_path, rung_params)

__all__ = ["fwd", "bwd", "fwd_workspace_bytes", "bwd_workspace_bytes", "rung_params", "base",
           "alpha_schedule", "lib", "library_path", "FibattnError"]
