"""GB300 (sm_103a) library for depth-staggered scaled-Fibonacci sparse
attention (arXiv 2606.28560).  The compute path is the CUDA library built
from ``csrc/`` and exposed through the C ABI of ``include/fibattn.h``; this
package only marshals arguments to it.
"""
from .binding import (FibattnError, alpha_schedule, base, bwd, bwd_workspace_bytes, check_status,  # noqa: F401
                      coverage, fwd, fwd_workspace_bytes, lib, library_path, residual_bytes, residual_views,
                      residuals_like, rotated_k_like, rung_params, staging_layout, theta_of_alpha_array)
from .autograd import (FibAttention, FibAttentionFunction, alpha_of_theta, attention_stack,  # noqa: F401
                       fib_attention, theta_of_alpha)

__all__ = ["fwd", "bwd", "fwd_workspace_bytes", "bwd_workspace_bytes", "rung_params", "base",
           "alpha_schedule", "lib", "library_path", "FibattnError", "rotated_k_like", "FibAttention",
           "FibAttentionFunction", "fib_attention", "attention_stack", "alpha_of_theta", "theta_of_alpha",
           "coverage", "residual_bytes", "residuals_like", "residual_views", "staging_layout", "check_status",
           "theta_of_alpha_array"]
