"""GB300-native ECASQ: the approximate-DP hot path of Entropy-Constrained
Adaptive Stochastic Quantization (arxiv 2608.18147) as hand-written CUDA for
sm_103a behind a C ABI (include/ecasq.h), with this thin Python binding.

The binding functions carry the C entry points' names (ecasq_solve,
ecasq_dp_pass, ecasq_refine, ecasq_quantize, ecasq_solve_batched, ...).
There is no CPU fallback: without libecasq.so and a GPU every call raises.
"""
from . import workloads
from .native import (DP_REFERENCE, EXACT_S, EXACT_TABLES, NO_REFINE_GUARD, ONE_PART_PUBLISH, RESIDENT_COSTS,
                     STREAMED_COSTS, TEST_SELF_SEED, TEST_STALL, UNSEEDED_SEARCH,
                     TIME_KERNELS,
                     EcasqError,
                     ecasq_dp_linear, ecasq_dp_pass, ecasq_dp_tables, ecasq_evaluate, ecasq_kernel_launches, ecasq_opt_dp, ecasq_prepare,
                     ecasq_quantize, ecasq_quantize_noalloc, ecasq_quantize_timeshare, ecasq_refine, ecasq_solve,
                     ecasq_solve_batched, ecasq_solve_grid, ecasq_solve_timeshare, ecasq_workspace_size,
                     ecasq_workspace_size_flags, lib, uniform_grid, workspace)

__all__ = ["workloads", "ecasq_solve", "ecasq_solve_grid", "ecasq_solve_timeshare", "ecasq_solve_batched",
           "ecasq_dp_pass", "ecasq_dp_tables", "ecasq_dp_linear", "ecasq_opt_dp", "ecasq_refine", "ecasq_evaluate", "ecasq_quantize",
           "ecasq_quantize_noalloc", "ecasq_quantize_timeshare", "ecasq_prepare", "ecasq_workspace_size",
           "ecasq_workspace_size_flags", "ecasq_kernel_launches", "workspace", "uniform_grid", "lib", "EcasqError",
           "EXACT_S", "EXACT_TABLES", "RESIDENT_COSTS", "NO_REFINE_GUARD", "DP_REFERENCE", "TIME_KERNELS", "TEST_STALL", "STREAMED_COSTS", "ONE_PART_PUBLISH",
           "UNSEEDED_SEARCH", "TEST_SELF_SEED"]
