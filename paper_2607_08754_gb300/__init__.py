"""GB300 (sm_103a) implementation of the SLORR regularizer hot path.

The compute lives in ``libslorr.so`` (CUDA kernels behind the C ABI of
``include/slorr.h``); ``paper_2607_08754_gb300.slorr`` is its ctypes binding.
"""

from .slorr import (  # noqa: F401
    Pipeline,
    Regularizer,
    SlorrError,
    load_library,
    slorr_create,
    slorr_cushion_ratio,
    slorr_default_options,
    slorr_destroy,
    slorr_executed_flops,
    slorr_flops,
    slorr_frob_sq_noalloc,
    slorr_get_coefficients,
    slorr_get_status,
    slorr_iterate_view,
    slorr_partition,
    slorr_pe_coefficients,
    slorr_pipeline_create,
    slorr_pipeline_destroy,
    slorr_pipeline_forward_backward,
    slorr_pipeline_get_status,
    slorr_pipeline_workspace_size,
    slorr_reg_descent_step,
    slorr_reg_forward_backward,
    slorr_reset_workspace,
    slorr_read_timing,
    slorr_run_steps,
    slorr_set_timing,
    slorr_status_string,
    slorr_workspace_size,
)
