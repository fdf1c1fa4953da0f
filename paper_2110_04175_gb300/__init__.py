"""GB300-native RelaySum step (RelaySGD, arXiv 2110.04175, Algorithm 1).

A thin Python binding over the C ABI of ``librelaysum.so`` (declared in
``include/relaysum.h``): the functions here have the C names and only
marshal arguments -- torch tensors become device pointers, a torch stream
becomes a ``cudaStream_t`` -- while every step of the method runs in the
library's CUDA kernels.  There is no CPU fallback: if the library has not
been built, the first call raises.

``RelayRun`` is a convenience owner of the device buffers of one run
(allocated with torch) that swaps the double-buffered messages between
steps.
"""
from __future__ import annotations

from ._native import (RELAY_EINVAL, RELAY_ECUDA, RELAY_ENOMEM, RELAY_ENOTTREE, RELAY_EUNSUPPORTED,
                      RELAY_ALGO_DME, RELAY_ALGO_GRAD, RELAY_ALGO_RELAYSGD, RELAY_KERNEL_AUTO,
                      RELAY_KERNEL_FUSED, RELAY_KERNEL_NODES, RELAY_KERNEL_WALK, RELAY_MAX_N, RELAY_OK,
                      RELAY_OPT_ADAM, RELAY_OPT_NESTEROV, RELAY_OPT_SGD, RELAY_HOST_FULL_OUTPUT,
                      RelayError, RelayHandle, RelayHostPlan, RelayRun, library_path,
                      relay_host_bytes, relay_host_plan_create, relay_host_staging_bytes, relay_step_host,
                      relay_steps_host,
                      relay_create, relay_destroy, relay_edges, relay_error_string,
                      relay_fill_objective, relay_init, relay_ld, relay_metrics,
                      relay_metrics_static, relay_metrics_workspace, relay_nbar, relay_num_edges,
                      relay_program, relay_set_coord_offset, relay_set_objective,
                      relay_set_algorithm, relay_set_local_optimizer, relay_set_lost_messages,
                      relay_set_objective_generated, relay_get_kernel,
                      relay_get_steps_kernel,
                      relay_set_kernel, relay_set_rebuild_mode, relay_set_strides,
                      relay_set_received_sums, relay_message_rows, relay_step, relay_step_windows,
                      relay_step_counts, relay_step_models, relay_steps)

from .lr_correction import lr_correction  # noqa: E402

__all__ = [
    "RELAY_OK", "RELAY_EINVAL", "RELAY_ENOTTREE", "RELAY_ECUDA", "RELAY_ENOMEM",
    "RELAY_EUNSUPPORTED", "RELAY_MAX_N", "RELAY_OPT_SGD", "RELAY_OPT_NESTEROV", "RELAY_OPT_ADAM",
    "RELAY_ALGO_RELAYSGD", "RELAY_ALGO_GRAD", "RELAY_ALGO_DME", "RELAY_KERNEL_AUTO",
    "RELAY_KERNEL_WALK", "RELAY_KERNEL_NODES", "RELAY_KERNEL_FUSED", "RELAY_HOST_FULL_OUTPUT", "RelayError",
    "RelayHandle", "RelayHostPlan", "RelayRun", "library_path",
    "relay_host_staging_bytes", "relay_host_plan_create", "relay_host_bytes", "relay_step_host", "relay_steps_host",
    "relay_create", "relay_destroy", "relay_ld", "relay_num_edges", "relay_edges",
    "relay_set_rebuild_mode", "relay_set_kernel", "relay_get_kernel", "relay_get_steps_kernel",
    "relay_set_strides", "relay_set_local_optimizer", "relay_set_received_sums", "relay_message_rows",
    "relay_set_lost_messages", "relay_set_algorithm", "relay_set_coord_offset", "relay_set_objective",
    "relay_set_objective_generated", "relay_fill_objective", "relay_init", "relay_step_counts",
    "relay_step_models", "relay_step", "relay_step_windows", "relay_steps",
    "relay_nbar", "relay_program", "relay_metrics", "relay_metrics_workspace",
    "relay_metrics_static",
    "relay_error_string", "lr_correction",
]
