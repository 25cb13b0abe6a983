"""GB300-native (sm_103a) evaluation of the joint attention-block loss L_JAB and its STE/LSQ scale
gradient, behind the C ABI of include/jab.h.

This package is a thin ctypes binding: it marshals torch tensors (device memory) and CUDA streams
into the C entry points of libjab.so, whose kernels do every step of the computation. Importing a
function that needs the library fails loudly when libjab.so has not been built; there is no
Python or CPU fallback.
"""
from .binding import (  # noqa: F401
    BlockDesc, JabError, JAB_OK, desc_from_shape, lib, lib_path, jab_workspace_size,
    jab_reference_forward, jab_loss_forward, jab_loss_forward_noalloc, jab_loss_backward_scales,
    jab_loss_backward_weights, jab_allocate_bits, jab_quantize,
    jab_init_scales, jab_get_device_status, jab_status_string, Workspace, jab_timing_enable,
    jab_timing_reset, jab_timing_read, jab_selftest_wait_timeout, jab_prepare_x,
    jab_loss_backward_scales_prepared, jab_flip_rate, jab_reference_projection,
    jab_loss_forward_kl, jab_hutchinson_trace, jab_omega_scores, jab_rademacher_probes,
    jab_set_deterministic, jab_selftest_bounds_check, jab_loss_backward_scales_kl,
)
