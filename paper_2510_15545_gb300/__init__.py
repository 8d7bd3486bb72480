"""TokenTiming verification hot path on one GB300 (sm_103a): DTW alignment of
draft and proxy target tokens, probability transfer and lossless speculative
verification with residual resampling (arXiv 2510.15545), behind the C ABI of
include/tt.h. The names below are the library's entry points; the library is
loaded on first use and a missing build raises."""
from .binding import (Batch, Params, StepCall, TTError, VocabTable, device_inputs, load,
                      step_outputs, tt_align, tt_status_string, tt_step, tt_step_noalloc,
                      tt_transfer, tt_verify, tt_version, tt_workspace_bytes, workspace)

__all__ = ["Batch", "Params", "StepCall", "TTError", "VocabTable", "device_inputs", "load",
           "step_outputs", "tt_align", "tt_status_string", "tt_step", "tt_step_noalloc",
           "tt_transfer", "tt_verify", "tt_version", "tt_workspace_bytes", "workspace"]
