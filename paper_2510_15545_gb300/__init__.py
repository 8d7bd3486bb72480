"""TokenTiming verification hot path on one GB300 (sm_103a): DTW alignment of
draft and proxy target tokens, probability transfer and lossless speculative
verification with residual resampling (arXiv 2510.15545), behind the C ABI of
include/tt.h, plus the re-encoding of the draft string into target tokens with
its Lemma-1 check and the delta-pos histogram of the alignment paths. The names
below are the library's entry points; the library is loaded on first use and a
missing build raises."""
from .binding import (AlignCall, Batch, Params, StepCall, TTError, VocabTable, device_inputs, load,
                      step_outputs, tt_align, tt_consistency, tt_dpos_hist, tt_encode,
                      tt_encode_workspace_bytes, tt_status_string, tt_step, tt_step_noalloc,
                      tt_transfer, tt_verify, tt_verify_sharded, tt_version, tt_workspace_bytes, vocab_index,
                      workspace)

__all__ = ["AlignCall", "Batch", "Params", "StepCall", "TTError", "VocabTable", "device_inputs", "load",
           "step_outputs", "tt_align", "tt_consistency", "tt_dpos_hist", "tt_encode",
           "tt_encode_workspace_bytes", "tt_status_string", "tt_step", "tt_step_noalloc",
           "tt_transfer", "tt_verify", "tt_verify_sharded", "tt_version", "tt_workspace_bytes", "vocab_index",
           "workspace"]
