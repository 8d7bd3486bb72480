// noalloc.cu -- tt_step_noalloc: the fused verification step for callers that
// cannot allocate device memory.
//
// Some callers cannot call cudaMalloc (or any allocating routine) where they
// run a verification step: runtimes whose device memory all belongs to one
// arena, serving loops that must not stall on the allocator, or hosts that
// only hand over input and output buffers. They cannot provide the workspace
// tt_step needs, so this entry point brings its own: a fixed array in the
// library's device image, set up once per device and reused by every call on
// that device.
#include <cstdint>

#include "tt_device.cuh"
#include "tt_launch.h"

namespace {

// The scratch of every call on a device; the device holds it from the moment
// the library's module is loaded there until the process exits.
static __device__ __align__(256) unsigned char tt_noalloc_scratch[TT_NOALLOC_SCRATCH_BYTES];

// Device address of the scratch array per device; host code cannot use the
// array's name as a device address, it is only a host-side stand-in.
void* g_scratch_ptr[64] = {nullptr};

}  // namespace

extern "C" tt_status tt_step_noalloc(const tt_batch* batch, const tt_vocab* vd,
                                     const tt_vocab* vt, const tt_logits* draft,
                                     const float* draft_probs, const tt_logits* target,
                                     const tt_params* prm, const tt_step_out* out,
                                     void* stream) {
  if (!batch || !prm || !target || !out) return TT_ERR_INVALID_ARG;
  if (batch->B < 0 || batch->n_draft < 0 || batch->n_target < 0) return TT_ERR_INVALID_ARG;
  // size check first: nothing touches the GPU before it passes
  const bool from_logits = draft_probs == nullptr || prm->full_q != 0;
  if (from_logits && !draft) return TT_ERR_INVALID_ARG;
  const int V_d = from_logits ? draft->n_cols : 0;
  const size_t need = tt_workspace_bytes_for(batch, V_d, target->n_cols, prm);
  if (need > size_t(TT_NOALLOC_SCRATCH_BYTES)) return TT_ERR_UNSUPPORTED;
  if (batch->B == 0) return TT_OK;

  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return TT_ERR_CUDA;
  if (g_scratch_ptr[dev] == nullptr) {  // set-up, once per device, on that device
    void* ptr = nullptr;
    if (cudaGetSymbolAddress(&ptr, tt_noalloc_scratch) != cudaSuccess || ptr == nullptr)
      return TT_ERR_CUDA;
    g_scratch_ptr[dev] = ptr;
  }
  void* ws = g_scratch_ptr[dev];
  // the row-pass error words must not carry a previous call's flags
  const tt::Workspace lay =
      tt::workspace_layout(ws, batch->B, batch->n_draft, batch->n_target, V_d, target->n_cols);
  if (cudaMemsetAsync(lay.err, 0, 2 * sizeof(int32_t), static_cast<cudaStream_t>(stream)) !=
      cudaSuccess)
    return TT_ERR_CUDA;
  return tt_step(batch, vd, vt, draft, draft_probs, target, prm, ws,
                 size_t(TT_NOALLOC_SCRATCH_BYTES), out, stream);
}
