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
#include <atomic>
#include <cstdint>
#include <mutex>

#include "tt_device.cuh"
#include "tt_launch.h"

namespace {

// The scratch of every call on a device; the device holds it from the moment
// the library's module is loaded there until the process exits.
static __device__ __align__(256) unsigned char tt_noalloc_scratch[TT_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;

// Device address of the scratch array per device, looked up once per device
// (under its once-flag) with that device current: host code cannot use the
// array's name as a device address, it is only a host-side stand-in.
std::once_flag g_once[kMaxDevices];
std::atomic<void*> g_scratch_ptr[kMaxDevices];
cudaError_t g_setup_error[kMaxDevices];

void look_up_scratch(int dev) {
  void* ptr = nullptr;
  const cudaError_t e = cudaGetSymbolAddress(&ptr, tt_noalloc_scratch);
  g_setup_error[dev] = e == cudaSuccess && ptr == nullptr ? cudaErrorInvalidSymbol : e;
  if (g_setup_error[dev] == cudaSuccess) g_scratch_ptr[dev].store(ptr, std::memory_order_release);
}

}  // namespace

extern "C" tt_status tt_step_noalloc(const tt_batch* batch, const tt_vocab* vd,
                                     const tt_vocab* vt, const tt_logits* draft,
                                     const float* draft_probs, const tt_logits* target,
                                     const tt_params* prm, const tt_step_out* out,
                                     void* stream) {
  // every check of tt_step first, on the host: a refused call queues nothing
  size_t need = 0;
  const tt_status chk =
      tt::step_check(batch, vd, vt, draft, draft_probs, target, prm, out, &need);
  if (chk != TT_OK) return chk;
  if (batch->B == 0) return TT_OK;
  if (need == 0 || need > size_t(TT_NOALLOC_SCRATCH_BYTES)) return TT_ERR_UNSUPPORTED;

  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return tt::record_cuda_error(e);
  if (dev < 0 || dev >= kMaxDevices) return TT_ERR_UNSUPPORTED;
  std::call_once(g_once[dev], look_up_scratch, dev);  // set-up, once per device
  void* ws = g_scratch_ptr[dev].load(std::memory_order_acquire);
  if (ws == nullptr) return tt::record_cuda_error(g_setup_error[dev]);
  // nothing in the scratch needs to start at zero: every value is written
  // before it is read, and the row pass's error report carries the call's tag
  return tt_step(batch, vd, vt, draft, draft_probs, target, prm, ws,
                 size_t(TT_NOALLOC_SCRATCH_BYTES), out, stream);
}
