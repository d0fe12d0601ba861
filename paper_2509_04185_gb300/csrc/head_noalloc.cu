// sbd_head_entropy_sample_noalloc: the LM-head call with its scratch in a
// fixed device array owned by the library instead of a caller workspace.
//
// Some callers cannot allocate device memory: a host framework that owns the
// whole device pool (a cudaMalloc would fail, or escape its accounting), a
// latency-critical loop that cannot afford the device synchronisation a
// cudaMalloc/cudaFree may imply, or a plug-in that has no allocator to borrow
// a workspace from.  They call this variant; it runs exactly the kernels of
// sbd_head_entropy_sample, with the workspace pointer set to the array below.
#include <mutex>

#include "sbd_internal.cuh"

namespace {

// The scratch.  Every GPU that loads the library holds these bytes until the
// process exits.  Host code must not pass the symbol itself to a kernel: on
// the host it names a shadow object, not device memory.
static __device__ __align__(256) unsigned char g_head_scratch[SBD_HEAD_NOALLOC_MAX_SCRATCH];

constexpr int kMaxDevices = 64;

struct ScratchTable {
  std::once_flag once[kMaxDevices];
  void* ptr[kMaxDevices] = {nullptr};
  cudaError_t err[kMaxDevices] = {cudaSuccess};
};
ScratchTable& table() {
  static ScratchTable t;
  return t;
}

// Once per device, with that device current: the device address of the array.
void resolve(int dev) {
  void* p = nullptr;
  cudaError_t e = cudaGetSymbolAddress(&p, g_head_scratch);
  table().err[dev] = e;
  table().ptr[dev] = e == cudaSuccess ? p : nullptr;
  if (e != cudaSuccess) cudaGetLastError();
}

}  // namespace

extern "C" sbd_status sbd_head_entropy_sample_noalloc(const sbd_head_desc* desc,
                                                      const void* hidden, const void* w,
                                                      const uint8_t* masked, const float* gumbel,
                                                      float tau, float* entropy, int32_t* token,
                                                      void* stream) {
  // An invalid descriptor reports 0 here and is diagnosed by the call below.
  const size_t need = sbd_head_entropy_sample_workspace_size(desc);
  if (need > (size_t)SBD_HEAD_NOALLOC_MAX_SCRATCH)
    return sbd::fail(SBD_ERR_UNSUPPORTED,
                     "this shape needs %zu bytes of scratch; the no-allocation variant holds "
                     "at most %u (use sbd_head_entropy_sample with a workspace)",
                     need, (unsigned)SBD_HEAD_NOALLOC_MAX_SCRATCH);
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return sbd::cuda_fail(e, "cudaGetDevice");
  if (dev < 0 || dev >= kMaxDevices)
    return sbd::fail(SBD_ERR_UNSUPPORTED, "device ordinal %d >= %d", dev, kMaxDevices);
  std::call_once(table().once[dev], resolve, dev);
  if (!table().ptr[dev])
    return sbd::cuda_fail(table().err[dev], "cudaGetSymbolAddress(no-allocation scratch)");
  return sbd_head_entropy_sample(desc, hidden, w, masked, gumbel, tau, entropy, token,
                                 table().ptr[dev], (size_t)SBD_HEAD_NOALLOC_MAX_SCRATCH, stream);
}
