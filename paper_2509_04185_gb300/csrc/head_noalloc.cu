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

// The device address of the array, per device, kept once it was obtained; a
// failed lookup is not kept, so the next call tries again.
struct ScratchTable {
  std::mutex mu;
  void* ptr[kMaxDevices] = {nullptr};
};
ScratchTable& table() {
  static ScratchTable t;
  return t;
}

// With device `dev` current: its address of the array, looked up on first use.
sbd_status scratch_address(int dev, void** out) {
  ScratchTable& t = table();
  std::lock_guard<std::mutex> lock(t.mu);
  if (!t.ptr[dev]) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_head_scratch);
    if (e != cudaSuccess) {
      cudaGetLastError();
      return sbd::cuda_fail(e, "cudaGetSymbolAddress(no-allocation scratch)");
    }
    t.ptr[dev] = p;
  }
  *out = t.ptr[dev];
  return SBD_OK;
}

}  // namespace

extern "C" sbd_status sbd_head_entropy_sample_noalloc(const sbd_head_desc* desc,
                                                      const void* hidden, const void* w,
                                                      const uint8_t* masked, const float* gumbel,
                                                      float tau, float* entropy, int32_t* token,
                                                      void* stream) {
  // An invalid descriptor reports 0 here and is diagnosed by the call below.
  // The floor needs no device, so a shape too large for any device is
  // rejected even before the device is queried.
  size_t need = desc ? sbd::head_workspace_floor(*desc) : 0;
  if (need <= (size_t)SBD_HEAD_NOALLOC_MAX_SCRATCH) {
    const size_t exact = sbd_head_entropy_sample_workspace_size(desc);
    if (exact > need) need = exact;
  }
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
  void* scratch = nullptr;
  const sbd_status st = scratch_address(dev, &scratch);
  if (st != SBD_OK) return st;
  return sbd_head_entropy_sample(desc, hidden, w, masked, gumbel, tau, entropy, token, scratch,
                                 (size_t)SBD_HEAD_NOALLOC_MAX_SCRATCH, stream);
}
