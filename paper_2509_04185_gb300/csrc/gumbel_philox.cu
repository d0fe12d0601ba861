// Counter-based Gumbel noise tensor (the noise of the in-kernel sampler,
// written out): out[r, v] = g(row_ids[r], v) with g as in philox.cuh.  One
// thread per Philox call, i.e. per 4 consecutive vocabulary ids of a row.
#include "philox.cuh"
#include "sbd_internal.cuh"

namespace {

using namespace sbd_dev;

__global__ void __launch_bounds__(256)
gumbel_fill_kernel(const int32_t* __restrict__ row_ids, int V, uint32_t seed_lo,
                   uint32_t seed_hi, uint32_t off_lo, uint32_t off_hi, float* __restrict__ out) {
  grid_dependency_wait();
  grid_dependents_launch();
  const int r = blockIdx.y;
  const int q = blockIdx.x * blockDim.x + threadIdx.x;   // call index = v div 4
  if (q * 4 >= V) return;
  const uint32_t n = (uint32_t)row_ids[r];
  const uint4 x = sbd_philox::philox4x32_10(make_uint4((uint32_t)q, n, off_lo, off_hi), seed_lo,
                                            seed_hi);
  float* o = out + (size_t)r * V + 4 * (size_t)q;
#pragma unroll
  for (int w = 0; w < 4; ++w)
    if (4 * q + w < V) o[w] = sbd_philox::gumbel_of_word(sbd_philox::word_of(x, w));
}

}  // namespace

namespace sbd {

sbd_status gumbel_fill_launch(int n_rows, const int32_t* row_ids, int V, uint64_t seed,
                              uint64_t offset, float* out, cudaStream_t st) {
  if (n_rows == 0 || V == 0) return SBD_OK;
  const int calls = (V + 3) / 4;
  uint32_t s_lo = (uint32_t)seed, s_hi = (uint32_t)(seed >> 32);
  uint32_t o_lo = (uint32_t)offset, o_hi = (uint32_t)(offset >> 32);
  void* args[] = {(void*)&row_ids, (void*)&V,    (void*)&s_lo, (void*)&s_hi,
                  (void*)&o_lo,    (void*)&o_hi, (void*)&out};
  return launch_pdl((const void*)gumbel_fill_kernel, dim3((calls + 255) / 256, n_rows), dim3(256),
                    0, st, args, "gumbel_fill_kernel launch");
}

}  // namespace sbd
