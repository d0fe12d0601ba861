// Entropy-bounded select (arXiv 2509.04185, Eq. 3; Algorithm 3 "unmask").
//
// One warp per sequence, one lane per block position (k <= 32).  The lanes
// sort their (entropy, position) keys ascending with a bitonic network of
// register shuffles, take an inclusive prefix sum of the sorted entropies,
// and accept the longest prefix of ranks whose preceding sum S_{j-1} is
// <= gamma (rank 1 always).  Accepted positions get their sampled token
// committed into the block buffer and their masked flag cleared.
#include "sbd_internal.cuh"

namespace {

using namespace sbd_dev;

constexpr int kWarpsPerBlock = 4;

__device__ __forceinline__ bool key_less(float ha, int ia, float hb, int ib) {
  return ha < hb || (ha == hb && ia < ib);
}

__global__ void __launch_bounds__(32 * kWarpsPerBlock)
eb_select_kernel(int B, int k, const float* __restrict__ entropy,
                 const int32_t* __restrict__ token, float gamma, uint8_t* __restrict__ masked,
                 int32_t* __restrict__ block_tokens, int32_t* __restrict__ n_unmasked) {
  grid_dependency_wait();
  grid_dependents_launch();
  const int lane = threadIdx.x & 31;
  const int b = blockIdx.x * kWarpsPerBlock + (threadIdx.x >> 5);
  if (b >= B) return;

  const bool in_block = lane < k;
  const bool is_masked = in_block && masked[(size_t)b * k + lane] != 0;
  float h = INFINITY;
  if (is_masked) {
    h = entropy[(size_t)b * k + lane];
    if (isnan(h)) h = INFINITY;              // a NaN sorts last among masked
  }
  // Unmasked lanes sort after every masked one (position key offset by 32).
  int key_pos = is_masked ? lane : lane + 32;

  // Bitonic sort of 32 (h, key_pos) pairs, ascending.
#pragma unroll
  for (int size = 2; size <= 32; size <<= 1) {
#pragma unroll
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      const float oh = __shfl_xor_sync(0xffffffffu, h, stride);
      const int op = __shfl_xor_sync(0xffffffffu, key_pos, stride);
      const bool ascending = (lane & size) == 0 || size == 32;
      const bool lower = (lane & stride) == 0;
      const bool other_less = key_less(oh, op, h, key_pos);
      const bool take_other = (lower == ascending) ? other_less : !other_less;
      if (take_other) {
        h = oh;
        key_pos = op;
      }
    }
  }

  const int n_masked = __popc(__ballot_sync(0xffffffffu, is_masked));
  // Inclusive prefix sum of the sorted masked entropies (fp32).
  float incl = (lane < n_masked) ? h : 0.f;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const float t = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += t;
  }
  float excl = __shfl_up_sync(0xffffffffu, incl, 1);   // S_{j-1} for rank j = lane + 1
  if (lane == 0) excl = 0.f;
  // Rank j >= 2 is refused when S_{j-1} > gamma (or is NaN); the accepted
  // count is the first refused rank, so the accepted set is a prefix.
  const bool refused = lane >= 1 && lane < n_masked && !(excl <= gamma);
  const unsigned refused_bits = __ballot_sync(0xffffffffu, refused);
  int s = refused_bits ? (__ffs(refused_bits) - 1) : n_masked;
  if (s > n_masked) s = n_masked;

  if (lane < s) {
    const int pos = key_pos;                       // original block position
    const size_t o = (size_t)b * k + pos;
    block_tokens[o] = token[o];
    masked[o] = 0;
  }
  if (lane == 0 && n_unmasked) n_unmasked[b] = s;
}

}  // namespace

namespace sbd {

sbd_status eb_launch(int B, int k, const float* entropy, const int32_t* token, float gamma,
                     uint8_t* masked, int32_t* block_tokens, int32_t* n_unmasked,
                     cudaStream_t st) {
  if (B == 0) return SBD_OK;
  const int blocks = (B + kWarpsPerBlock - 1) / kWarpsPerBlock;
  void* args[] = {(void*)&B,      (void*)&k,      (void*)&entropy,      (void*)&token,
                  (void*)&gamma,  (void*)&masked, (void*)&block_tokens, (void*)&n_unmasked};
  return launch_pdl((const void*)eb_select_kernel, dim3(blocks), dim3(32 * kWarpsPerBlock), 0, st,
                    args, "eb_select_kernel launch");
}

}  // namespace sbd
