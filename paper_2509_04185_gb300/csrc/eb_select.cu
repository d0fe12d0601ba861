// Unmasking step (arXiv 2509.04185, Algorithm 3 "unmask"): the entropy-
// bounded rule of Eq. 3 and the confidence-ordered rules of the Appendix
// "Sampling algorithm" (EB-Sampler with the confidence proxy, Factor).
//
// One warp per sequence, one lane per block position (k <= 32).  The lanes
// sort their (key, position) pairs ascending with a bitonic network of
// register shuffles -- key = entropy for Eq. 3, minus the confidence for the
// confidence-ordered rules -- carrying the entropy along.  Then:
//   Eq. 3           exclusive prefix sum of the sorted entropies; rank j >= 2
//                   is accepted while S_{j-1} <= gamma;
//   general EB      inclusive prefix sum minus inclusive prefix max of the
//                   entropies in confidence order, <= gamma;
//   Factor          (n + 1) c^n < f (or (n + 1)(1 - c^n) < f) tested at every
//                   rank n; the largest passing rank, at least 1.
// Accepted positions get their sampled token committed into the block buffer
// and their masked flag cleared.
#include "sbd_internal.cuh"

namespace {

using namespace sbd_dev;

constexpr int kWarpsPerBlock = 4;

__device__ __forceinline__ bool key_less(float ha, int ia, float hb, int ib) {
  return ha < hb || (ha == hb && ia < ib);
}

template <int Rule>
__global__ void __launch_bounds__(32 * kWarpsPerBlock)
select_kernel(int B, int k, const float* __restrict__ entropy,
              const float* __restrict__ confidence, const int32_t* __restrict__ token,
              float threshold, uint8_t* __restrict__ masked, int32_t* __restrict__ block_tokens,
              int32_t* __restrict__ n_unmasked) {
  constexpr bool kByEntropy = Rule == SBD_SELECT_EB_ENTROPY;
  grid_dependency_wait();
  grid_dependents_launch();
  const int lane = threadIdx.x & 31;
  const int b = blockIdx.x * kWarpsPerBlock + (threadIdx.x >> 5);
  if (b >= B) return;

  // All loads are issued before any is used (the kernel is latency-bound);
  // the values of unmasked lanes are not used.
  const bool in_block = lane < k;
  const size_t at = (size_t)b * k + lane;
  const uint8_t m_raw = in_block ? masked[at] : (uint8_t)0;
  const float h_raw = in_block ? entropy[at] : 0.f;
  const float c_raw = (in_block && !kByEntropy) ? confidence[at] : 0.f;
  int tok = in_block ? token[at] : 0;
  const bool is_masked = m_raw != 0;
  float h = INFINITY;      // entropy
  float key = INFINITY;    // sort key, ascending
  if (is_masked) {
    h = h_raw;
    if (kByEntropy) {
      key = isnan(h) ? INFINITY : h;         // a NaN sorts last among masked
      h = key;
    } else {
      key = isnan(c_raw) ? INFINITY : -c_raw;   // confidence descending
    }
  }
  // Unmasked lanes sort after every masked one (position key offset by 32).
  int key_pos = is_masked ? lane : lane + 32;

  // Bitonic sort of 32 (key, position) pairs, ascending; the entropy and the
  // sampled token ride along.
#pragma unroll
  for (int size = 2; size <= 32; size <<= 1) {
#pragma unroll
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      const float ok = __shfl_xor_sync(0xffffffffu, key, stride);
      const int op = __shfl_xor_sync(0xffffffffu, key_pos, stride);
      const float oh = kByEntropy ? ok : __shfl_xor_sync(0xffffffffu, h, stride);
      const int ot = __shfl_xor_sync(0xffffffffu, tok, stride);
      const bool ascending = (lane & size) == 0 || size == 32;
      const bool lower = (lane & stride) == 0;
      const bool other_less = key_less(ok, op, key, key_pos);
      const bool take_other = (lower == ascending) ? other_less : !other_less;
      if (take_other) {
        key = ok;
        key_pos = op;
        h = oh;
        tok = ot;
      }
    }
  }

  const int n_masked = __popc(__ballot_sync(0xffffffffu, is_masked));
  const bool ranked = lane < n_masked;                // rank n = lane + 1
  int s;
  if (Rule == SBD_SELECT_EB_ENTROPY || Rule == SBD_SELECT_EB_CONFIDENCE) {
    // Inclusive prefix sum (and, for the general bound, prefix max) of the
    // entropies in sorted order (fp32).
    float incl = ranked ? h : 0.f;
    float pmax = ranked ? h : -INFINITY;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const float t = __shfl_up_sync(0xffffffffu, incl, o);
      const float tm = __shfl_up_sync(0xffffffffu, pmax, o);
      if (lane >= o) {
        incl += t;
        pmax = fmaxf(pmax, tm);
      }
    }
    bool refused;
    if (kByEntropy) {
      float excl = __shfl_up_sync(0xffffffffu, incl, 1);   // S_{j-1} for rank j = lane + 1
      if (lane == 0) excl = 0.f;
      refused = lane >= 1 && ranked && !(excl <= threshold);
    } else {
      refused = lane >= 1 && ranked && !(incl - pmax <= threshold);
    }
    // The accepted count is the first refused rank, so the accepted set is a
    // prefix (rank 1 is never refused).
    const unsigned refused_bits = __ballot_sync(0xffffffffu, refused);
    s = refused_bits ? (__ffs(refused_bits) - 1) : n_masked;
  } else {
    const float c = key == INFINITY ? NAN : -key;       // n-th largest confidence
    const float n1 = (float)(lane + 2);                 // n + 1
    const float lhs = Rule == SBD_SELECT_FACTOR ? n1 * c : n1 * (1.f - c);
    const unsigned pass = __ballot_sync(0xffffffffu, ranked && lhs < threshold);
    s = pass ? (32 - __clz(pass)) : 1;                  // the largest passing rank
  }
  if (s > n_masked) s = n_masked;

  if (lane < s) {
    const int pos = key_pos;                       // original block position
    const size_t o = (size_t)b * k + pos;
    block_tokens[o] = tok;
    masked[o] = 0;
  }
  if (lane == 0 && n_unmasked) n_unmasked[b] = s;
}

}  // namespace

namespace sbd {

sbd_status select_launch(int rule, int B, int k, const float* entropy, const float* confidence,
                         const int32_t* token, float threshold, uint8_t* masked,
                         int32_t* block_tokens, int32_t* n_unmasked, cudaStream_t st) {
  if (B == 0) return SBD_OK;
  const void* fn;
  switch (rule) {
    case SBD_SELECT_EB_ENTROPY: fn = (const void*)select_kernel<SBD_SELECT_EB_ENTROPY>; break;
    case SBD_SELECT_EB_CONFIDENCE:
      fn = (const void*)select_kernel<SBD_SELECT_EB_CONFIDENCE>;
      break;
    case SBD_SELECT_FACTOR: fn = (const void*)select_kernel<SBD_SELECT_FACTOR>; break;
    case SBD_SELECT_FACTOR_COMPLEMENT:
      fn = (const void*)select_kernel<SBD_SELECT_FACTOR_COMPLEMENT>;
      break;
    default: return fail(SBD_ERR_INVALID_ARG, "unknown selection rule %d", rule);
  }
  const int blocks = (B + kWarpsPerBlock - 1) / kWarpsPerBlock;
  void* args[] = {(void*)&B,         (void*)&k,      (void*)&entropy,
                  (void*)&confidence, (void*)&token,  (void*)&threshold,
                  (void*)&masked,    (void*)&block_tokens, (void*)&n_unmasked};
  return launch_pdl(fn, dim3(blocks), dim3(32 * kWarpsPerBlock), 0, st, args,
                    "select_kernel launch");
}

}  // namespace sbd
