// Internal declarations and sm_103a inline-PTX helpers of libsbd.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/sbd.h"

namespace sbd {

// ---------------------------------------------------------------- host side

// Records a formatted message for sbd_last_error() and returns `st`.
sbd_status fail(sbd_status st, const char* fmt, ...);
sbd_status cuda_fail(cudaError_t e, const char* what);
inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
// Queries the current device once (SM count, error-word address) and
// fails with the reason recorded when that is impossible; every entry point
// that launches calls it before num_sms() / device_error_word().
sbd_status device_ready();
int num_sms();                       // SMs of the current device (cached per device)
int* device_error_word();            // device address of the error word (current device)

// cuTensorMapEncodeTiled through the runtime's driver entry point.
sbd_status encode_tensor_map(CUtensorMap* map, CUtensorMapDataType dtype, uint32_t rank,
                             void* base, const uint64_t* dims, const uint64_t* strides_bytes,
                             const uint32_t* box, CUtensorMapSwizzle swizzle);

// Kernel launchers (each in the .cu file of its kernel).  Arguments were
// validated by the API layer.
struct AttnPlan {
  int B, k, Hq, Hkv, G, D, Lmax, M, splits;
  bool order;         // CTAs take sequences longest first (more than one wave)
  bool cluster;       // the splits of a (sequence, KV head) merge in a cluster (tcgen05 path)
  int n_causal;       // block rows i < n_causal see block keys j <= i only
  float scale_log2;   // softmax scale * log2(e)
  bool bf16;
};
size_t attn_workspace_bytes(const AttnPlan& p);
AttnPlan attn_plan(const sbd_attn_desc& d);
// kc_app / vc_app: when not NULL (the caches, writable), the keys and values
// of block rows i < p.n_causal are written at cache position L_b + i.
sbd_status attn_launch(const AttnPlan& p, const void* q, const void* kc, const void* vc,
                       const int32_t* lens, const void* kb, const void* vb, void* out,
                       void* ws, void* kc_app, void* vc_app, cudaStream_t st);

size_t attn_tc_smem_bytes(int D);
// Whether the tcgen05 attention kernel can run the `splits` CTAs of every
// (sequence, KV head) of plan p as one thread-block cluster, all at once.
bool attn_tc_cluster_ok(const AttnPlan& p, int splits);
sbd_status attn_tc_launch(const AttnPlan& p, const CUtensorMap& tk, const CUtensorMap& tv,
                          const void* q, const int32_t* lens, const void* kb, const void* vb,
                          void* out, float* part_o, float* part_lse, void* kc_app,
                          void* vc_app, cudaStream_t st);

struct HeadPlan {
  int B, k, H, V, rows_alloc, n_ctas;
  bool bf16;
};
HeadPlan head_plan(const sbd_head_desc& d);
size_t head_workspace_bytes(const HeadPlan& p);
// A lower bound of head_workspace_bytes for a descriptor, with no device
// query (the per-CTA partials of one CTA); 0 for an invalid descriptor.
size_t head_workspace_floor(const sbd_head_desc& d);
// Counter-based noise in place of a noise buffer (philox.cuh).
struct PhiloxNoise {
  uint64_t seed, offset;
};
// y[T, N] = x[T, K] W[N, K]^T, bf16 in and out, fp32 accumulation; T <= 512.
// At few rows K is split over CTAs (linear_ksplit ranges), with fp32 partials
// in the workspace (linear_workspace_bytes) summed by a second kernel.
int linear_ksplit(int T, int K, int N);
size_t linear_workspace_bytes(int T, int K, int N);
sbd_status linear_launch(int T, int K, int N, const void* x, const void* w, void* y, void* ws,
                         cudaStream_t st);
sbd_status head_launch(const HeadPlan& p, const void* hidden, const void* w,
                       const uint8_t* masked, const float* gumbel, float tau, float* entropy,
                       float* confidence, int32_t* token, void* ws, cudaStream_t st,
                       const PhiloxNoise* philox = nullptr);
sbd_status gumbel_fill_launch(int n_rows, const int32_t* row_ids, int V, uint64_t seed,
                              uint64_t offset, float* out, cudaStream_t st);

// rule: an sbd_select_rule value (SBD_SELECT_EB_ENTROPY for sbd_eb_select)
sbd_status select_launch(int rule, int B, int k, const float* entropy, const float* confidence,
                         const int32_t* token, float threshold, uint8_t* masked,
                         int32_t* block_tokens, int32_t* n_unmasked, cudaStream_t st);

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Launch with programmatic dependent launch allowed: the kernel may be
// scheduled while its predecessor on the stream finishes; every library
// kernel calls griddepcontrol.wait before it touches global memory.
// cluster_x > 1: CTAs of consecutive blockIdx.x form thread-block clusters of
// that size.
sbd_status launch_pdl(const void* fn, dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                      void** args, const char* what, int cluster_x = 1);
// How many clusters of cluster_x CTAs (with `smem` bytes of dynamic shared
// memory each) the current device can hold at once; 0 when the shape cannot
// be launched as clusters.
int max_active_clusters(const void* fn, dim3 grid, dim3 block, size_t smem, int cluster_x);

}  // namespace sbd

// ---------------------------------------------------------------- device side
namespace sbd_dev {

// Upper bound of every spin-wait inside a kernel (ns of %globaltimer).
constexpr uint64_t kWaitLimitNs = 2000000000ull;

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint64_t globaltimer() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ void record_error(int* word, int code) {
  if (word) atomicOr(word, code);
}

// ---- mbarrier
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count)
               : "memory");
}
__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ bool mbar_test_parity(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
// Non-blocking test of the same condition (for polling several barriers).
__device__ __forceinline__ bool mbar_poll_parity(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
// The sequence of CTA z when a launch spans more than one wave of CTAs: the
// one of rank z in descending cache length (ties by index), so that the
// longest sequences start first (longest-processing-time-first list
// scheduling of the CTAs onto the SMs).  Every thread of the CTA takes part;
// *out_b is set by one of them, and the caller's barrier publishes it.
// Lengths are clamped to [0, Lmax] as in the kernels.
__device__ __forceinline__ void longest_first_pick(const int32_t* lens, int B, int Lmax, int z,
                                                   int* out_b) {
  for (int i = threadIdx.x; i < B; i += blockDim.x) {
    const int li = min(max(lens[i], 0), Lmax);
    int rank = 0;
    for (int j = 0; j < B; ++j) {
      const int lj = min(max(lens[j], 0), Lmax);
      rank += (lj > li || (lj == li && j < i)) ? 1 : 0;
    }
    if (rank == z) *out_b = i;
  }
}

// Waits until the phase with the given parity has completed, for at most
// kWaitLimitNs.  Returns false (and records SBD_DEVERR_TIMEOUT) on time-out.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, int* err) {
  if (mbar_test_parity(bar, parity)) return true;
  const uint64_t t0 = globaltimer();
  for (uint32_t n = 1;; ++n) {
    if (mbar_test_parity(bar, parity)) return true;
    // the clock is read every 64 polls only
    if ((n & 63u) == 0 && globaltimer() - t0 > kWaitLimitNs) {
      record_error(err, SBD_DEVERR_TIMEOUT);
      return false;
    }
  }
}

// ---- proxies / fences
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// ---- TMA (tiled tensor copies global -> shared, completion on an mbarrier)
__device__ __forceinline__ void tma_prefetch_desc(const CUtensorMap* map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}
__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, uint64_t* bar,
                                            int c0, int c1) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4}], [%2];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(smem_u32(bar)), "r"(c0), "r"(c1)
      : "memory");
}
__device__ __forceinline__ void tma_load_2d_hint(void* dst, const CUtensorMap* map,
                                                 uint64_t* bar, int c0, int c1,
                                                 uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      ".L2::cache_hint [%0], [%1, {%3, %4}], [%2], %5;" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(smem_u32(bar)), "r"(c0), "r"(c1), "l"(policy)
      : "memory");
}
__device__ __forceinline__ void tma_load_4d(void* dst, const CUtensorMap* map, uint64_t* bar,
                                            int c0, int c1, int c2, int c3) {
  asm volatile(
      "cp.async.bulk.tensor.4d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4, %5, %6}], [%2];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(smem_u32(bar)), "r"(c0), "r"(c1), "r"(c2),
      "r"(c3)
      : "memory");
}
// Prefetch of a tensor tile into L2 (no shared memory, no completion).
__device__ __forceinline__ void tma_prefetch_l2_2d(const CUtensorMap* map, int c0, int c1) {
  asm volatile("cp.async.bulk.prefetch.tensor.2d.L2.global.tile [%0, {%1, %2}];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(c0), "r"(c1)
               : "memory");
}
// A hint that the 128-byte line holding p (global memory) is read soon.
__device__ __forceinline__ void prefetch_l2(const void* p) {
  asm volatile("prefetch.global.L2 [%0];" ::"l"(p) : "memory");
}
__device__ __forceinline__ void tma_prefetch_l2_4d(const CUtensorMap* map, int c0, int c1, int c2,
                                                   int c3) {
  asm volatile("cp.async.bulk.prefetch.tensor.4d.L2.global.tile [%0, {%1, %2, %3, %4}];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(c0), "r"(c1), "r"(c2), "r"(c3)
               : "memory");
}
__device__ __forceinline__ uint64_t l2_policy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}

// ---- programmatic dependent launch
__device__ __forceinline__ void grid_dependency_wait() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
}
__device__ __forceinline__ void grid_dependents_launch() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// ---- warp-level helpers
// 2^x by the SFU's ex2.approx.ftz instruction (PTX ISA: max relative error
// about 2^-22; results below 2^-126 flush to zero).  For probabilities that
// are rounded to bf16 or summed in fp32 right after.
__device__ __forceinline__ float ex2_ftz(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Running statistics of one logit row over a subset of the vocabulary, in
// base-2 units (y = z * log2 e):  m = max y,  S = sum 2^(y-m),
// T = sum 2^(y-m) (y-m); plus the best Gumbel score and its vocabulary id.
struct RowStats {
  float m, S, T, best;
  int idx;
};

__device__ __forceinline__ RowStats rowstats_empty() {
  RowStats r;
  r.m = -INFINITY;
  r.S = 0.f;
  r.T = 0.f;
  r.best = -INFINITY;
  r.idx = 0x7fffffff;
  return r;
}

// Merge of two disjoint subsets (log-sum-exp rescaling of S and T; argmax
// with ties to the lowest id).
__device__ __forceinline__ RowStats rowstats_merge(const RowStats& a, const RowStats& b) {
  RowStats r;
  r.m = fmaxf(a.m, b.m);
  if (r.m == -INFINITY) {
    r.S = 0.f;
    r.T = 0.f;
  } else {
    const float da = a.m - r.m, db = b.m - r.m;   // <= 0, -inf for empty sides
    const float ea = (a.S > 0.f) ? exp2f(da) : 0.f;
    const float eb = (b.S > 0.f) ? exp2f(db) : 0.f;
    r.S = ea * a.S + eb * b.S;
    r.T = (a.S > 0.f ? ea * (a.T + da * a.S) : 0.f) + (b.S > 0.f ? eb * (b.T + db * b.S) : 0.f);
  }
  const bool take_b = (b.best > a.best) || (b.best == a.best && b.idx < a.idx);
  r.best = take_b ? b.best : a.best;
  r.idx = take_b ? b.idx : a.idx;
  return r;
}

}  // namespace sbd_dev
