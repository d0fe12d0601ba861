// LM head over the masked block positions, reduced in the same kernel to a
// softmax entropy and a Gumbel-max token per position (arXiv 2509.04185,
// Eqs. 6-7 and Algorithm 3 "compute probabilities"; EB input of Eq. 3).
//
// Kernels, in launch order on one stream:
//   compact_rows_kernel  gathers the hidden rows of masked positions into a
//                        dense [rows_alloc, H] buffer and a row map; writes
//                        entropy = +inf / token = -1 for unmasked positions;
//   head_pair_kernel     (bf16) the LM head on CTA pairs (clusters of 2) with
//                        2-SM tcgen05 MMAs of M = 256: W and the masked
//                        hidden rows stream into shared-memory rings by TMA,
//                        rank 0 issues the MMAs into double-buffered fp32
//                        accumulators in tensor memory of both CTAs, and the
//                        epilogue warps reduce every logit to running
//                        statistics (max, sum of exponentials, entropy
//                        numerator, best Gumbel score and id) -- logits
//                        never reach HBM.  Two layouts, chosen from the
//                        live row count (see the kernel);
//   head_tc_kernel       (bf16) the same on single CTAs with 1-SM MMAs,
//                        swap-AB: 128 vocab rows of W are the M side (A,
//                        K-major), the masked hidden rows the N side (B,
//                        K-major); eight epilogue warps (two per TMEM lane
//                        quadrant, alternate 16-column chunks) reduce each
//                        logit column over the lanes.  The fallback where no
//                        cluster of two fits or the vocabulary is one tile;
//   head_f32_kernel      (fp32) the same reduction over exact fp32 FMAs;
//   head_combine_kernel  merges the per-CTA statistics of each row into the
//                        entropy (nats), the token and, when asked for, the
//                        confidence max_v p_v = 1 / S.
//
// Both tcgen05 kernels also serve sbd_linear (y = x W^T, a template
// switch): the same main loop over all rows of x, an epilogue that stores
// the outputs (or, with K split over CTAs, fp32 partials that
// linear_reduce_kernel sums); head_tc_kernel up to 160 rows, the pair
// kernel's rows layout above.
#include <math.h>

#include <mutex>

#include "philox.cuh"
#include "sbd_internal.cuh"

namespace {

using namespace sbd_dev;

constexpr int kBM = 128;              // vocab rows per tile (MMA M)
constexpr int kBK = 64;               // hidden columns per TMA box (one 128-B swizzle atom)
constexpr int kABytes = kBM * kBK * 2;  // one W box
constexpr int kMaxStages = 16;
// A pipeline stage holds up to this many consecutive boxes along the hidden
// dimension (longer contiguous reads of every W row per stage), and the ring
// gets this many bytes of shared memory.  One CTA per SM; W is loaded with
// an L2 evict-first policy, the hidden rows (re-read by every CTA) in boxes
// of up to 128 rows.
constexpr int kMaxBoxes = 4;
constexpr int kRingBytes = 216 * 1024;
// Epilogue warps (warps 2, 3, ...): warp w reads the TMEM lanes of quadrant
// w % 4, and the two warps of one quadrant take alternate 16-column chunks.
constexpr int kEpiWarps = 8;
// Chunks of Gumbel noise an epilogue warp keeps in flight ahead of the one
// it reduces (loads from HBM take longer than the reduction of one chunk).
// Measured on GB300 with 2 to 6 chunks: 3 is best or within 0.5 us of it at
// every row count (15 rows 156.6 -> 155.0 us against 2; 512 rows -6 %); 6
// spills registers.
constexpr int kGAhead = 3;
constexpr int kEpiThreads = 32 * kEpiWarps;
constexpr int kHeadThreads = 64 + kEpiThreads;   // warp 0 TMA, warp 1 MMA, then the epilogue
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

// Shared-memory scratch of the tensor-core epilogue for `rows` hidden rows:
// per TMEM quadrant and row the running (m, S, T, best) and best id, then
// the row map; rounded to 1 KB.
__host__ __device__ constexpr int head_scratch_bytes(int rows) {
  return (4 * rows * (16 + 4) + rows * 4 + 1023) & ~1023;
}

// ------------------------------------------------------------ tcgen05 PTX
__device__ __forceinline__ void tc_alloc(uint32_t* dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                   smem_u32(dst_smem)),
               "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tc_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
// D[tmem] (+)= A[smem desc] * B[smem desc]^T, bf16 inputs, fp32 accumulate.
__device__ __forceinline__ void tc_mma_bf16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                            uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// Arrives once on the mbarrier when every tcgen05 op issued so far by this
// thread has completed.
__device__ __forceinline__ void tc_commit(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
          smem_u32(bar))
      : "memory");
}
// 32 lanes x 16 consecutive 32-bit columns: thread t gets lane (base + t).
__device__ __forceinline__ void tc_ld_32x32b_x16(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
}
__device__ __forceinline__ void tc_wait_ld() {
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// Shared-memory matrix descriptor: K-major operand laid out by TMA with the
// 128-byte swizzle, rows 128 B apart, 8-row groups 1024 B apart.
__device__ __forceinline__ uint64_t sw128_kmajor_desc(uint32_t smem_addr) {
  uint64_t d = 0;
  d |= (uint64_t)((smem_addr & 0x3FFFFu) >> 4);   // start address
  d |= (uint64_t)(16u >> 4) << 16;                 // leading byte offset (unused here)
  d |= (uint64_t)(1024u >> 4) << 32;               // stride byte offset: 8 rows x 128 B
  d |= (uint64_t)1u << 46;                         // descriptor version (tcgen05)
  d |= (uint64_t)2u << 61;                         // 128-byte swizzle
  return d;
}
// Instruction descriptor, kind::f16: bf16 A and B (K-major), fp32 D.
__host__ __device__ constexpr uint32_t idesc_bf16_f32(int M, int N) {
  return (1u << 4)                  // D format: f32
         | (1u << 7)                // A format: bf16
         | (1u << 10)               // B format: bf16
         | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

// ---- the CTA-pair (2-SM) forms.  Two CTAs of a cluster share one MMA of
// M = 256: each holds 128 rows of A and half of B's N rows (rank 0 the first
// half) at the same shared-memory offsets, and each gets its 128 rows of D
// in its own tensor memory.  Every tcgen05 instruction of a pair kernel uses
// cta_group::2; allocation and release are performed by one warp of each
// CTA together.
__device__ __forceinline__ void tc_alloc_pair(uint32_t* dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                   smem_u32(dst_smem)),
               "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tc_dealloc_pair(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}
// Issued by one thread of the pair's rank-0 CTA.
__device__ __forceinline__ void tc_mma_bf16_pair(uint32_t d_tmem, uint64_t a_desc,
                                                 uint64_t b_desc, uint32_t idesc,
                                                 uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// One arrival on the mbarrier at this offset in every CTA of `cta_mask`
// once the pair's tcgen05 ops issued so far by this thread have completed.
__device__ __forceinline__ void tc_commit_pair(uint64_t* bar, uint16_t cta_mask) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64"
      " [%0], %1;" ::"r"(smem_u32(bar)),
      "h"(cta_mask)
      : "memory");
}
// TMA load into this CTA's shared memory whose completion is counted on an
// mbarrier of either CTA of the pair (bar: shared::cluster address).
__device__ __forceinline__ void tma_load_2d_pair(void* dst, const CUtensorMap* map, uint32_t bar,
                                                 int c0, int c1) {
  asm volatile(
      "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.tile"
      ".mbarrier::complete_tx::bytes [%0], [%1, {%3, %4}], [%2];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(bar), "r"(c0), "r"(c1)
      : "memory");
}
__device__ __forceinline__ void tma_load_2d_pair_hint(void* dst, const CUtensorMap* map,
                                                      uint32_t bar, int c0, int c1,
                                                      uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.tile"
      ".mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1, {%3, %4}], [%2], %5;" ::"r"(
          smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(bar), "r"(c0), "r"(c1), "l"(policy)
      : "memory");
}
__device__ __forceinline__ void pair_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\t"
               "barrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ uint32_t pair_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
// The shared::cluster address of this CTA's shared location `p` in the
// pair's rank-0 CTA.
__device__ __forceinline__ uint32_t at_rank0(const void* p) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, 0;" : "=r"(r) : "r"(smem_u32(p)));
  return r;
}
__device__ __forceinline__ void mbar_arrive_cluster(uint32_t bar) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(bar)
               : "memory");
}
// mbar_wait for a barrier that CTAs of the cluster arrive on.
__device__ __forceinline__ bool mbar_wait_cluster(uint64_t* bar, uint32_t parity, int* err) {
  const uint64_t t0 = globaltimer();
  for (uint32_t n = 0;; ++n) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    if (ok) return true;
    if ((n & 63u) == 63u && globaltimer() - t0 > kWaitLimitNs) {
      record_error(err, SBD_DEVERR_TIMEOUT);
      return false;
    }
  }
}

// ------------------------------------------------------------ epilogue math
__device__ __forceinline__ RowStats shfl_xor_stats(const RowStats& a, int o) {
  RowStats r;
  r.m = __shfl_xor_sync(0xffffffffu, a.m, o);
  r.S = __shfl_xor_sync(0xffffffffu, a.S, o);
  r.T = __shfl_xor_sync(0xffffffffu, a.T, o);
  r.best = __shfl_xor_sync(0xffffffffu, a.best, o);
  r.idx = __shfl_xor_sync(0xffffffffu, a.idx, o);
  return r;
}

// Statistics of one logit (this lane's vocabulary id v, one column).
__device__ __forceinline__ RowStats lane_stats(float z, bool valid, float g, float tau, int v) {
  RowStats r;
  r.m = valid ? z * kLog2e : -INFINITY;
  r.S = valid ? 1.f : 0.f;
  r.T = 0.f;
  r.best = valid ? fmaf(tau, g, z) : -INFINITY;
  r.idx = valid ? v : 0x7fffffff;
  return r;
}

// Reduces one column over the 32 lanes of a warp; every lane gets the result.
__device__ __forceinline__ RowStats warp_column_stats(float z, bool valid, float g, float tau,
                                                      int v) {
  RowStats st = lane_stats(z, valid, g, tau, v);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) st = rowstats_merge(st, shfl_xor_stats(st, o));
  return st;
}

// Statistics of 16 logit columns over the 32 vocabulary rows of a warp
// (lane = row, vocabulary id v0 + lane; z the logits, g the Gumbel noise).
// Two passes: the column maxima of z log2(e) and of the Gumbel score
// z + tau g go through a transposed max butterfly (16 + 8 + 4 + 2 + 1 steps
// instead of 16 x 5); every lane then takes exp2 of its logits against the
// column maxima, and the sums of the exponentials and of their entropy terms
// go through the same butterfly with additions.  The best id is the lowest
// lane that reaches the column's best score (ties to the lowest id).  On
// return lanes 2c and 2c + 1 hold column c.
__device__ __forceinline__ RowStats chunk16_stats(const float (&z)[16], const float (&g)[16],
                                                  bool valid, float tau, int v0, int lane) {
  float s[16], sc[16], ms[16], mb[16];
#pragma unroll
  for (int j = 0; j < 16; ++j) {
    s[j] = valid ? z[j] * kLog2e : -INFINITY;
    sc[j] = valid ? fmaf(tau, g[j], z[j]) : -INFINITY;
    ms[j] = s[j];
    mb[j] = sc[j];
  }
#pragma unroll
  for (int lvl = 0; lvl < 4; ++lvl) {
    const int b = 16 >> lvl;
    const int half = 8 >> lvl;
    const bool upper = (lane & b) != 0;
#pragma unroll
    for (int i = 0; i < half; ++i) {
      const float ks = upper ? ms[i + half] : ms[i];
      const float ss = upper ? ms[i] : ms[i + half];
      const float kb = upper ? mb[i + half] : mb[i];
      const float sb = upper ? mb[i] : mb[i + half];
      ms[i] = fmaxf(ks, __shfl_xor_sync(0xffffffffu, ss, b));
      mb[i] = fmaxf(kb, __shfl_xor_sync(0xffffffffu, sb, b));
    }
  }
  ms[0] = fmaxf(ms[0], __shfl_xor_sync(0xffffffffu, ms[0], 1));
  mb[0] = fmaxf(mb[0], __shfl_xor_sync(0xffffffffu, mb[0], 1));

  const int my_col = (lane >> 1) & 15;
  unsigned my_hits = 0u;
  float e[16], t[16];
#pragma unroll
  for (int j = 0; j < 16; ++j) {
    const float m = __shfl_sync(0xffffffffu, ms[0], 2 * j);
    const float best = __shfl_sync(0xffffffffu, mb[0], 2 * j);
    const float d = s[j] - m;                  // <= 0 on valid lanes
    e[j] = valid ? ex2_ftz(d) : 0.f;
    t[j] = valid ? e[j] * d : 0.f;
    const unsigned hits = __ballot_sync(0xffffffffu, valid && sc[j] == best);
    if (my_col == j) my_hits = hits;
  }
#pragma unroll
  for (int lvl = 0; lvl < 4; ++lvl) {
    const int b = 16 >> lvl;
    const int half = 8 >> lvl;
    const bool upper = (lane & b) != 0;
#pragma unroll
    for (int i = 0; i < half; ++i) {
      const float ke = upper ? e[i + half] : e[i];
      const float se = upper ? e[i] : e[i + half];
      const float kt = upper ? t[i + half] : t[i];
      const float st = upper ? t[i] : t[i + half];
      e[i] = ke + __shfl_xor_sync(0xffffffffu, se, b);
      t[i] = kt + __shfl_xor_sync(0xffffffffu, st, b);
    }
  }
  e[0] += __shfl_xor_sync(0xffffffffu, e[0], 1);
  t[0] += __shfl_xor_sync(0xffffffffu, t[0], 1);
  RowStats r;
  r.m = ms[0];
  r.S = e[0];
  r.T = t[0];
  r.best = mb[0];
  r.idx = my_hits ? v0 + __ffs(my_hits) - 1 : 0x7fffffff;
  return r;
}

struct StatsRef {
  float4* msTb;   // (m, S, T, best)
  int* idx;
};
__device__ __forceinline__ RowStats load_stats(const StatsRef& s, int i) {
  const float4 v = s.msTb[i];
  RowStats r;
  r.m = v.x;
  r.S = v.y;
  r.T = v.z;
  r.best = v.w;
  r.idx = s.idx[i];
  return r;
}
__device__ __forceinline__ void store_stats(const StatsRef& s, int i, const RowStats& r) {
  s.msTb[i] = make_float4(r.m, r.S, r.T, r.best);
  s.idx[i] = r.idx;
}

// ------------------------------------------------------------ compaction
__global__ void __launch_bounds__(256)
compact_rows_kernel(const uint8_t* __restrict__ hidden, const uint8_t* __restrict__ masked,
                    int BK, int row_bytes, uint8_t* __restrict__ hidden_c,
                    int32_t* __restrict__ row_map, int32_t* __restrict__ n_rows,
                    float* __restrict__ entropy, int32_t* __restrict__ token,
                    float* __restrict__ confidence) {
  grid_dependency_wait();
  grid_dependents_launch();
  const int row = blockIdx.x;
  const int t = threadIdx.x;
  // masked rows before `row`, and in total (BK <= 2 * blockDim.x)
  int before = 0, total = 0;
  for (int base = 0; base < BK; base += blockDim.x) {
    const int i = base + t;
    const bool mt = i < BK && masked[i] != 0;
    before += __syncthreads_count(mt && i < row);
    total += __syncthreads_count(mt);
  }
  int dst;
  bool copy = false;
  if (row < BK) {
    if (masked[row]) {
      dst = before;
      copy = true;
      if (t == 0) row_map[dst] = row;
    } else {
      dst = total + (row - before);
      if (t == 0) {
        entropy[row] = INFINITY;
        token[row] = -1;
        if (confidence) confidence[row] = 0.f;
      }
    }
  } else {
    dst = row;
  }
  const int n16 = row_bytes / 16;
  uint4* out = reinterpret_cast<uint4*>(hidden_c + (size_t)dst * row_bytes);
  const uint4* in = reinterpret_cast<const uint4*>(hidden + (size_t)row * row_bytes);
  for (int c = t; c < n16; c += blockDim.x) out[c] = copy ? in[c] : make_uint4(0, 0, 0, 0);
  if (row == 0 && t == 0) *n_rows = total;
}

// ------------------------------------------------------------ bf16 tcgen05
struct HeadArgs {
  const float* gumbel;   // noise rows [B*k, V] (noise from a buffer)
  uint32_t seed_lo, seed_hi, off_lo, off_hi;   // counter-based noise (kPhilox)
  const int32_t* row_map;
  const int32_t* n_rows;
  float4* part_msTb;     // [gridDim.x][rows_alloc]
  int32_t* part_idx;
  int* err;
  int V, H, rows_alloc, n_tiles;
  int ring_bytes;       // shared memory of the TMA ring (shaped in the kernel)
  uint32_t tmem_cols;
  float tau;
  int h_big;            // tallest hidden-row box encoded: 16, 64 or 128 rows
  __nv_bfloat16* y;     // kLinear: output [linear_rows, V]
  int linear_rows;      // kLinear: rows of x, all live
  int ksplit;           // kLinear: K ranges per output tile (1: y written directly)
  float* part_y;        // kLinear, ksplit > 1: fp32 partials [ksplit][linear_rows][V]
};

// kPhilox: the Gumbel noise is generated in the epilogue (philox.cuh)
// instead of read from a [B*k, V] buffer.  kLinear: the plain product
// y = x W^T in bf16 (all rows of x live, no compaction, no noise); the
// epilogue stores the accumulators instead of reducing them.
template <bool kPhilox, bool kLinear>
__global__ void __launch_bounds__(kHeadThreads, 1)
head_tc_kernel(const __grid_constant__ CUtensorMap tmap_w,
               const __grid_constant__ CUtensorMap tmap_h,
               const __grid_constant__ CUtensorMap tmap_h64,
               const __grid_constant__ CUtensorMap tmap_h128, const HeadArgs a) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[kMaxStages];
  __shared__ __align__(8) uint64_t empty_bar[kMaxStages];
  __shared__ __align__(8) uint64_t tmem_full[2];
  __shared__ __align__(8) uint64_t tmem_empty[2];
  __shared__ uint32_t tmem_base_sh;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t sbase = (smem_u32(smem_raw) + 1023u) & ~1023u;
  uint8_t* gbase = smem_raw + (sbase - smem_u32(smem_raw));

  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmap_w);
    tma_prefetch_desc(&tmap_h);
  }
  if (warp == 1) tc_alloc(&tmem_base_sh, a.tmem_cols);
  // Everything below reads what the compaction kernel wrote.
  grid_dependency_wait();
  const int R = kLinear ? a.linear_rows : *a.n_rows;
  const int n_eff = R <= 16 ? 16 : ((R + 15) / 16) * 16;   // MMA N
  // Two accumulator buffers whenever two of the live width fit in the
  // tensor memory of the launch (half of it each), so that the epilogue of
  // one tile overlaps the MMAs of the next; one above 256 live rows.
  const int n_acc = 2 * n_eff <= (int)a.tmem_cols ? 2 : 1;
  const uint32_t acc_stride = a.tmem_cols / 2;
  // Epilogue scratch for the n_eff live rows first, then the ring, which
  // also gets what the allocation kept for the scratch of rows_alloc rows.
  uint8_t* ep = gbase;
  const int ep_bytes = head_scratch_bytes(n_eff);
  const int ring_bytes = a.ring_bytes + head_scratch_bytes(a.rows_alloc) - ep_bytes;
  uint8_t* ring = gbase + ep_bytes;
  const uint32_t rbase = sbase + ep_bytes;
  // Statistics of TMEM lane quadrant w (computed, not indexed from an array:
  // a per-thread array of the four would live in local memory).
  auto wstats = [&](int w) -> StatsRef {
    StatsRef r;
    r.msTb = reinterpret_cast<float4*>(ep) + w * n_eff;
    r.idx = reinterpret_cast<int*>(ep + (size_t)4 * n_eff * sizeof(float4)) + w * n_eff;
    return r;
  };
  int* rmap = reinterpret_cast<int*>(ep + (size_t)4 * n_eff * (sizeof(float4) + 4));
  // Ring shape from the actual row count: a stage holds `boxes` 64-column
  // boxes of W (16 KB each) and of the n_eff hidden rows.  Above two boxes,
  // as many as still leave 3 stages; two boxes as long as 2 stages fit;
  // then as many stages as fit.  (Two boxes in 2 stages measured faster
  // than one box in 4-5: 160 rows 233 -> 219 us, 256 rows 255 -> 249 us;
  // four boxes in 2 stages slower than two in 4 at 60 rows.)
  const int b_box = n_eff * kBK * 2;
  // kLinear at few rows: each output tile's K is cut into `ksplit` ranges,
  // and the (tile, range) units are spread over the CTAs
  const int ksplit = kLinear ? a.ksplit : 1;
  const int n_units = a.n_tiles * ksplit;
  auto fits = [&](int bx, int n_st) { return ring_bytes / (bx * (kABytes + b_box)) >= n_st; };
  int boxes = kMaxBoxes;
  while (boxes > 1 &&
         ((a.H / kBK) % (boxes * ksplit) != 0 || !fits(boxes, boxes > 2 ? 3 : 2)))
    boxes >>= 1;
  const int stage_bytes = boxes * (kABytes + b_box);     // [A boxes | B boxes]
  int stages = ring_bytes / stage_bytes;
  if (stages > kMaxStages) stages = kMaxStages;
  // Epilogue warps with a chunk of 16 columns to reduce, per TMEM quadrant;
  // the others skip the tile loop.
  const int n_chunks = (R + 15) / 16;
  const int n_sub = n_chunks < kEpiWarps / 4 ? (n_chunks > 0 ? n_chunks : 1) : kEpiWarps / 4;
  if (threadIdx.x == 0) {
    for (int s = 0; s < stages; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&tmem_full[i], 1);
      mbar_init(&tmem_empty[i], 4 * n_sub);   // one arrival per working epilogue warp
    }
    fence_mbar_init();
  }
  if (warp >= 2) {
    const int te = threadIdx.x - 64;
    for (int i = te; i < n_eff; i += kEpiThreads) {
      rmap[i] = (!kLinear && i < R) ? a.row_map[i] : 0;
      for (int w = 0; w < 4; ++w) store_stats(wstats(w), i, rowstats_empty());
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = tmem_base_sh;
  const int num_kb = a.H / (kBK * boxes) / ksplit;   // stages per unit

  if (R > 0) {
    if (warp == 0) {
      // ------------------------------------------------ TMA producer
      if (lane == 0) {
        const uint64_t policy = l2_policy_evict_first();
        // the stage and its phase are counters, not quotients (see
        // head_pair_kernel's producer)
        int it = 0, s = 0;
        uint32_t ph = 0;
        bool ok = true;
        for (int u = blockIdx.x; ok && u < n_units; u += gridDim.x) {
          const int tile = u / ksplit, kb0 = (u % ksplit) * num_kb;
          for (int kb = 0; kb < num_kb; ++kb, ++it) {
            if (!mbar_wait(&empty_bar[s], ph ^ 1, a.err)) {
              ok = false;
              break;
            }
            uint8_t* st = ring + (size_t)s * stage_bytes;
            mbar_arrive_expect_tx(&full_bar[s], stage_bytes);
            for (int x = 0; x < boxes; ++x) {
              const int col = ((kb0 + kb) * boxes + x) * kBK;
              tma_load_2d_hint(st + x * kABytes, &tmap_w, &full_bar[s], col, tile * kBM, policy);
              // the n_eff hidden rows the MMA reads, in the tallest boxes that
              // fit: these rows come from L2 for every vocabulary tile, where
              // the copy rate per SM grows with the box size
              uint8_t* hb = st + boxes * kABytes + x * b_box;
              int r0 = 0;
              if (a.h_big >= 128)
                for (; r0 + 128 <= n_eff; r0 += 128)
                  tma_load_2d(hb + r0 * 128, &tmap_h128, &full_bar[s], col, r0);
              if (a.h_big >= 64)
                for (; r0 + 64 <= n_eff; r0 += 64)
                  tma_load_2d(hb + r0 * 128, &tmap_h64, &full_bar[s], col, r0);
              for (; r0 < n_eff; r0 += 16) tma_load_2d(hb + r0 * 128, &tmap_h, &full_bar[s], col, r0);
            }
            if (++s == stages) {
              s = 0;
              ph ^= 1u;
            }
          }
        }
        // copies still in flight must land before the CTA exits
        for (int q = it - stages > 0 ? it - stages : 0; q < it; ++q)
          mbar_wait(&full_bar[q % stages], (q / stages) & 1, a.err);
      }
    } else if (warp == 1) {
      // ------------------------------------------------ MMA issuer
      if (lane == 0) {
        // N is split into MMAs of at most 256 columns
        const int n_hi = n_eff > 256 ? n_eff - 256 : 0;
        const uint32_t idesc_lo = idesc_bf16_f32(kBM, n_eff > 256 ? 256 : n_eff);
        const uint32_t idesc_hi = idesc_bf16_f32(kBM, n_hi > 0 ? n_hi : 16);
        int it = 0, local = 0, s = 0;
        uint32_t ph = 0;
        bool ok = true;
        for (int u = blockIdx.x; ok && u < n_units; u += gridDim.x, ++local) {
          const int acc = n_acc == 2 ? (local & 1) : 0;
          const uint32_t use = (uint32_t)(n_acc == 2 ? (local >> 1) : local);
          if (!mbar_wait(&tmem_empty[acc], (use & 1) ^ 1, a.err)) break;
          tc_fence_after();
          const uint32_t d_tmem = tmem_base + (uint32_t)acc * acc_stride;
          for (int kb = 0; kb < num_kb; ++kb, ++it) {
            if (!mbar_wait(&full_bar[s], ph, a.err)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t st = rbase + (uint32_t)(s * stage_bytes);
            for (int x = 0; x < boxes; ++x) {
              const uint64_t adesc = sw128_kmajor_desc(st + x * kABytes);
              const uint64_t bdesc = sw128_kmajor_desc(st + boxes * kABytes + x * b_box);
#pragma unroll
              for (int kk = 0; kk < kBK / 16; ++kk) {
                const uint32_t accum = (kb != 0 || x != 0 || kk != 0);
                tc_mma_bf16(d_tmem, adesc + 2 * kk, bdesc + 2 * kk, idesc_lo, accum);
                if (n_hi > 0)   // rows 256.. of B: 256 x 128 B further on, 256 columns on
                  tc_mma_bf16(d_tmem + 256, adesc + 2 * kk, bdesc + (256 * 128 >> 4) + 2 * kk,
                              idesc_hi, accum);
              }
            }
            tc_commit(&empty_bar[s]);
            if (++s == stages) {
              s = 0;
              ph ^= 1u;
            }
          }
          if (ok) tc_commit(&tmem_full[acc]);
        }
      }
    } else {
      // ------------------------------------------------ epilogue warps
      const int quad = warp & 3;               // TMEM lanes 32*quad .. 32*quad+31
      const StatsRef my_stats = wstats(quad);
      const int sub = (warp - 2) / 4;          // chunks sub, sub + n_sub, ... of 16 columns
      const bool noisy = !kLinear && a.tau != 0.f && (kPhilox || a.gumbel != nullptr);
      const uint32_t lane_addr = (uint32_t)(quad * 32) << 16;
      int local = 0;
      for (int u = blockIdx.x; sub < n_sub && u < n_units; u += gridDim.x, ++local) {
        const int tile = u / ksplit, ks = u % ksplit;
        const int acc = n_acc == 2 ? (local & 1) : 0;
        const uint32_t use = (uint32_t)(n_acc == 2 ? (local >> 1) : local);
        const int v0 = tile * kBM + quad * 32;
        const int v = v0 + lane;
        const bool valid = v < a.V;
        const uint32_t t_acc = tmem_base + lane_addr + (uint32_t)acc * acc_stride;
        // Gumbel noise of the first kGAhead chunks is loaded while the MMAs
        // run; each chunk's reduction then loads the chunk kGAhead further on.
        const int stride = 16 * n_sub;
        const int c_first = 16 * sub;
        float gq[kGAhead][16];
        if constexpr (!kPhilox) {
#pragma unroll
          for (int d = 0; d < kGAhead; ++d)
#pragma unroll
            for (int j = 0; j < 16; ++j) {
              const int cn = c_first + d * stride + j;
              gq[d][j] = (noisy && valid && cn < R) ? __ldg(a.gumbel + (size_t)rmap[cn] * a.V + v) : 0.f;
            }
        }
        // the tcgen05.ld below is warp-collective: the warp goes on as a whole
        if (!__all_sync(0xffffffffu, mbar_wait(&tmem_full[acc], use & 1, a.err))) break;
        tc_fence_after();
        for (int c0 = c_first; c0 < R; c0 += stride) {
          float g[16];
          if constexpr (!kPhilox) {
#pragma unroll
            for (int j = 0; j < 16; ++j) g[j] = gq[0][j];
#pragma unroll
            for (int d = 0; d + 1 < kGAhead; ++d)
#pragma unroll
              for (int j = 0; j < 16; ++j) gq[d][j] = gq[d + 1][j];
#pragma unroll
            for (int j = 0; j < 16; ++j) {
              const int cn = c0 + kGAhead * stride + j;
              gq[kGAhead - 1][j] =
                  (noisy && valid && cn < R) ? __ldg(a.gumbel + (size_t)rmap[cn] * a.V + v) : 0.f;
            }
          } else if (noisy) {
            // The four lanes 4q..4q+3 share vocabulary ids 4(v div 4) ..
            // +3, i.e. one Philox counter per row: each lane computes the
            // calls of 4 of the chunk's 16 rows, and a 4 x 4 transpose inside
            // the group gives every lane word v mod 4 of all 16.
            const uint32_t vq = (uint32_t)v >> 2;
            const int i4 = lane & 3;
#pragma unroll
            for (int t = 0; t < 4; ++t) {
              const int rr = c0 + 4 * t + i4;
              const uint32_t n = rr < R ? (uint32_t)rmap[rr] : 0u;
              const uint4 x = sbd_philox::philox4x32_10(make_uint4(vq, n, a.off_lo, a.off_hi),
                                                        a.seed_lo, a.seed_hi);
              uint32_t b[4] = {0u, 0u, 0u, 0u};
#pragma unroll
              for (int d = 0; d < 4; ++d) {
                // send word (i ^ d); receive word i of the call of row 4t + (i ^ d)
                const uint32_t send = sbd_philox::word_of(x, i4 ^ d);
                const uint32_t recv = d == 0 ? send : __shfl_xor_sync(0xffffffffu, send, d);
#pragma unroll
                for (int jj = 0; jj < 4; ++jj) b[jj] = (jj == (i4 ^ d)) ? recv : b[jj];
              }
#pragma unroll
              for (int jj = 0; jj < 4; ++jj) g[4 * t + jj] = sbd_philox::gumbel_of_word(b[jj]);
            }
          } else {
#pragma unroll
            for (int j = 0; j < 16; ++j) g[j] = 0.f;
          }
          uint32_t r[16];
          tc_ld_32x32b_x16(t_acc + (uint32_t)c0, r);
          tc_wait_ld();
          if constexpr (kLinear) {
            // y[c0 + j, v] (or its fp32 partial of K range ks): for each j the
            // warp's lanes store 32 consecutive v
            if (valid) {
              if (ksplit == 1) {
#pragma unroll
                for (int j = 0; j < 16; ++j)
                  if (c0 + j < R)
                    a.y[(size_t)(c0 + j) * a.V + v] = __float2bfloat16_rn(__uint_as_float(r[j]));
              } else {
                float* py = a.part_y + (size_t)ks * R * a.V;
#pragma unroll
                for (int j = 0; j < 16; ++j)
                  if (c0 + j < R) py[(size_t)(c0 + j) * a.V + v] = __uint_as_float(r[j]);
              }
            }
          } else {
            float z[16];
#pragma unroll
            for (int j = 0; j < 16; ++j) z[j] = __uint_as_float(r[j]);
            const RowStats st = chunk16_stats(z, g, valid, a.tau, v0, lane);
            const int col = c0 + ((lane >> 1) & 15);
            if ((lane & 1) == 0 && col < R)
              store_stats(my_stats, col, rowstats_merge(load_stats(my_stats, col), st));
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&tmem_empty[acc]);
      }
      asm volatile("bar.sync 1, %0;" ::"n"(kEpiThreads) : "memory");
      const int te = threadIdx.x - 64;
      if constexpr (!kLinear) {
        for (int col = te; col < R; col += kEpiThreads) {
          RowStats s = load_stats(wstats(0), col);
          for (int w = 1; w < 4; ++w) s = rowstats_merge(s, load_stats(wstats(w), col));
          const size_t o = (size_t)blockIdx.x * a.rows_alloc + col;
          a.part_msTb[o] = make_float4(s.m, s.S, s.T, s.best);
          a.part_idx[o] = s.idx;
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tc_dealloc(tmem_base, a.tmem_cols);
  }
}

// ------------------------------------------------------------ bf16 tcgen05, CTA pairs
// head_pair_kernel: the LM head on CTA pairs (clusters of 2) running 2-SM
// MMAs of M = 256.  A unit of work is a pair tile of 256 vocabulary rows
// (128 W rows in each CTA).  Both CTAs' copies complete on rank 0's full
// barriers; rank 0's thread issues the MMAs and commits them to the barriers
// of both CTAs; the epilogue warps of rank 1 release an accumulator on rank
// 0's barrier.  Two layouts, chosen from the live row count R:
//  - Rows mode (R > kPairVocabLanesMax = 160): the hidden rows are the A side
//    (TMEM lane = hidden row, 128 per CTA) and W the B side (N = 256), so
//    that each CTA's accumulator holds its rows' logits over all 256 ids of
//    the tile.  Each epilogue thread owns one row and folds its logits into
//    running statistics in registers, with no exchange between lanes; the
//    two warps of a lane quadrant take alternate 16-column chunks and merge
//    at the end.  Above 256 live rows there are two row groups; the pairs
//    take one group each, and the two pairs of a tile run at the same time
//    (W's lines come from L2 for the second).
//  - Vocabulary mode (R <= kPairVocabLanesMax): as in head_tc_kernel, W is
//    the A side (TMEM lane = vocabulary row) and the live rows the B side
//    (N = R padded to 32, half of them in each CTA), with the column
//    reductions over lanes.  The MMA's work then grows with R instead of
//    being fixed at 256 rows.
// Measured on GB300: a 2-SM MMA of N = 256 takes ~65 ns, the same rate per
// SM as a 1-SM MMA; what the pair gains is that each SM reads half of the
// hidden rows from L2 (the B operand is split between the two CTAs).  The
// vocabulary layout's time grows with its padded N (when the threshold was
// set: 131 live rows 192 us, 160 rows 198 us, 161-192 rows, padded to 192,
// 222 us) while the rows layout took ~212 us anywhere from 129 to 256 rows;
// re-checked on the current kernel, the rows layout is still slower at 131
// rows (190.0 against 187.5 us).  Below that the rows layout's fixed
// 256-row MMAs also cost power (it ran at ~1750 MHz and ~950 W at 60 live
// rows, against 2070 MHz and ~450 W for head_tc_kernel) and lost to it.
constexpr int kPairRows = 128;                 // hidden rows of one CTA per unit (M / 2)
constexpr int kPairVocabLanesMax = 160;        // live rows up to which the vocabulary layout runs

// One 16-column chunk of a row's logits z (vocabulary ids v0 .. v0 + 15, valid
// below V) and Gumbel noise g folded into the running statistics.
__device__ __forceinline__ void fold_chunk16(RowStats& st, const float (&z)[16],
                                             const float (&g)[16], float tau, int v0, int V) {
  float y[16];
  float mc = -INFINITY;
#pragma unroll
  for (int j = 0; j < 16; ++j) {
    y[j] = v0 + j < V ? z[j] * kLog2e : -INFINITY;
    mc = fmaxf(mc, y[j]);
  }
  if (mc == -INFINITY) return;                  // no valid id in this chunk
  const float m_new = fmaxf(st.m, mc);
  float s_add = 0.f, t_add = 0.f;
#pragma unroll
  for (int j = 0; j < 16; ++j) {
    // invalid ids: 2^-1000 flushes to 0, and 0 * -1000 adds nothing to T
    const float d = v0 + j < V ? y[j] - m_new : -1000.f;
    const float e = ex2_ftz(d);
    s_add += e;
    t_add = fmaf(e, d, t_add);
  }
  if (st.S > 0.f) {
    // rescale the old sums to the new maximum: T' = 2^dm (T + dm S)
    const float dm = st.m - m_new;
    const float alpha = ex2_ftz(dm);
    st.T = fmaf(alpha, fmaf(dm, st.S, st.T), t_add);
    st.S = fmaf(alpha, st.S, s_add);
  } else {
    st.T = t_add;
    st.S = s_add;
  }
  st.m = m_new;
#pragma unroll
  for (int j = 0; j < 16; ++j) {
    // ids ascend within the chunk: a strict > keeps the lowest id on ties
    const float sc = fmaf(tau, g[j], z[j]);
    if (v0 + j < V && sc > st.best) {
      st.best = sc;
      st.idx = v0 + j;
    }
  }
}

// kLinear: sbd_linear's product y = x W^T (all rows of x live, no noise),
// always in the rows layout, the epilogue storing each row's outputs; with
// a.ksplit > 1 each (pair tile, K range) is a unit and the epilogue stores
// fp32 partials for linear_reduce_kernel.
// Two values rounded to bf16 (nearest even), the first in the low half.
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&v);
}

template <bool kPhilox, bool kLinear>
__global__ void __launch_bounds__(kHeadThreads, 1)
head_pair_kernel(const __grid_constant__ CUtensorMap tmap_w,
                 const __grid_constant__ CUtensorMap tmap_h,
                 const __grid_constant__ CUtensorMap tmap_h64,
                 const __grid_constant__ CUtensorMap tmap_h128, const HeadArgs a) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[kMaxStages];
  __shared__ __align__(8) uint64_t empty_bar[kMaxStages];
  __shared__ __align__(8) uint64_t tmem_full[2];
  __shared__ __align__(8) uint64_t tmem_empty[2];
  __shared__ __align__(8) uint64_t drain_bar;
  __shared__ uint32_t tmem_base_sh;
  __shared__ float4 half_msTb[kPairRows];   // the second warp of each quadrant's row statistics
  __shared__ int half_idx[kPairRows];
  static_assert(!(kPhilox && kLinear), "the linear form has no noise");

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t sbase = (smem_u32(smem_raw) + 1023u) & ~1023u;
  uint8_t* gbase = smem_raw + (sbase - smem_u32(smem_raw));
  const int rank = (int)pair_rank();
  const int pair = (int)(blockIdx.x >> 1), n_pairs = (int)(gridDim.x >> 1);

  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmap_w);
    tma_prefetch_desc(&tmap_h);
  }
  // Everything below reads what the compaction kernel wrote.
  grid_dependency_wait();
  const int R = kLinear ? a.linear_rows : *a.n_rows;
  // The layout: hidden rows on the lanes above kPairVocabLanesMax live rows,
  // vocabulary rows on the lanes up to it.
  const bool rows_mode = kLinear || R > kPairVocabLanesMax;
  // Row groups of 2 x 128 rows (rows mode); each pair takes one group and
  // every per_group-th tile from its first one.
  const int n_groups = R > 2 * kPairRows ? 2 : 1;
  const int per_group = n_pairs / n_groups;
  const int grp = pair % n_groups;
  const bool working = R > 0 && pair < per_group * n_groups;
  const int t_first = pair / n_groups;
  // kLinear: K ranges per pair tile; a "tile" index below runs over
  // (pair tile, K range) pairs
  const int ksplit = kLinear ? a.ksplit : 1;
  const int n_tk = a.n_tiles * ksplit;
  // this CTA's hidden rows row0 .. row0 + 127 (live below R), and the peer's
  const int row0 = grp * 2 * kPairRows + rank * kPairRows;
  auto live_rows = [&](int r0) { return R - r0 < 0 ? 0 : (R - r0 > kPairRows ? kPairRows : R - r0); };
  const int live = live_rows(row0);
  const int live16 = (live + 15) / 16 * 16;                       // rows loaded
  const int peer16 = (live_rows(grp * 2 * kPairRows + (1 - rank) * kPairRows) + 15) / 16 * 16;
  // Ring: a stage holds `boxes` 64-column boxes of the hidden rows, then as
  // many of W (128 rows).  A hidden box takes the rows rank 0 of the group
  // loads (the larger share; the same layout in both CTAs): the MMA reads
  // 128 rows from its start, and the rows past the live ones come from the
  // next box or from W in the same stage, landed and only feeding the
  // accumulator lanes of rows that are not live.  So the ring holds as much
  // W as the live rows leave room for; as many boxes as still leave 3 stages.
  //
  // Vocabulary mode: the live rows padded to G (a multiple of 32), each CTA
  // loading G / 2 of them as its half of the B side; a stage holds `boxes`
  // boxes of W, then as many of the hidden rows.  The epilogue's running
  // statistics (per lane quadrant and row) and the row map sit in shared
  // memory before the ring.
  const int G = ((R > 0 ? R : 1) + 31) / 32 * 32;
  const int n_eff = R <= 16 ? 16 : (R + 15) / 16 * 16;
  const int ep_bytes = rows_mode ? 0 : head_scratch_bytes(n_eff);
  uint8_t* ep = gbase;
  uint8_t* ring = gbase + ep_bytes;
  const uint32_t rbase = sbase + (uint32_t)ep_bytes;
  const int ring_bytes = a.ring_bytes - ep_bytes;
  const int h_box = rows_mode ? ((live_rows(grp * 2 * kPairRows) + 15) / 16 * 16) * kBK * 2
                              : (G / 2) * kBK * 2;
  // At least three stages.  (Two stages of longer W runs had measured 1-1.4 %
  // faster at 131 and 160 live rows while the control threads divided by
  // the stage count; with counters three are 1.5-2 % faster there.)
  const int min_stages = 3;
  int boxes = kMaxBoxes;
  while (boxes > 1 && ((a.H / kBK) % (boxes * ksplit) != 0 ||
                       ring_bytes / (boxes * (kABytes + h_box)) < min_stages))
    boxes >>= 1;
  const int stage_bytes = boxes * (kABytes + h_box);
  int stages = ring_bytes / stage_bytes;
  if (stages > kMaxStages) stages = kMaxStages;
  const int num_kb = a.H / (kBK * boxes) / ksplit;                 // stages per unit
  // offsets in a stage of W box x and hidden box x; the hidden rows loaded
  const int w_off0 = rows_mode ? boxes * h_box : 0;
  const int h_off0 = rows_mode ? 0 : boxes * kABytes;
  const int h_first = rows_mode ? row0 : rank * (G / 2);
  const int h_count = rows_mode ? live16 : G / 2;
  // bytes landing per stage on rank 0's barrier: W and hidden rows of both CTAs
  const uint32_t tx_pair = rows_mode
      ? (uint32_t)boxes * (2u * kABytes + (uint32_t)(live16 + peer16) * 128u)
      : 2u * (uint32_t)stage_bytes;
  // vocabulary mode: statistics of TMEM lane quadrant w, and the row map
  auto wstats = [&](int w) -> StatsRef {
    StatsRef r;
    r.msTb = reinterpret_cast<float4*>(ep) + w * n_eff;
    r.idx = reinterpret_cast<int*>(ep + (size_t)4 * n_eff * sizeof(float4)) + w * n_eff;
    return r;
  };
  int* rmap = reinterpret_cast<int*>(ep + (size_t)4 * n_eff * (sizeof(float4) + 4));
  if (threadIdx.x == 0) {
    for (int s = 0; s < stages; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&tmem_full[i], 1);
      mbar_init(&tmem_empty[i], 2 * kEpiWarps);   // every epilogue warp of both CTAs
    }
    mbar_init(&drain_bar, 1);
    fence_mbar_init();
  }
  if (!rows_mode && warp >= 2) {
    for (int i = threadIdx.x - 64; i < n_eff; i += kEpiThreads) {
      rmap[i] = i < R ? a.row_map[i] : 0;
      for (int w = 0; w < 4; ++w) store_stats(wstats(w), i, rowstats_empty());
    }
  }
  // Both CTAs run and their barriers are initialised before either one
  // signals the other's; the pair then allocates its tensor memory.
  pair_sync();
  if (warp == 1) tc_alloc_pair(&tmem_base_sh, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = tmem_base_sh;

  if (working) {
    if (warp == 0) {
      // ------------------------------------------------ TMA producer
      if (lane == 0) {
        // W is read once: evict-first, except where two row groups share it
        const bool w_hint = n_groups == 1;
        const uint64_t policy = l2_policy_evict_first();
        // This thread shares an SM sub-partition with two busy epilogue warps
        // and issues every copy, so its loop keeps little arithmetic per
        // stage: the stage and its phase are counters, not quotients by the
        // (run-time) stage count.  On GB300 that took the 60-row call from
        // 174.5 to 166.6 us and the 512-row one 8 % down (same for the MMA
        // thread below).
        int it = 0, s = 0;
        uint32_t ph = 0;
        bool ok = true;
        for (int tk = t_first; ok && tk < n_tk; tk += per_group) {
          const int t = tk / ksplit, kb0 = (tk % ksplit) * num_kb;
          const int w_row = (2 * t + rank) * kBM;
          for (int kb = 0; kb < num_kb; ++kb, ++it) {
            if (!mbar_wait(&empty_bar[s], ph ^ 1, a.err)) {
              ok = false;
              break;
            }
            uint8_t* st = ring + (size_t)s * stage_bytes;
            if (rank == 0) mbar_arrive_expect_tx(&full_bar[s], tx_pair);
            const uint32_t fb = at_rank0(&full_bar[s]);
            for (int x = 0; x < boxes; ++x) {
              const int col = ((kb0 + kb) * boxes + x) * kBK;
              uint8_t* wb = st + w_off0 + x * kABytes;
              if (w_hint) tma_load_2d_pair_hint(wb, &tmap_w, fb, col, w_row, policy);
              else tma_load_2d_pair(wb, &tmap_w, fb, col, w_row);
              // the hidden rows in the tallest boxes that fit (from L2)
              uint8_t* hb = st + h_off0 + x * h_box;
              int r0 = 0;
              if (a.h_big >= 128)
                for (; r0 + 128 <= h_count; r0 += 128)
                  tma_load_2d_pair(hb + r0 * 128, &tmap_h128, fb, col, h_first + r0);
              if (a.h_big >= 64)
                for (; r0 + 64 <= h_count; r0 += 64)
                  tma_load_2d_pair(hb + r0 * 128, &tmap_h64, fb, col, h_first + r0);
              for (; r0 < h_count; r0 += 16)
                tma_load_2d_pair(hb + r0 * 128, &tmap_h, fb, col, h_first + r0);
            }
            if (++s == stages) {
              s = 0;
              ph ^= 1u;
            }
          }
        }
        // Copies still in flight must land before the CTA exits.  Rank 1
        // cannot wait on rank 0's full barriers: it waits until the MMAs
        // released its last stages, which they do only after they arrived.
        bool landed = true;
        for (int q = it - stages > 0 ? it - stages : 0; landed && q < it; ++q)
          landed = rank == 0 ? mbar_wait(&full_bar[q % stages], (q / stages) & 1, a.err)
                             : mbar_wait(&empty_bar[q % stages], (q / stages) & 1, a.err);
      }
    } else if (warp == 1) {
      // ------------------------------------------------ MMA issuer (rank 0)
      if (lane == 0 && rank == 0) {
        // rows mode: A = hidden rows, B = W (N = 256 vocabulary ids);
        // vocabulary mode: A = W, B = hidden rows (N = G)
        const uint32_t idesc = idesc_bf16_f32(2 * kPairRows, rows_mode ? 2 * kBM : G);
        int it = 0, local = 0, s = 0;
        uint32_t ph = 0;
        bool ok = true;
        for (int tk = t_first; ok && tk < n_tk; tk += per_group, ++local) {
          const int acc = local & 1;
          const uint32_t use = (uint32_t)(local >> 1);
          // both CTAs' epilogue warps release the accumulator here
          if (!mbar_wait_cluster(&tmem_empty[acc], (use & 1) ^ 1, a.err)) break;
          tc_fence_after();
          const uint32_t d_tmem = tmem_base + (uint32_t)acc * 256u;
          for (int kb = 0; kb < num_kb; ++kb, ++it) {
            if (!mbar_wait(&full_bar[s], ph, a.err)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t st = rbase + (uint32_t)(s * stage_bytes);
            for (int x = 0; x < boxes; ++x) {
              const uint32_t w_s = st + (uint32_t)(w_off0 + x * kABytes);
              const uint32_t h_s = st + (uint32_t)(h_off0 + x * h_box);
              const uint64_t adesc = sw128_kmajor_desc(rows_mode ? h_s : w_s);
              const uint64_t bdesc = sw128_kmajor_desc(rows_mode ? w_s : h_s);
#pragma unroll
              for (int kk = 0; kk < kBK / 16; ++kk)
                tc_mma_bf16_pair(d_tmem, adesc + 2 * kk, bdesc + 2 * kk, idesc,
                                 (kb != 0 || x != 0 || kk != 0) ? 1u : 0u);
            }
            tc_commit_pair(&empty_bar[s], 0x3);
            if (++s == stages) {
              s = 0;
              ph ^= 1u;
            }
          }
          if (ok) tc_commit_pair(&tmem_full[acc], 0x3);
        }
        // the MMAs read both CTAs' shared memory: none may be in flight when
        // the pair leaves (this matters after a time-out only)
        tc_commit_pair(&drain_bar, 0x1);
        mbar_wait(&drain_bar, 0, a.err);
      }
    } else if (rows_mode) {
      // ------------------------------------------------ epilogue warps, rows mode
      const int quad = warp & 3;               // TMEM lanes 32*quad .. 32*quad+31
      const int sub = (warp - 2) >> 2;         // 16-column chunks sub, sub + 2, ... of a unit
      const int h = row0 + quad * 32 + lane;   // this thread's hidden row
      const bool row_live = h < R;
      const bool warp_live = __any_sync(0xffffffffu, row_live);
      const int n = !kLinear && row_live ? a.row_map[h] : 0;
      const bool noisy = !kLinear && a.tau != 0.f && (kPhilox || a.gumbel != nullptr);
      const float* grow = noisy && !kPhilox ? a.gumbel + (size_t)n * a.V : nullptr;
      // kLinear: 16-byte stores of 8 outputs where the row stride allows
      const bool y_vec = ((reinterpret_cast<uintptr_t>(a.y) | (uintptr_t)a.V * 2u) & 15u) == 0;
      const bool p_vec = ((reinterpret_cast<uintptr_t>(a.part_y) | (uintptr_t)a.V * 4u) & 15u) == 0;
      const bool vec4 = ((reinterpret_cast<uintptr_t>(a.gumbel) | (uintptr_t)a.V * 4u) & 15u) == 0;
      const uint32_t lane_addr = (uint32_t)(quad * 32) << 16;
      constexpr int kChunks = 2 * kBM / 16 / 2;   // chunks of one warp per unit
      auto load_noise = [&](int v0, float (&g)[16]) {
        if (!(noisy && row_live)) {
#pragma unroll
          for (int j = 0; j < 16; ++j) g[j] = 0.f;
        } else if constexpr (kPhilox) {
          // one call gives the words of ids 4q .. 4q + 3 (v0 is a multiple of 16)
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            const uint4 x = sbd_philox::philox4x32_10(
                make_uint4(((uint32_t)v0 >> 2) + (uint32_t)i, (uint32_t)n, a.off_lo, a.off_hi),
                a.seed_lo, a.seed_hi);
#pragma unroll
            for (int w = 0; w < 4; ++w) g[4 * i + w] = sbd_philox::gumbel_of_word(sbd_philox::word_of(x, w));
          }
        } else if (vec4) {
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            const float4 q4 = v0 + 4 * i < a.V ? __ldg(reinterpret_cast<const float4*>(grow + v0) + i)
                                               : make_float4(0.f, 0.f, 0.f, 0.f);
            g[4 * i] = q4.x;
            g[4 * i + 1] = q4.y;
            g[4 * i + 2] = q4.z;
            g[4 * i + 3] = q4.w;
          }
        } else {
#pragma unroll
          for (int j = 0; j < 16; ++j) g[j] = v0 + j < a.V ? __ldg(grow + v0 + j) : 0.f;
        }
      };
      RowStats st = rowstats_empty();
      int local = 0;
      for (int tk = t_first; tk < n_tk; tk += per_group, ++local) {
        const int t = tk / ksplit, ks = tk % ksplit;
        const int acc = local & 1;
        const uint32_t use = (uint32_t)(local >> 1);
        const int vt = t * 2 * kBM;                     // first vocabulary id of the tile
        const uint32_t t_acc = tmem_base + lane_addr + (uint32_t)acc * 256u;
        // noise of the first kGAhead chunks is read while the MMAs run
        float gq[kGAhead][16];
        if constexpr (!kPhilox) {
#pragma unroll
          for (int d = 0; d < kGAhead; ++d) load_noise(vt + 16 * (sub + 2 * d), gq[d]);
        }
        // the tcgen05.ld below is warp-collective: the warp goes on as a whole
        if (!__all_sync(0xffffffffu, mbar_wait(&tmem_full[acc], use & 1, a.err))) break;
        tc_fence_after();
        if (warp_live) {
#pragma unroll 1
          for (int c = 0; c < kChunks; ++c) {
            const int col = 16 * (sub + 2 * c);
            float g[16];
            if constexpr (!kPhilox) {
#pragma unroll
              for (int j = 0; j < 16; ++j) g[j] = gq[0][j];
#pragma unroll
              for (int d = 0; d + 1 < kGAhead; ++d)
#pragma unroll
                for (int j = 0; j < 16; ++j) gq[d][j] = gq[d + 1][j];
              if (c + kGAhead < kChunks) load_noise(vt + col + 32 * kGAhead, gq[kGAhead - 1]);
            } else {
              load_noise(vt + col, g);
            }
            uint32_t r[16];
            tc_ld_32x32b_x16(t_acc + (uint32_t)col, r);
            tc_wait_ld();
            if (row_live) {
              float z[16];
#pragma unroll
              for (int j = 0; j < 16; ++j) z[j] = __uint_as_float(r[j]);
              if constexpr (kLinear) {
                // y[h, vt + col + j], j < 16, below out_features (a.V), or
                // with K ranges the fp32 partial of range ks
                const int n0 = vt + col;
                if (ksplit > 1) {
                  float* pr = a.part_y + ((size_t)ks * R + h) * a.V + n0;
                  if (p_vec && n0 + 16 <= a.V) {
#pragma unroll
                    for (int i = 0; i < 4; ++i)
                      reinterpret_cast<float4*>(pr)[i] =
                          make_float4(z[4 * i], z[4 * i + 1], z[4 * i + 2], z[4 * i + 3]);
                  } else {
#pragma unroll
                    for (int j = 0; j < 16; ++j)
                      if (n0 + j < a.V) pr[j] = z[j];
                  }
                } else {
                  __nv_bfloat16* yr = a.y + (size_t)h * a.V + n0;
                  if (y_vec && n0 + 16 <= a.V) {
                    uint4 q0, q1;
                    q0.x = pack_bf16x2(z[0], z[1]);
                    q0.y = pack_bf16x2(z[2], z[3]);
                    q0.z = pack_bf16x2(z[4], z[5]);
                    q0.w = pack_bf16x2(z[6], z[7]);
                    q1.x = pack_bf16x2(z[8], z[9]);
                    q1.y = pack_bf16x2(z[10], z[11]);
                    q1.z = pack_bf16x2(z[12], z[13]);
                    q1.w = pack_bf16x2(z[14], z[15]);
                    reinterpret_cast<uint4*>(yr)[0] = q0;
                    reinterpret_cast<uint4*>(yr)[1] = q1;
                  } else {
#pragma unroll
                    for (int j = 0; j < 16; ++j)
                      if (n0 + j < a.V) yr[j] = __float2bfloat16_rn(z[j]);
                  }
                }
              } else {
                fold_chunk16(st, z, g, a.tau, vt + col, a.V);
              }
            }
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          if (rank == 1) mbar_arrive_cluster(at_rank0(&tmem_empty[acc]));
          else mbar_arrive(&tmem_empty[acc]);
        }
      }
      // the two warps of a quadrant merge their halves of each row
      const int slot = quad * 32 + lane;
      if constexpr (!kLinear) {
      if (sub == 1) {
        half_msTb[slot] = make_float4(st.m, st.S, st.T, st.best);
        half_idx[slot] = st.idx;
      }
      asm volatile("bar.sync 1, %0;" ::"n"(kEpiThreads) : "memory");
      if (sub == 0 && row_live) {
        RowStats o;
        o.m = half_msTb[slot].x;
        o.S = half_msTb[slot].y;
        o.T = half_msTb[slot].z;
        o.best = half_msTb[slot].w;
        o.idx = half_idx[slot];
        st = rowstats_merge(st, o);
        const size_t off = (size_t)blockIdx.x * a.rows_alloc + h;
        a.part_msTb[off] = make_float4(st.m, st.S, st.T, st.best);
        a.part_idx[off] = st.idx;
      }
      }
    } else if constexpr (!kLinear) {
      // ------------------------------------------------ epilogue warps, vocabulary mode
      // As in head_tc_kernel: thread = vocabulary row (TMEM lane), chunks of
      // 16 hidden-row columns reduced over the warp (chunk16_stats) and
      // merged into the quadrant's statistics in shared memory.
      const int quad = warp & 3;
      const StatsRef my_stats = wstats(quad);
      const int sub = (warp - 2) >> 2;          // chunks sub, sub + 2, ... of 16 columns
      const bool noisy = a.tau != 0.f && (kPhilox || a.gumbel != nullptr);
      const uint32_t lane_addr = (uint32_t)(quad * 32) << 16;
      constexpr int kStride = 32;
      const int c_first = 16 * sub;
      int local = 0;
      for (int t = t_first; t < a.n_tiles; t += per_group, ++local) {
        const int acc = local & 1;
        const uint32_t use = (uint32_t)(local >> 1);
        const int v0 = (2 * t + rank) * kBM + quad * 32;
        const int v = v0 + lane;
        const bool valid = v < a.V;
        const uint32_t t_acc = tmem_base + lane_addr + (uint32_t)acc * 256u;
        // Gumbel noise of the first kGAhead chunks is loaded while the MMAs
        // run; each chunk's reduction then loads the chunk kGAhead further on.
        float gq[kGAhead][16];
        if constexpr (!kPhilox) {
#pragma unroll
          for (int d = 0; d < kGAhead; ++d)
#pragma unroll
            for (int j = 0; j < 16; ++j) {
              const int cn = c_first + d * kStride + j;
              gq[d][j] = (noisy && valid && cn < R) ? __ldg(a.gumbel + (size_t)rmap[cn] * a.V + v) : 0.f;
            }
        }
        // the tcgen05.ld below is warp-collective: the warp goes on as a whole
        if (!__all_sync(0xffffffffu, mbar_wait(&tmem_full[acc], use & 1, a.err))) break;
        tc_fence_after();
        for (int c0 = c_first; c0 < R; c0 += kStride) {
          float g[16];
          if constexpr (!kPhilox) {
#pragma unroll
            for (int j = 0; j < 16; ++j) g[j] = gq[0][j];
#pragma unroll
            for (int d = 0; d + 1 < kGAhead; ++d)
#pragma unroll
              for (int j = 0; j < 16; ++j) gq[d][j] = gq[d + 1][j];
#pragma unroll
            for (int j = 0; j < 16; ++j) {
              const int cn = c0 + kGAhead * kStride + j;
              gq[kGAhead - 1][j] =
                  (noisy && valid && cn < R) ? __ldg(a.gumbel + (size_t)rmap[cn] * a.V + v) : 0.f;
            }
          } else if (noisy) {
            // lanes 4q .. 4q + 3 share one Philox counter per row: each lane
            // computes the calls of 4 of the chunk's 16 rows, and a 4 x 4
            // transpose inside the group gives every lane word v mod 4 of all 16
            const uint32_t vq = (uint32_t)v >> 2;
            const int i4 = lane & 3;
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              const int rr = c0 + 4 * q + i4;
              const uint32_t n = rr < R ? (uint32_t)rmap[rr] : 0u;
              const uint4 x = sbd_philox::philox4x32_10(make_uint4(vq, n, a.off_lo, a.off_hi),
                                                        a.seed_lo, a.seed_hi);
              uint32_t b[4] = {0u, 0u, 0u, 0u};
#pragma unroll
              for (int d = 0; d < 4; ++d) {
                const uint32_t send = sbd_philox::word_of(x, i4 ^ d);
                const uint32_t recv = d == 0 ? send : __shfl_xor_sync(0xffffffffu, send, d);
#pragma unroll
                for (int jj = 0; jj < 4; ++jj) b[jj] = (jj == (i4 ^ d)) ? recv : b[jj];
              }
#pragma unroll
              for (int jj = 0; jj < 4; ++jj) g[4 * q + jj] = sbd_philox::gumbel_of_word(b[jj]);
            }
          } else {
#pragma unroll
            for (int j = 0; j < 16; ++j) g[j] = 0.f;
          }
          uint32_t r[16];
          tc_ld_32x32b_x16(t_acc + (uint32_t)c0, r);
          tc_wait_ld();
          float z[16];
#pragma unroll
          for (int j = 0; j < 16; ++j) z[j] = __uint_as_float(r[j]);
          const RowStats cs = chunk16_stats(z, g, valid, a.tau, v0, lane);
          const int col = c0 + ((lane >> 1) & 15);
          if ((lane & 1) == 0 && col < R)
            store_stats(my_stats, col, rowstats_merge(load_stats(my_stats, col), cs));
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          if (rank == 1) mbar_arrive_cluster(at_rank0(&tmem_empty[acc]));
          else mbar_arrive(&tmem_empty[acc]);
        }
      }
      asm volatile("bar.sync 1, %0;" ::"n"(kEpiThreads) : "memory");
      for (int col = threadIdx.x - 64; col < R; col += kEpiThreads) {
        RowStats m4 = load_stats(wstats(0), col);
        for (int w = 1; w < 4; ++w) m4 = rowstats_merge(m4, load_stats(wstats(w), col));
        const size_t off = (size_t)blockIdx.x * a.rows_alloc + col;
        a.part_msTb[off] = make_float4(m4.m, m4.S, m4.T, m4.best);
        a.part_idx[off] = m4.idx;
      }
    }
  }
  // Partials of the live rows this CTA does not own (rows mode, or no work):
  // empty statistics (the combine merges every CTA's partial of every row).
  if (!kLinear && warp >= 2 && (rows_mode || !working)) {
    const RowStats e = rowstats_empty();
    for (int r = threadIdx.x - 64; r < R; r += kEpiThreads) {
      if (working && r >= row0 && r < row0 + kPairRows) continue;
      const size_t off = (size_t)blockIdx.x * a.rows_alloc + r;
      a.part_msTb[off] = make_float4(e.m, e.S, e.T, e.best);
      a.part_idx[off] = e.idx;
    }
  }
  tc_fence_before();
  __syncthreads();
  // neither CTA releases its tensor memory or leaves while the other may
  // still signal its barriers or read its shared memory
  pair_sync();
  if (warp == 1) {
    tc_fence_after();
    tc_dealloc_pair(tmem_base, 512);
  }
  pair_sync();
}

// ------------------------------------------------------------ fp32 SIMT
// One CTA per 128 vocab rows (thread = row) and the live hidden rows in
// groups of 32.  W and the group's hidden rows pass through shared memory in
// chunks of 32 columns, loaded coalesced, so each W element is read from
// global memory once per group; each thread keeps its 32 logits in
// registers.  Every logit is still the sequential fp32 FMA chain over H in
// ascending order (padding columns add 0 * 0).  The same column statistics
// as the tensor-core epilogue.
constexpr int kF32Cols = 32;
template <bool kPhilox>
__global__ void __launch_bounds__(128)
head_f32_kernel(const float* __restrict__ hidden_c, const float* __restrict__ w,
                const float* __restrict__ gumbel, const int32_t* __restrict__ row_map,
                const int32_t* __restrict__ n_rows, float tau, int V, int H, int rows_alloc,
                float4* __restrict__ part_msTb, int32_t* __restrict__ part_idx,
                uint4 philox_sk) {
  grid_dependency_wait();
  __shared__ float4 sm[4][32];
  __shared__ int si[4][32];
  __shared__ float w_s[128][kF32Cols + 1];   // +1: rows land in distinct banks
  __shared__ float h_s[32][kF32Cols];
  const int R = *n_rows;
  const int v0 = blockIdx.x * 128;
  const int v = v0 + threadIdx.x;
  const bool valid = v < V;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const bool noisy = tau != 0.f && (kPhilox || gumbel != nullptr);
  for (int r0 = 0; r0 < R; r0 += 32) {
    const int nr = min(32, R - r0);
    float zr[32];
#pragma unroll
    for (int j = 0; j < 32; ++j) zr[j] = 0.f;
    for (int c0 = 0; c0 < H; c0 += kF32Cols) {
      const int nc = min(kF32Cols, H - c0);
      __syncthreads();   // the previous chunk is consumed
      for (int e = threadIdx.x; e < 128 * kF32Cols; e += 128) {
        const int rr = e / kF32Cols, cc = e % kF32Cols;
        w_s[rr][cc] = (v0 + rr < V && cc < nc) ? w[(size_t)(v0 + rr) * H + c0 + cc] : 0.f;
      }
      for (int e = threadIdx.x; e < 32 * kF32Cols; e += 128) {
        const int jj = e / kF32Cols, cc = e % kF32Cols;
        h_s[jj][cc] = (jj < nr && cc < nc) ? hidden_c[(size_t)(r0 + jj) * H + c0 + cc] : 0.f;
      }
      __syncthreads();
#pragma unroll
      for (int j = 0; j < 32; ++j) {
        if (j < nr) {
          float acc = zr[j];
#pragma unroll 8
          for (int cc = 0; cc < kF32Cols; ++cc) acc = fmaf(h_s[j][cc], w_s[threadIdx.x][cc], acc);
          zr[j] = acc;
        }
      }
    }
    RowStats mine = rowstats_empty();
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      if (j >= nr) break;
      const float z = zr[j];
      float g = 0.f;
      if (noisy && valid) {
        if constexpr (kPhilox) {
          // philox_sk = (seed low, seed high, offset low, offset high)
          const uint4 x = sbd_philox::philox4x32_10(
              make_uint4((uint32_t)v >> 2, (uint32_t)row_map[r0 + j], philox_sk.z, philox_sk.w),
              philox_sk.x, philox_sk.y);
          g = sbd_philox::gumbel_of_word(sbd_philox::word_of(x, v & 3));
        } else {
          g = gumbel[(size_t)row_map[r0 + j] * V + v];
        }
      }
      const RowStats cs = warp_column_stats(z, valid, g, tau, v);
      if (lane == j) mine = cs;
    }
    if (lane < nr) {
      sm[warp][lane] = make_float4(mine.m, mine.S, mine.T, mine.best);
      si[warp][lane] = mine.idx;
    }
    __syncthreads();
    if (threadIdx.x < nr) {
      RowStats s;
      s.m = sm[0][threadIdx.x].x;
      s.S = sm[0][threadIdx.x].y;
      s.T = sm[0][threadIdx.x].z;
      s.best = sm[0][threadIdx.x].w;
      s.idx = si[0][threadIdx.x];
      for (int w2 = 1; w2 < 4; ++w2) {
        RowStats o;
        o.m = sm[w2][threadIdx.x].x;
        o.S = sm[w2][threadIdx.x].y;
        o.T = sm[w2][threadIdx.x].z;
        o.best = sm[w2][threadIdx.x].w;
        o.idx = si[w2][threadIdx.x];
        s = rowstats_merge(s, o);
      }
      const size_t o = (size_t)blockIdx.x * rows_alloc + r0 + threadIdx.x;
      part_msTb[o] = make_float4(s.m, s.S, s.T, s.best);
      part_idx[o] = s.idx;
    }
    __syncthreads();
  }
}

// ------------------------------------------------------------ combine
// One warp per masked row: merge the per-CTA statistics, then
// H = ln 2 * (log2 S - T / S)  (nats) and the winning token.  Latency-bound:
// the row count, the row map and up to 256 CTAs' statistics (8 per lane) are
// all requested before any of them is used.
__global__ void __launch_bounds__(128)
head_combine_kernel(const float4* __restrict__ part_msTb, const int32_t* __restrict__ part_idx,
                    int n_parts, int rows_alloc, const int32_t* __restrict__ row_map,
                    const int32_t* __restrict__ n_rows, float* __restrict__ entropy,
                    int32_t* __restrict__ token, float* __restrict__ confidence) {
  constexpr int kPerLane = 8;
  grid_dependency_wait();
  const int r = blockIdx.x * 4 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (r >= rows_alloc) return;
  const int rows = *n_rows;
  const int row = row_map[r];        // read before the check: r < rows_alloc
  RowStats s = rowstats_empty();
  for (int c0 = 0; c0 < n_parts; c0 += 32 * kPerLane) {
    float4 v[kPerLane];
    int id[kPerLane];
#pragma unroll
    for (int e = 0; e < kPerLane; ++e) {
      const int c = c0 + e * 32 + lane;
      if (c < n_parts) {
        v[e] = part_msTb[(size_t)c * rows_alloc + r];
        id[e] = part_idx[(size_t)c * rows_alloc + r];
      }
    }
#pragma unroll
    for (int e = 0; e < kPerLane; ++e) {
      if (c0 + e * 32 + lane < n_parts) {
        RowStats o;
        o.m = v[e].x;
        o.S = v[e].y;
        o.T = v[e].z;
        o.best = v[e].w;
        o.idx = id[e];
        s = rowstats_merge(s, o);
      }
    }
  }
  if (r >= rows) return;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    RowStats t;
    t.m = __shfl_xor_sync(0xffffffffu, s.m, o);
    t.S = __shfl_xor_sync(0xffffffffu, s.S, o);
    t.T = __shfl_xor_sync(0xffffffffu, s.T, o);
    t.best = __shfl_xor_sync(0xffffffffu, s.best, o);
    t.idx = __shfl_xor_sync(0xffffffffu, s.idx, o);
    s = rowstats_merge(s, t);
  }
  if (lane == 0) {
    entropy[row] = kLn2 * (log2f(s.S) - s.T / s.S);
    token[row] = s.idx;
    // the largest probability is the max term's: 2^0 / S
    if (confidence) confidence[row] = 1.f / s.S;
  }
}

// ------------------------------------------------------------ workspace
struct HeadWs {
  uint8_t* hidden_c;
  int32_t* row_map;
  int32_t* n_rows;
  float4* part_msTb;
  int32_t* part_idx;
  size_t bytes;
};

HeadWs head_ws_layout(const sbd::HeadPlan& p, void* base) {
  HeadWs w;
  const uintptr_t c = reinterpret_cast<uintptr_t>(base);
  size_t off = 0;
  const size_t elem = p.bf16 ? 2 : 4;
  w.hidden_c = reinterpret_cast<uint8_t*>(c + off);
  off = sbd::align_up(off + (size_t)p.rows_alloc * p.H * elem, 256);
  w.row_map = reinterpret_cast<int32_t*>(c + off);
  off = sbd::align_up(off + (size_t)p.rows_alloc * 4, 256);
  w.n_rows = reinterpret_cast<int32_t*>(c + off);
  off = sbd::align_up(off + 4, 256);
  w.part_msTb = reinterpret_cast<float4*>(c + off);
  off = sbd::align_up(off + (size_t)p.n_ctas * p.rows_alloc * sizeof(float4), 256);
  w.part_idx = reinterpret_cast<int32_t*>(c + off);
  off = sbd::align_up(off + (size_t)p.n_ctas * p.rows_alloc * 4, 256);
  w.bytes = off;
  return w;
}


// Shared memory of the ring: kRingBytes, within what a CTA can have next to
// the epilogue scratch.
int head_ring_bytes(int rows_alloc) {
  const int per_cta = 224 * 1024 - 1024 - 1024;
  int budget = kRingBytes;
  if (budget > per_cta - head_scratch_bytes(rows_alloc)) budget = per_cta - head_scratch_bytes(rows_alloc);
  return budget;
}

size_t head_smem_bytes(int rows_alloc) {
  return 1024 + (size_t)head_scratch_bytes(rows_alloc) + head_ring_bytes(rows_alloc);
}

// The LM head runs on CTA pairs (head_pair_kernel) from this many allocated
// rows, i.e. always (at 15 live rows it measured 161.1 us against 162.5 us
// for head_tc_kernel, which remains for a device that cannot hold a cluster
// of two and for a vocabulary of one tile); its shared memory is the ring
// alone.
constexpr int kPairMinRows = 16;
// its ring: what is left of the 227 KB of a CTA next to its static shared
// memory (barriers and 2.5 KB of row statistics) and the 1 KB alignment
constexpr int kPairRingBytes = 222 * 1024;
constexpr size_t kPairSmemBytes = 1024 + kPairRingBytes;

// How many clusters of two CTAs of `fn` the current device holds at once
// (0: none).  Kept per (device, kernel): the call is on every launch's host
// path.
int head_pair_slots(const void* fn) {
  struct Entry {
    int dev;
    const void* fn;
    int clusters;
  };
  static std::mutex mu;
  static Entry cache[16];
  static int n_cache = 0;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  {
    std::lock_guard<std::mutex> lock(mu);
    for (int i = 0; i < n_cache; ++i)
      if (cache[i].dev == dev && cache[i].fn == fn) return cache[i].clusters;
  }
  const int clusters =
      sbd::max_active_clusters(fn, dim3(2), dim3(kHeadThreads), kPairSmemBytes, 2);
  std::lock_guard<std::mutex> lock(mu);
  if (n_cache < 16) cache[n_cache++] = Entry{dev, fn, clusters};
  return clusters;
}

// y = the sum over K ranges of the fp32 partials of sbd_linear, in bf16.
__global__ void __launch_bounds__(256)
linear_reduce_kernel(const float* __restrict__ part, int ksplit, long long tn,
                     __nv_bfloat16* __restrict__ y) {
  grid_dependency_wait();
  grid_dependents_launch();
  const long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= tn) return;
  float acc = 0.f;
  for (int ks = 0; ks < ksplit; ++ks) acc += part[(size_t)ks * tn + i];
  y[i] = __float2bfloat16_rn(acc);
}

}  // namespace

namespace sbd {

HeadPlan head_plan(const sbd_head_desc& d) {
  HeadPlan p;
  p.B = d.batch;
  p.k = d.block_k;
  p.H = d.hidden;
  p.V = d.vocab;
  p.bf16 = d.dtype == SBD_DTYPE_BF16;
  const int bk = d.batch * d.block_k;
  p.rows_alloc = bk <= 16 ? 16 : ((bk + 15) / 16) * 16;
  const int n_tiles = (d.vocab + kBM - 1) / kBM;
  if (p.bf16) {
    const int slots = num_sms();
    p.n_ctas = n_tiles < slots ? n_tiles : slots;
  } else {
    p.n_ctas = n_tiles;
  }
  return p;
}

size_t head_workspace_bytes(const HeadPlan& p) { return head_ws_layout(p, nullptr).bytes; }

size_t head_workspace_floor(const sbd_head_desc& d) {
  if (d.batch < 0 || d.block_k < 1 || d.hidden < 1 || d.vocab < 1 ||
      (long long)d.batch * d.block_k > 512 ||
      (d.dtype != SBD_DTYPE_F32 && d.dtype != SBD_DTYPE_BF16))
    return 0;
  HeadPlan p;
  p.B = d.batch;
  p.k = d.block_k;
  p.H = d.hidden;
  p.V = d.vocab;
  p.bf16 = d.dtype == SBD_DTYPE_BF16;
  const int bk = d.batch * d.block_k;
  p.rows_alloc = bk <= 16 ? 16 : ((bk + 15) / 16) * 16;
  p.n_ctas = 1;
  return head_ws_layout(p, nullptr).bytes;
}

sbd_status head_launch(const HeadPlan& p, const void* hidden, const void* w,
                       const uint8_t* masked, const float* gumbel, float tau, float* entropy,
                       float* confidence, int32_t* token, void* ws, cudaStream_t st,
                       const PhiloxNoise* philox) {
  const int BK = p.B * p.k;
  if (BK == 0) return SBD_OK;
  HeadWs W = head_ws_layout(p, ws);
  const int elem = p.bf16 ? 2 : 4;
  sbd_status s;
  {
    const uint8_t* hid = (const uint8_t*)hidden;
    int bk = BK, rb = p.H * elem;
    uint8_t* hc = W.hidden_c;
    int32_t* rm = W.row_map;
    int32_t* nr = W.n_rows;
    void* args[] = {(void*)&hid, (void*)&masked,  (void*)&bk,    (void*)&rb,
                    (void*)&hc,  (void*)&rm,      (void*)&nr,    (void*)&entropy,
                    (void*)&token, (void*)&confidence};
    s = launch_pdl((const void*)compact_rows_kernel, dim3(p.rows_alloc), dim3(256), 0, st, args,
                   "compact_rows_kernel launch");
    if (s != SBD_OK) return s;
  }
  cudaError_t e;
  int* err = device_error_word();
  int n_parts = p.n_ctas;   // CTAs that write per-row partials
  if (p.bf16) {
    CUtensorMap tw, th, th64, th128;
    {
      const uint64_t dims[2] = {(uint64_t)p.H, (uint64_t)p.V};
      const uint64_t strides[1] = {(uint64_t)p.H * 2};
      const uint32_t box[2] = {(uint32_t)kBK, (uint32_t)kBM};
      s = encode_tensor_map(&tw, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, (void*)w, dims, strides,
                            box, CU_TENSOR_MAP_SWIZZLE_128B);
      if (s != SBD_OK) return s;
    }
    {
      const uint64_t dims[2] = {(uint64_t)p.H, (uint64_t)p.rows_alloc};
      const uint64_t strides[1] = {(uint64_t)p.H * 2};
      const uint32_t box[2] = {(uint32_t)kBK, 16u};
      s = encode_tensor_map(&th, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, (void*)W.hidden_c, dims,
                            strides, box, CU_TENSOR_MAP_SWIZZLE_128B);
      if (s != SBD_OK) return s;
      th64 = th;
      th128 = th;
      if (p.rows_alloc >= 64) {
        const uint32_t box64[2] = {(uint32_t)kBK, 64u};
        s = encode_tensor_map(&th64, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, (void*)W.hidden_c, dims,
                              strides, box64, CU_TENSOR_MAP_SWIZZLE_128B);
        if (s != SBD_OK) return s;
      }
      if (p.rows_alloc >= 128) {
        const uint32_t box128[2] = {(uint32_t)kBK, 128u};
        s = encode_tensor_map(&th128, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, (void*)W.hidden_c,
                              dims, strides, box128, CU_TENSOR_MAP_SWIZZLE_128B);
        if (s != SBD_OK) return s;
      }
    }
    HeadArgs a;
    a.gumbel = gumbel;
    a.seed_lo = philox ? (uint32_t)philox->seed : 0u;
    a.seed_hi = philox ? (uint32_t)(philox->seed >> 32) : 0u;
    a.off_lo = philox ? (uint32_t)philox->offset : 0u;
    a.off_hi = philox ? (uint32_t)(philox->offset >> 32) : 0u;
    a.row_map = W.row_map;
    a.n_rows = W.n_rows;
    a.part_msTb = W.part_msTb;
    a.part_idx = W.part_idx;
    a.err = err;
    a.V = p.V;
    a.H = p.H;
    a.rows_alloc = p.rows_alloc;
    a.n_tiles = (p.V + kBM - 1) / kBM;
    a.y = nullptr;
    a.linear_rows = 0;
    a.ksplit = 1;
    a.part_y = nullptr;
    a.h_big = p.rows_alloc >= 128 ? 128 : (p.rows_alloc >= 64 ? 64 : 16);
    a.tau = tau;
    // CTA pairs from kPairMinRows allocated rows: as many as the device holds
    // at once, the pair tiles need and the workspace has partials for
    // (p.n_ctas), an even number when there may be two row groups.
    const void* fn_pair = philox ? (const void*)head_pair_kernel<true, false>
                                 : (const void*)head_pair_kernel<false, false>;
    const int pair_tiles = (p.V + 2 * kBM - 1) / (2 * kBM);
    const int n_groups_max = p.rows_alloc > 2 * kPairRows ? 2 : 1;
    int n_pairs = 0;
    if (p.rows_alloc >= kPairMinRows && p.n_ctas >= 2) {
      n_pairs = head_pair_slots(fn_pair);
      if (n_pairs > pair_tiles * n_groups_max) n_pairs = pair_tiles * n_groups_max;
      if (n_pairs > p.n_ctas / 2) n_pairs = p.n_ctas / 2;
      if (n_groups_max == 2) n_pairs &= ~1;
    }
    const void* fn;
    size_t smem;
    if (n_pairs > 0) {
      fn = fn_pair;
      smem = kPairSmemBytes;
      a.ring_bytes = kPairRingBytes;
      a.n_tiles = pair_tiles;
      a.tmem_cols = 512;
      n_parts = 2 * n_pairs;
    } else {
      fn = philox ? (const void*)head_tc_kernel<true, false> : (const void*)head_tc_kernel<false, false>;
      smem = head_smem_bytes(p.rows_alloc);
      a.ring_bytes = head_ring_bytes(p.rows_alloc);
      // tensor memory for two accumulators of the allocated width (one of it
      // above 256 rows); the kernel picks the buffer count from the live rows
      const int n_acc_alloc = 2 * p.rows_alloc <= 512 ? 2 : 1;
      uint32_t cols = 32;
      while (cols < (uint32_t)(n_acc_alloc * p.rows_alloc)) cols <<= 1;
      a.tmem_cols = cols;
    }
    e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return cuda_fail(e, "cudaFuncSetAttribute(LM head kernel)");
    void* args[] = {(void*)&tw, (void*)&th, (void*)&th64, (void*)&th128, (void*)&a};
    s = launch_pdl(fn, dim3(n_parts), dim3(kHeadThreads), smem, st, args,
                   n_pairs > 0 ? "head_pair_kernel launch" : "head_tc_kernel launch",
                   n_pairs > 0 ? 2 : 1);
    if (s != SBD_OK) return s;
  } else {
    const float* hc = (const float*)W.hidden_c;
    const float* wf = (const float*)w;
    const int32_t* rm = W.row_map;
    const int32_t* nr = W.n_rows;
    int V = p.V, H = p.H, ra = p.rows_alloc;
    float4* pm = W.part_msTb;
    int32_t* pi = W.part_idx;
    uint4 sk = make_uint4(0u, 0u, 0u, 0u);
    if (philox)
      sk = make_uint4((uint32_t)philox->seed, (uint32_t)(philox->seed >> 32),
                      (uint32_t)philox->offset, (uint32_t)(philox->offset >> 32));
    void* args[] = {(void*)&hc, (void*)&wf, (void*)&gumbel, (void*)&rm, (void*)&nr,
                    (void*)&tau, (void*)&V,  (void*)&H,      (void*)&ra, (void*)&pm,
                    (void*)&pi, (void*)&sk};
    const void* fn =
        philox ? (const void*)head_f32_kernel<true> : (const void*)head_f32_kernel<false>;
    s = launch_pdl(fn, dim3(p.n_ctas), dim3(128), 0, st, args, "head_f32_kernel launch");
    if (s != SBD_OK) return s;
  }
  {
    const float4* pm = W.part_msTb;
    const int32_t* pi = W.part_idx;
    int np = n_parts, ra = p.rows_alloc;
    const int32_t* rm = W.row_map;
    const int32_t* nr = W.n_rows;
    void* args[] = {(void*)&pm, (void*)&pi, (void*)&np,      (void*)&ra,   (void*)&rm,
                    (void*)&nr, (void*)&entropy, (void*)&token, (void*)&confidence};
    s = launch_pdl((const void*)head_combine_kernel, dim3((p.rows_alloc + 3) / 4), dim3(128), 0,
                   st, args, "head_combine_kernel launch");
    if (s != SBD_OK) return s;
  }
  return SBD_OK;
}

// y[T, N] = x[T, K] W[N, K]^T in bf16 with fp32 accumulation: the LM-head
// kernel's main loop (W streamed once through the ring, x's rows from L2)
// with a storing epilogue.
// The largest K split sbd_linear may use: powers of two up to 16, each K
// range at least 4 column blocks long, at most 512 (tile, range) units and
// at most 64 MB of fp32 partials.  A function of the shape only, so that
// the workspace size does not depend on the device.
static int linear_max_split(int T, int K, int N) {
  const int kb64 = K / kBK, n_tiles = (N + kBM - 1) / kBM;
  int ks = 1;
  while (ks < 16 && kb64 % (2 * ks) == 0 && kb64 / (2 * ks) >= 4 &&
         (long long)n_tiles * 2 * ks <= 512 &&
         (long long)2 * ks * T * N * (long long)sizeof(float) <= (64ll << 20))
    ks *= 2;
  return ks;
}

int linear_ksplit(int T, int K, int N) {
  // A time model per SM: a tile streams its 128 x K weights (~45 GB/s per
  // SM at the HBM peak) or runs its 2 x 128 x n x K flops (~14.8 TFLOP/s
  // per SM), whichever is longer; a unit of a split also writes its
  // T x 128 fp32 partials, and the sum over ranges reads them all back in
  // a second launch.  The split with the shortest modelled time wins.
  const int max_ks = linear_max_split(T, K, N);
  const int sms = num_sms();
  const int n_tiles = (N + kBM - 1) / kBM;
  const double n_eff = T <= 16 ? 16.0 : (double)((T + 15) / 16 * 16);
  const double t_mem = 128.0 * K * 2 / 45e3, t_mma = 2.0 * 128 * n_eff * K / 14.8e6;  // us
  const double t_tile = t_mem > t_mma ? t_mem : t_mma;
  const double t_part = (double)T * 128 * 4 / 45e3;
  int best = 1;
  double best_cost = (double)((n_tiles + sms - 1) / sms) * t_tile;
  for (int ks = 2; ks <= max_ks; ks *= 2) {
    const double waves = (double)((n_tiles * ks + sms - 1) / sms);
    const double cost = waves * (t_tile / ks + t_part) + (double)ks * T * N * 4 / 6e6 + 2.0;
    if (cost < best_cost) {
      best_cost = cost;
      best = ks;
    }
  }
  return best;
}

// K ranges for the CTA-pair linear (rows layout): the same kind of time
// model per pair of SMs.  A unit streams 128 W rows x K / ks per SM
// (~45 GB/s per SM at the HBM peak) or runs K / (16 ks) 2-SM MMAs of
// ~65 ns, whichever is longer; with ranges it also writes its rows' fp32
// partials, and the sum over ranges reads them all back in a second launch.
// At most linear_max_split (what the workspace holds).
static int pair_linear_ksplit(int T, int K, int N, int n_pairs) {
  const int max_ks = linear_max_split(T, K, N);
  const int pair_tiles = (N + 2 * kBM - 1) / (2 * kBM);
  const int n_groups = T > 2 * kPairRows ? 2 : 1;
  const int per_group = n_pairs / n_groups > 0 ? n_pairs / n_groups : 1;
  const double t_mem = 128.0 * K * 2 / 45e3, t_mma = K / 16.0 * 0.065;   // us
  const double t_unit = t_mem > t_mma ? t_mem : t_mma;
  const int rows_cta = (T < 2 * kPairRows ? T : 2 * kPairRows) / 2;
  const double t_part = (double)rows_cta * 2 * kBM * 4 / 45e3;
  int best = 1;
  double best_cost = (double)((pair_tiles + per_group - 1) / per_group) * t_unit;
  for (int ks = 2; ks <= max_ks; ks *= 2) {
    const double waves = (double)((pair_tiles * ks + per_group - 1) / per_group);
    const double cost = waves * (t_unit / ks + t_part) + (double)ks * T * N * 4 / 6e6 + 2.0;
    if (cost < best_cost) {
      best_cost = cost;
      best = ks;
    }
  }
  return best;
}

size_t linear_workspace_bytes(int T, int K, int N) {
  const int ks = linear_max_split(T, K, N);
  return ks > 1 ? (size_t)ks * T * N * sizeof(float) : 0;
}

sbd_status linear_launch(int T, int K, int N, const void* x, const void* w, void* y, void* ws,
                         cudaStream_t st) {
  if (T == 0 || N == 0) return SBD_OK;
  const int rows_alloc = T <= 16 ? 16 : ((T + 15) / 16) * 16;
  CUtensorMap tw, tx, tx64, tx128;
  sbd_status s;
  {
    const uint64_t dims[2] = {(uint64_t)K, (uint64_t)N};
    const uint64_t strides[1] = {(uint64_t)K * 2};
    const uint32_t box[2] = {(uint32_t)kBK, (uint32_t)kBM};
    s = encode_tensor_map(&tw, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, (void*)w, dims, strides, box,
                          CU_TENSOR_MAP_SWIZZLE_128B);
    if (s != SBD_OK) return s;
  }
  {
    // rows of x past T (up to the MMA's multiple of 16) are read as zeros
    const uint64_t dims[2] = {(uint64_t)K, (uint64_t)T};
    const uint64_t strides[1] = {(uint64_t)K * 2};
    const uint32_t box[2] = {(uint32_t)kBK, 16u};
    s = encode_tensor_map(&tx, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, (void*)x, dims, strides, box,
                          CU_TENSOR_MAP_SWIZZLE_128B);
    if (s != SBD_OK) return s;
    tx64 = tx;
    tx128 = tx;
    if (T >= 64) {
      const uint32_t box64[2] = {(uint32_t)kBK, 64u};
      s = encode_tensor_map(&tx64, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, (void*)x, dims, strides,
                            box64, CU_TENSOR_MAP_SWIZZLE_128B);
      if (s != SBD_OK) return s;
    }
    if (T >= 128) {
      const uint32_t box128[2] = {(uint32_t)kBK, 128u};
      s = encode_tensor_map(&tx128, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, (void*)x, dims, strides,
                            box128, CU_TENSOR_MAP_SWIZZLE_128B);
      if (s != SBD_OK) return s;
    }
  }
  HeadArgs a{};
  a.err = device_error_word();
  a.V = N;
  a.H = K;
  a.rows_alloc = rows_alloc;
  a.n_tiles = (N + kBM - 1) / kBM;
  a.h_big = T >= 128 ? 128 : (T >= 64 ? 64 : 16);
  a.tau = 0.f;
  a.y = (__nv_bfloat16*)y;
  a.linear_rows = T;
  a.part_y = (float*)ws;
  // Above the pair kernel's vocabulary-lane limit: CTA pairs in the rows
  // layout, as many as the device holds at once and the units need (an
  // even number with two row groups), with their own choice of K ranges.
  int ksplit = linear_ksplit(T, K, N);
  const void* fn = nullptr;
  int n_ctas = 0, cluster = 1;
  size_t smem = 0;
  if (T > kPairVocabLanesMax) {
    const void* fn_pair = (const void*)head_pair_kernel<false, true>;
    const int pair_tiles = (N + 2 * kBM - 1) / (2 * kBM);
    const int n_groups = T > 2 * kPairRows ? 2 : 1;
    int n_pairs = head_pair_slots(fn_pair);
    if (n_groups == 2) n_pairs &= ~1;
    if (n_pairs > 0) {
      const int ks = pair_linear_ksplit(T, K, N, n_pairs);
      if (n_pairs > pair_tiles * n_groups * ks) n_pairs = pair_tiles * n_groups * ks;
      if (n_groups == 2) n_pairs &= ~1;
      if (n_pairs > 0) {
        ksplit = ks;
        fn = fn_pair;
        n_ctas = 2 * n_pairs;
        cluster = 2;
        smem = kPairSmemBytes;
        a.n_tiles = pair_tiles;
        a.ring_bytes = kPairRingBytes;
        a.tmem_cols = 512;
      }
    }
  }
  if (!fn) {
    fn = (const void*)head_tc_kernel<false, true>;
    smem = head_smem_bytes(rows_alloc);
    a.ring_bytes = head_ring_bytes(rows_alloc);
    const int n_acc_alloc = 2 * rows_alloc <= 512 ? 2 : 1;
    uint32_t cols = 32;
    while (cols < (uint32_t)(n_acc_alloc * rows_alloc)) cols <<= 1;
    a.tmem_cols = cols;
    const int slots = num_sms();
    const int units = a.n_tiles * ksplit;
    n_ctas = units < slots ? units : slots;
  }
  a.ksplit = ksplit;
  cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return cuda_fail(e, "cudaFuncSetAttribute(linear kernel)");
  void* args[] = {(void*)&tw, (void*)&tx, (void*)&tx64, (void*)&tx128, (void*)&a};
  s = launch_pdl(fn, dim3(n_ctas), dim3(kHeadThreads), smem, st, args,
                 cluster > 1 ? "head_pair_kernel (linear) launch" : "head_tc_kernel (linear) launch",
                 cluster);
  if (s != SBD_OK || ksplit == 1) return s;
  const float* part = (const float*)ws;
  long long tn = (long long)T * N;
  __nv_bfloat16* yb = (__nv_bfloat16*)y;
  int ks = ksplit;
  void* rargs[] = {(void*)&part, (void*)&ks, (void*)&tn, (void*)&yb};
  return launch_pdl((const void*)linear_reduce_kernel, dim3((unsigned)((tn + 255) / 256)), dim3(256),
                    0, st, rargs, "linear_reduce_kernel launch");
}

}  // namespace sbd
