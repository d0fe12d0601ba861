// Block attention on the tcgen05 tensor cores (arXiv 2509.04185, Eq. 5;
// inference mask of Fig. 3) for bf16 inputs.
//
// One CTA per (KV split, KV head, sequence), the G query heads of a KV head
// packed with the k block rows into one row tile (row r = i*G + g, padded to
// 128); both products run on tcgen05 with their accumulators in tensor
// memory.  Keys stream in tiles
// of 64 (one TMA stage each) and the products run on pairs of tiles:
//
//   S_q = Q K_q^T     A = Q (shared, K-major), B = the pair's K (shared,
//                     K-major), M = 128 rows, N = 128 keys, fp32 in TMEM
//                     (2 buffers);
//   O  += P_q V_q     A = P_q (bf16, shared, K-major), B = the pair's V
//                     (shared, MN-major: keys are K, head dims N), fp32 O in
//                     TMEM.
//
// Pairs, not single tiles: an M = 128, K = 16 tcgen05.mma measured about the
// same time for N = 64, 128 and 256 (~135 cycles), so 64-key score products
// left the tensor pipe the bottleneck (1300 cycles of MMA per 64 keys; 760
// with 128-key pairs).  The two tiles of a pair sit back to back in every
// 128-byte sub-tile of the ring, so that they form one 128-row operand.
//
// Warp roles: warp 0 streams K/V tiles with TMA (a ring of 3 pairs), the k
// block keys/values included (the last tile of the last split); warp 1
// owns the tensor memory and one thread issues the MMAs, computing S_{q+1}
// while the softmax of pair q runs; warps 2-9 are the softmax, two per TMEM
// lane quadrant (and, with 64 packed rows or fewer, each row copied to a
// second quadrant, so that four warps share a row): a thread reads its share
// of a row's 128 scores with tcgen05.ld, applies the mask (cache key < L_b,
// block key < k, or j <= i for a causal block row i < n_causal) and the
// scale, and writes its part of P_q = 2^(s - m_ref) as bf16 into shared
// memory.  The warps sharing a row agree on the pair's row maximum through a
// shared-memory exchange.  The reference max m_ref only moves (and O is
// rescaled in tensor memory) when the running max exceeds it by more than
// 2^8, which keeps every P entry <= 256; l and O use the same reference, so
// the result is exact.  The epilogue normalises O by l and writes the output
// (one split) or the split partial and its log-sum-exp.
#include <math.h>

#include <mutex>

#include "sbd_internal.cuh"

namespace {

using namespace sbd_dev;

constexpr int kTileKeys = 64;              // keys per TMA stage
constexpr int kPairKeys = 2 * kTileKeys;   // keys per MMA step (two stages)
constexpr int kMaxStages = 8;
constexpr int kMaxPairs = kMaxStages / 2;
constexpr int kRows = 128;                 // MMA M (packed rows, padded)
constexpr int kSoftWarps = 8;              // two per TMEM lane quadrant
constexpr int kThreads = 64 + 32 * kSoftWarps;   // producer, MMA, softmax warps
constexpr float kRescaleThreshold = 8.f;   // log2 units

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
__device__ __forceinline__ void tc_mma(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                       uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// The same with the A operand read from tensor memory (M = 128 lanes, K
// packed as bf16 pairs along the columns).
__device__ __forceinline__ void tc_mma_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc,
                                          uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void tc_commit(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
          smem_u32(bar))
      : "memory");
}
__device__ __forceinline__ void tc_ld16(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
}
__device__ __forceinline__ void tc_st16(uint32_t taddr, const uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
      "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
      "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]),
      "r"(r[15])
      : "memory");
}
__device__ __forceinline__ void tc_wait_ld() {
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tc_wait_st() {
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

// Shared-memory descriptor of a 128-byte-swizzled operand: lbo/sbo in bytes.
// K-major: rows 128 B apart, 8-row groups `sbo` apart (lbo unused).
// MN-major: 64-element atoms along MN `lbo` apart, 8-row groups along K
// `sbo` apart.
__device__ __forceinline__ uint64_t sw128_desc(uint32_t addr, uint32_t lbo, uint32_t sbo) {
  uint64_t d = 0;
  d |= (uint64_t)((addr & 0x3FFFFu) >> 4);
  d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
  d |= (uint64_t)((sbo >> 4) & 0x3FFFu) << 32;
  d |= (uint64_t)1u << 46;
  d |= (uint64_t)2u << 61;
  return d;
}
// kind::f16 instruction descriptor: bf16 A and B, fp32 D; b_mn = B is MN-major.
__device__ __forceinline__ uint32_t idesc_bf16(int M, int N, bool b_mn) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((b_mn ? 1u : 0u) << 16) |
         ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

// ------------------------------------------------------------ clusters
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\t"
               "barrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
// The address of this CTA's shared-memory location `addr` in CTA `rank` of
// the cluster.
__device__ __forceinline__ uint32_t mapa_shared(uint32_t addr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
  return r;
}
__device__ __forceinline__ float ld_cluster_f32(uint32_t addr) {
  float v;
  asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(addr) : "memory");
  return v;
}
__device__ __forceinline__ float4 ld_cluster_v4(uint32_t addr) {
  float4 v;
  asm volatile("ld.shared::cluster.v4.f32 {%0,%1,%2,%3}, [%4];"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "r"(addr)
               : "memory");
  return v;
}
__device__ __forceinline__ float2 ld_cluster_v2(uint32_t addr) {
  float2 v;
  asm volatile("ld.shared::cluster.v2.f32 {%0,%1}, [%2];" : "=f"(v.x), "=f"(v.y) : "r"(addr) : "memory");
  return v;
}

// Address of (row, 16-byte chunk c) inside a [rows x 128 B] swizzled tile.
__device__ __forceinline__ uint32_t swz(uint32_t base, int row, int chunk) {
  return base + row * 128 + (((chunk ^ (row & 7)) & 7) << 4);
}
__device__ __forceinline__ void st_shared_v4(uint32_t addr, uint4 v) {
  asm volatile("st.shared.v4.b32 [%0], {%1,%2,%3,%4};" ::"r"(addr), "r"(v.x), "r"(v.y), "r"(v.z),
               "r"(v.w)
               : "memory");
}
// bf16 bit pattern of the smallest bf16 >= x (x not NaN), and back.
__device__ __forceinline__ uint16_t bf16_bits_round_up(float x) {
  const uint32_t u = __float_as_uint(x);
  const bool neg = (u >> 31) != 0;
  // positive: round the magnitude up; negative: truncate the magnitude
  return (uint16_t)((neg ? u : u + 0xFFFFu) >> 16);
}
__device__ __forceinline__ float bf16_bits_to_float(uint16_t b) {
  return __uint_as_float((uint32_t)b << 16);
}
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

struct TcArgs {
  const __nv_bfloat16* q;
  const __nv_bfloat16* kb;
  const __nv_bfloat16* vb;
  const int32_t* lens;
  __nv_bfloat16* out;
  float* part_o;
  float* part_lse;
  int* err;
  __nv_bfloat16* kc_app;     // writable caches for the causal rows' keys/values, or NULL
  __nv_bfloat16* vc_app;
  int B, k, Hq, Hkv, G, M, Lmax, splits, n_causal;
  int order;                 // blockIdx.z -> sequence by descending length
  int cluster;               // the splits of a (sequence, KV head) form one cluster and
                             // merge their partials in shared memory (no part_o / part_lse)
  float scale_log2;
};

// ------------------------------------------------ merge in the cluster
// The CTAs of a cluster are the splits of one (sequence, KV head), each
// holding its normalised partial rows (cpart_s: kRows x (D + 4) floats) and
// their log2-sum-exps (after them) in shared memory.  After a cluster
// barrier every CTA's partials are visible to the others; CTA `rank` merges
// rows rank, rank + S, ... (softmax warp sw takes one row at a time, lane s
// reading split s's log2-sum-exp, D / 32 columns a lane) and writes them
// out; a second barrier keeps every CTA's shared memory alive until the
// others have read it.  All threads of every CTA reach both barriers: no
// role leaves the kernel early, and every wait before them is bounded.
template <int D>
__device__ __forceinline__ void cluster_merge(const TcArgs& a, int b, int hkv, uint32_t cpart_s,
                                              int sw, int lane) {
  cluster_sync_all();
  if (sw >= 0 && sw < kSoftWarps) {
    constexpr int kCStride = D + 4;
    constexpr int kPer = D / 32;
    const uint32_t clse_s = cpart_s + (uint32_t)(kRows * kCStride * 4);
    const int S = a.splits;
    const int rank = (int)cluster_ctarank();
    for (int r = rank + S * sw; r < a.M; r += S * kSoftWarps) {
      const float l = lane < S ? ld_cluster_f32(mapa_shared(clse_s + 4u * r, lane)) : -INFINITY;
      const float gm = warp_max(l);
      const float w = (lane < S && gm != -INFINITY) ? exp2f(l - gm) : 0.f;
      const float wsum = warp_sum(w);
      float v[16][kPer];
#pragma unroll
      for (int s2 = 0; s2 < 16; ++s2) {
        if (s2 < S) {
          const uint32_t src = mapa_shared(cpart_s + 4u * (r * kCStride + kPer * lane), s2);
          if constexpr (kPer == 4) {
            const float4 x = ld_cluster_v4(src);
            v[s2][0] = x.x; v[s2][1] = x.y; v[s2][2] = x.z; v[s2][3] = x.w;
          } else {
            const float2 x = ld_cluster_v2(src);
            v[s2][0] = x.x; v[s2][1] = x.y;
          }
        }
      }
      float acc[kPer];
#pragma unroll
      for (int c = 0; c < kPer; ++c) acc[c] = 0.f;
#pragma unroll
      for (int s2 = 0; s2 < 16; ++s2) {
        const float ws = __shfl_sync(0xffffffffu, w, s2);    // 0 past S
        if (s2 < S && ws > 0.f) {
#pragma unroll
          for (int c = 0; c < kPer; ++c) acc[c] = fmaf(ws, v[s2][c], acc[c]);
        }
      }
      const float inv = wsum > 0.f ? 1.f / wsum : 0.f;
      __nv_bfloat16* dst =
          a.out + (((size_t)b * a.k + r / a.G) * a.Hq + hkv * a.G + r % a.G) * D + kPer * lane;
      if constexpr (kPer == 4) {
        uint2 o2;
        o2.x = pack_bf16(acc[0] * inv, acc[1] * inv);
        o2.y = pack_bf16(acc[2] * inv, acc[3] * inv);
        *reinterpret_cast<uint2*>(dst) = o2;
      } else {
        *reinterpret_cast<uint32_t*>(dst) = pack_bf16(acc[0] * inv, acc[1] * inv);
      }
    }
  }
  cluster_sync_all();
}

// Softmax work split over the 128 columns of a pair.  R = 1: packed row r
// lives in TMEM lane r, and the two warps of its lane quadrant take 64 of the
// pair's 128 columns each (one tile each).  R = 2 (M <= 64): rows are also
// copied to lanes 64 + r (the MMA pads to 128 rows anyway), so four warps on
// all four SM sub-partitions share a row, 32 columns each: copy 0 (lanes
// 0-63) takes the pair's first tile, copy 1 (lanes 64-127) the second.  The
// warps sharing a row exchange their partial maxima through shared memory at
// a named barrier and take identical decisions.
//
// PV with R = 2.  A tcgen05.mma of M = 128 and K = 16 costs nearly as much
// at N = 128 as at N = 256 (47.6 against 65.4 ns of throughput on GB300),
// and the MMAs lie on the chain S -> softmax -> P -> PV, so N = D would pay
// almost a full instruction for half its work.  Each copy of a row
// therefore accumulates its own tile only: lane r of P holds the row's
// probabilities over the keys of its copy's tile, and one instruction with
// B = [V of 16 keys of tile 0 | V of the same 16 rows of tile 1] (N = 2 D)
// adds P_copy0 V_tile0 to columns
// [0, D) and P_copy1 V_tile1 to columns [D, 2 D) of O (the other two blocks
// of the product land in columns no lane reads).  4 instructions per pair
// instead of 8; the two partial sums of a row are added in the epilogue.
template <int D, int R>
__global__ void __launch_bounds__(kThreads, 1)
attn_tc_kernel(const __grid_constant__ CUtensorMap tmap_k,
               const __grid_constant__ CUtensorMap tmap_v,
               const __grid_constant__ CUtensorMap tmap_kb,
               const __grid_constant__ CUtensorMap tmap_vb, const TcArgs a) {
  constexpr int kSub = D / 64;                     // 128-B column sub-tiles of a key row
  constexpr int kQBytes = kRows * 128;             // one Q (or P) sub-tile: 16 KB
  constexpr int kKVSub = kTileKeys * 128;          // one tile's K or V sub-tile: 8 KB
  constexpr int kPairSub = 2 * kKVSub;             // a pair's K or V sub-tile: 16 KB
  constexpr int kPairBytes = 2 * kSub * kPairSub;  // K sub-tiles then V sub-tiles
  constexpr uint32_t kTmemCols = 512;              // S0 | S1 (128 each) | O (R * D)
  constexpr uint32_t kOCol = 2 * kPairKeys;
  static_assert(R == 1 || R == 2, "row copies");
  static_assert(kOCol + R * D <= kTmemCols, "O fits the allocation");
  // With D = 128 the K region of a pair (32 KB) is exactly a P block, and K is
  // dead once S of the pair is computed: P is written there, and the ring gets
  // the shared memory separate P buffers would take.
  constexpr bool kPInK = D == 128;
  constexpr int kPairs = kPInK ? 3 : 4;            // ring depth in pairs
  constexpr int kStages = 2 * kPairs;              // ring depth in 64-key tiles
  static_assert(kQBytes == kPairSub, "a P sub-tile fills a pair's K sub-tile");

  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t kv_full[kMaxStages], kv_empty[kMaxPairs];
  __shared__ __align__(8) uint64_t s_full[2], s_free[2], p_full[2], pv_done[2];
  __shared__ __align__(8) uint64_t q_ready, tail_bar;
  __shared__ uint32_t tmem_base_sh;
  // Exchange buffer of the softmax warps: partial row maxima as bf16 rounded
  // up ([pair parity][warp][lane]), then, at the end, fp32 partial row sums
  // ([warp][lane]).  1 KB: the ring and Q take the rest of the 227 KB.
  __shared__ __align__(16) uint32_t red_buf[kSoftWarps * 32];
  uint16_t* red_max = reinterpret_cast<uint16_t*>(red_buf);
  float* red_l = reinterpret_cast<float*>(red_buf);

  const uint32_t sbase = (smem_u32(smem_raw) + 1023u) & ~1023u;
  const uint32_t q_s = sbase;                              // kSub x 16 KB
  const uint32_t p_s = q_s + kSub * kQBytes;               // 2 x 32 KB unless kPInK
  const uint32_t kv_s = p_s + (kPInK ? 0 : 4 * kQBytes);   // kPairs x kPairBytes
  // Tile j of this split lives in pair slot (j / 2) mod kPairs, half j mod 2.
  // K: the two tiles of a pair sit back to back in every sub-tile, so that a
  // pair's keys form one 128-row operand of S.  V: the sub-tiles are ordered
  // (tile 0, columns 0-63), (tile 0, 64-127), (tile 1, 0-63), (tile 1,
  // 64-127), 8 KB apart, so that the D columns of one tile, or of both tiles
  // side by side, form one MN-major operand of PV with a constant stride.
  auto k_chunk = [&](int j, int h) -> uint32_t {
    return kv_s + ((j >> 1) % kPairs) * kPairBytes + h * kPairSub + (j & 1) * kKVSub;
  };
  auto v_chunk = [&](int j, int h) -> uint32_t {
    return kv_s + ((j >> 1) % kPairs) * kPairBytes + kSub * kPairSub + ((j & 1) * kSub + h) * kKVSub;
  };
  // P block of pair q: R = 1, two 16 KB sub-tiles (keys 0-63, 64-127); R = 2,
  // one sub-tile whose row r holds lane r's keys (its copy's tile)
  auto p_block = [&](int q) -> uint32_t {
    return kPInK ? k_chunk(2 * q, 0) : p_s + (q & 1) * 2 * kQBytes;
  };

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int split = blockIdx.x, hkv = blockIdx.y;
  __shared__ int b_pick;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) mbar_init(&kv_full[s], 1);
    for (int s = 0; s < kPairs; ++s) mbar_init(&kv_empty[s], 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&s_full[i], 1);
      mbar_init(&s_free[i], kSoftWarps);      // one arrival per softmax warp
      mbar_init(&p_full[i], kSoftWarps);
      mbar_init(&pv_done[i], 1);
    }
    mbar_init(&q_ready, kSoftWarps);
    mbar_init(&tail_bar, 1);
    fence_mbar_init();
  }
  // All 512 tensor-memory columns are taken only after the previous grid is
  // done, so that no CTA of it can be left waiting for them.
  grid_dependency_wait();
  if (a.order) {
    longest_first_pick(a.lens, a.B, a.Lmax, blockIdx.z, &b_pick);
    __syncthreads();
  }
  const int b = a.order ? b_pick : (int)blockIdx.z;
  if (warp == 1) tc_alloc(&tmem_base_sh, kTmemCols);

  int len = a.lens[b];
  if (len < 0 || len > a.Lmax) {
    if (threadIdx.x == 0 && split == 0 && hkv == 0) record_error(a.err, SBD_DEVERR_CACHE_LEN);
    len = len < 0 ? 0 : a.Lmax;
  }
  const int n_cache_tiles = (len + kTileKeys - 1) / kTileKeys;
  const int n_tiles = n_cache_tiles + 1;
  const int t_begin = (int)((long long)split * n_tiles / a.splits);
  const int t_end = (int)((long long)(split + 1) * n_tiles / a.splits);
  const int n = t_end - t_begin;                  // 64-key tiles of this split
  const int np = (n + 1) / 2;                     // pairs (the last may hold one tile)

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base_sh;

  if (warp == 0) {
    // ------------------------------------------------ producer warp
    if (lane == 0) {
      tma_prefetch_desc(&tmap_k);
      tma_prefetch_desc(&tmap_v);
      if (t_end == n_tiles) {
        tma_prefetch_desc(&tmap_kb);
        tma_prefetch_desc(&tmap_vb);
      }
    }
    for (int j = 0; j < n; ++j) {
      const int t = t_begin + j;
      const int stage = j % kStages;
      // a pair slot is reused once the PV product of its previous pair is done
      if ((j & 1) == 0) {
        const int q = j >> 1;
        const bool freed = mbar_wait(&kv_empty[q % kPairs], ((q / kPairs) & 1) ^ 1, a.err);
        if (!__all_sync(0xffffffffu, freed)) break;
      }
      if (t < n_cache_tiles) {
        const int valid = min(kTileKeys, len - t * kTileKeys);
        const bool tail = valid < kTileKeys;
        uint64_t* bar = tail ? &tail_bar : &kv_full[stage];
        if (lane == 0) {
          mbar_arrive_expect_tx(bar, 2 * kSub * kKVSub);
          for (int h = 0; h < kSub; ++h) {
            tma_load_4d(smem_raw + (k_chunk(j, h) - smem_u32(smem_raw)), &tmap_k, bar, 64 * h, hkv,
                        t * kTileKeys, b);
            tma_load_4d(smem_raw + (v_chunk(j, h) - smem_u32(smem_raw)), &tmap_v, bar, 64 * h, hkv,
                        t * kTileKeys, b);
          }
        }
        if (tail) {
          // The last cache tile: value rows past the length may hold anything
          // (NaN); zero them so that zero probabilities stay zero.
          mbar_wait(&tail_bar, 0, a.err);
          for (int c = lane; c < (kTileKeys - valid) * kSub * 8; c += 32) {
            const int row = valid + c / (kSub * 8), h = (c / 8) % kSub, cc = c % 8;
            st_shared_v4(swz(v_chunk(j, h), row, cc), make_uint4(0, 0, 0, 0));
          }
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) mbar_arrive(&kv_full[stage]);
        }
      } else {
        // Block keys/values (not cached): one TMA box per sub-tile from the
        // [B, k, Hkv, D] block tensors, like a cache tile; rows k..63 lie
        // outside those tensors and arrive as zeros.
        if (lane == 0) {
          mbar_arrive_expect_tx(&kv_full[stage], 2 * kSub * kKVSub);
          for (int h = 0; h < kSub; ++h) {
            tma_load_4d(smem_raw + (k_chunk(j, h) - smem_u32(smem_raw)), &tmap_kb, &kv_full[stage],
                        64 * h, hkv, 0, b);
            tma_load_4d(smem_raw + (v_chunk(j, h) - smem_u32(smem_raw)), &tmap_vb, &kv_full[stage],
                        64 * h, hkv, 0, b);
          }
        }
        if (a.kc_app) {
          // First iteration of a block: the causal rows' keys/values also
          // enter the cache at len .. len + n_causal - 1 (positions >= len are
          // read by no split of this call, or masked and zeroed where they
          // are).  Plain copies, all of a batch's loads before its stores;
          // nothing in this call waits for them.
          if (len + a.n_causal <= a.Lmax) {
            constexpr int kCpr = kSub * 8;             // 16-byte chunks per row
            constexpr int kBatch = 8;                  // chunks per lane per batch
            const int n_app = a.n_causal * kCpr;
            for (int c0 = 0; c0 < n_app; c0 += 32 * kBatch) {
              uint4 kv[kBatch], vv[kBatch];
#pragma unroll
              for (int e = 0; e < kBatch; ++e) {
                const int c = c0 + e * 32 + lane;
                if (c < n_app) {
                  const size_t off = (((size_t)b * a.k + c / kCpr) * a.Hkv + hkv) * D + (c % kCpr) * 8;
                  kv[e] = *reinterpret_cast<const uint4*>(a.kb + off);
                  vv[e] = *reinterpret_cast<const uint4*>(a.vb + off);
                }
              }
#pragma unroll
              for (int e = 0; e < kBatch; ++e) {
                const int c = c0 + e * 32 + lane;
                if (c < n_app) {
                  const size_t dst =
                      (((size_t)b * a.Lmax + len + c / kCpr) * a.Hkv + hkv) * D + (c % kCpr) * 8;
                  *reinterpret_cast<uint4*>(a.kc_app + dst) = kv[e];
                  *reinterpret_cast<uint4*>(a.vc_app + dst) = vv[e];
                }
              }
            }
          } else if (lane == 0) {
            record_error(a.err, SBD_DEVERR_CACHE_LEN);
          }
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer
    if (lane == 0 && n > 0) {
      const uint32_t id_o = idesc_bf16(kRows, D, true);
      bool ok = mbar_wait(&q_ready, 0, a.err);
      tc_fence_after();
      // S of pair q: M = 128 rows, N = 128 keys (64 for a last single tile),
      // K = D; the B operand is the pair's K sub-tiles.
      auto issue_s = [&](int q) {
        const int nt = min(2, n - 2 * q);
        const uint32_t kb = k_chunk(2 * q, 0);
        const uint32_t d = tmem + (uint32_t)((q & 1) * kPairKeys);
        const uint32_t id_s = idesc_bf16(kRows, nt * kTileKeys, false);
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint64_t ad = sw128_desc(q_s + (kk / 4) * kQBytes + (kk % 4) * 32, 16, 1024);
          const uint64_t bd = sw128_desc(kb + (kk / 4) * kPairSub + (kk % 4) * 32, 16, 1024);
          tc_mma(d, ad, bd, id_s, kk > 0);
        }
        tc_commit(&s_full[q & 1]);
      };
      // O += P V over the pair's keys, 16 keys per instruction (R = 1), or
      // 16 keys of each tile per instruction into the two copies' halves of
      // O (R = 2; N = D only for a last pair of one tile, whose second copy
      // has no keys).
      auto issue_pv = [&](int q) {
        const int nt = min(2, n - 2 * q);
        const uint32_t pb = p_block(q);
        const uint32_t vb = v_chunk(2 * q, 0);
        if constexpr (R == 1) {
#pragma unroll
          for (int kk = 0; kk < 8; ++kk) {
            if (kk >= 4 * nt) break;
            const uint64_t ad = sw128_desc(pb + (kk / 4) * kQBytes + (kk % 4) * 32, 16, 1024);
            const uint64_t bd = sw128_desc(vb + (kk / 4) * kSub * kKVSub + (kk % 4) * 16 * 128,
                                           kKVSub, 1024);
            tc_mma(tmem + kOCol, ad, bd, id_o, (q > 0 || kk > 0) ? 1u : 0u);
          }
        } else {
          const uint32_t id_pv = idesc_bf16(kRows, nt * D, true);
#pragma unroll
          for (int kk = 0; kk < 4; ++kk) {
            const uint64_t ad = sw128_desc(pb + kk * 32, 16, 1024);
            const uint64_t bd = sw128_desc(vb + kk * 16 * 128, kKVSub, 1024);
            tc_mma(tmem + kOCol, ad, bd, id_pv, (q > 0 || kk > 0) ? 1u : 0u);
          }
        }
        tc_commit(&pv_done[q & 1]);
        tc_commit(&kv_empty[q % kPairs]);
      };
      // In order: S_{q+1} is issued before waiting for P_q, so the scores of
      // the next pair are computed while the softmax of this one runs; and
      // since S_{q+1} is issued after PV_{q-1}, the completion of S_{q+1}
      // (s_full) implies PV_{q-1} is done, which keeps every later parity
      // wait on pv_done at most one phase behind.
      auto wait_issue_s = [&](int q) -> bool {
        const int j0 = 2 * q, nt = min(2, n - j0);
        for (int e = 0; e < nt; ++e)
          if (!mbar_wait(&kv_full[(j0 + e) % kStages], ((j0 + e) / kStages) & 1, a.err)) return false;
        if (!mbar_wait(&s_free[q & 1], ((q >> 1) & 1) ^ 1, a.err)) return false;
        tc_fence_after();
        issue_s(q);
        return true;
      };
      if (ok) ok = wait_issue_s(0);
      // (Issuing PV_q ahead of S_{q+1} when P_q is ready first measured
      // slower: the next softmax then waits longer for its scores.)
      for (int q = 0; q < np && ok; ++q) {
        if (q + 1 < np && !wait_issue_s(q + 1)) break;
        if (!mbar_wait(&p_full[q & 1], (q >> 1) & 1, a.err)) break;
        tc_fence_after();
        issue_pv(q);
      }
    }
  } else {
    // ------------------------------------------------ softmax warps
    constexpr int kCW = kPairKeys / (2 * R);     // columns per warp: 64 or 32
    constexpr int kQuadStride = 4 / R;           // lane quadrants between copies of a row
    constexpr int kRowsPerCopy = kRows / R;
    constexpr int kGroupThreads = 64 * R;        // the warps that share a row
    const int sw = warp - 2;                     // 0..7
    const int quad = warp & 3;                   // TMEM lanes 32*quad .. +31
    const int sub = sw >> 2;                     // 0 or 1 within the quadrant
    const int lane_t = quad * 32 + lane;         // TMEM lane
    const int row = lane_t % kRowsPerCopy;       // packed row
    const int dup = lane_t / kRowsPerCopy;       // copy of the row (R = 2): its tile
    const int cbase = kCW * (dup * 2 + sub);     // this warp's columns of a pair
    const int half = cbase / kTileKeys;          // ... all inside one tile
    const int coff = cbase % kTileKeys;          // first column inside that tile
    const bool owns_o = dup == 0;                // this lane writes row `row` out
    // this lane's O: R = 1 the row's, R = 2 its copy's partial (own tile)
    const uint32_t o_col = kOCol + (uint32_t)(dup * D);
    const int bar_id = 1 + quad % kQuadStride;  // one named barrier per row group
    const uint32_t lane_addr = (uint32_t)(quad * 32) << 16;
    // softmax warp index of (quadrant q, sub s)
    auto sw_of = [](int q_, int s_) { return 4 * s_ + ((q_ - 2) & 3); };
    // quadrant of copy d of this lane's row
    auto quad_of = [&](int d) { return quad % kQuadStride + kQuadStride * d; };
    // Q row -> shared (swizzled, K-major); each sub-warp copies half a row;
    // padding rows are zero.
    {
      const __nv_bfloat16* qrow =
          row < a.M ? a.q + (((size_t)b * a.k + row / a.G) * a.Hq + hkv * a.G + row % a.G) * D
                    : nullptr;
#pragma unroll
      for (int c = sub * (D / 16); c < (sub + 1) * (D / 16); ++c) {
        const uint4 v = qrow ? *reinterpret_cast<const uint4*>(qrow + c * 8) : make_uint4(0, 0, 0, 0);
        st_shared_v4(swz(q_s + (c / 8) * kQBytes, lane_t, c % 8), v);
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(&q_ready);
    }
    float m_ref = -INFINITY, l = 0.f;
    bool ok = true;
    // Every softmax warp runs all np iterations and meets its group barrier
    // once per iteration, also after a bounded wait gave up (then it only
    // keeps the barrier count), so that no named barrier waits forever.
    for (int q = 0; q < np; ++q) {
      const int j = 2 * q + half;                // the tile this warp's columns are in
      const int t = t_begin + j;
      int valid;
      if (j >= n) {
        valid = 0;                               // a last pair of one tile
      } else if (t < n_cache_tiles) {
        valid = min(kTileKeys, len - t * kTileKeys);
      } else {
        // causal rows of the block see the block keys j <= i only
        valid = row / a.G < a.n_causal ? row / a.G + 1 : a.k;
      }
      if (ok && !mbar_wait(&s_full[q & 1], (q >> 1) & 1, a.err)) ok = false;
      // tcgen05.ld/st are warp-collective: the warp goes on only as a whole
      ok = __all_sync(0xffffffffu, ok);
      float s[kCW];
      float mloc = -INFINITY;
      if (ok) {
        tc_fence_after();
        const uint32_t sa = tmem + lane_addr + (uint32_t)((q & 1) * kPairKeys + cbase);
        uint32_t r[kCW / 16][16];
#pragma unroll
        for (int h = 0; h < kCW / 16; ++h) tc_ld16(sa + 16 * h, r[h]);
        tc_wait_ld();
#pragma unroll
        for (int h = 0; h < kCW / 16; ++h)
#pragma unroll
          for (int e = 0; e < 16; ++e) s[16 * h + e] = __uint_as_float(r[h][e]);
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&s_free[q & 1]);
        // masked keys only exist in the last cache tile, the block tile and
        // the empty half of a last single-tile pair
        if (valid < coff + kCW) {
#pragma unroll
          for (int c = 0; c < kCW; ++c)
            if (coff + c >= valid) s[c] = -INFINITY;
        }
        float mx[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) mx[e] = s[e];
#pragma unroll
        for (int c = 8; c < kCW; c += 8)
#pragma unroll
          for (int e = 0; e < 8; ++e) mx[e] = fmaxf(mx[e], s[c + e]);
        mloc = fmaxf(fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])),
                     fmaxf(fmaxf(mx[4], mx[5]), fmaxf(mx[6], mx[7])));
      }
      // The group agrees on max_w(round_up_bf16(m_w)) >= the row maximum: a
      // reference at or above the maximum is all the lazy rescale needs (l and
      // O share it), and every warp of the group takes the same value.
      red_max[((q & 1) * kSoftWarps + sw) * 32 + lane] = bf16_bits_round_up(mloc);
      asm volatile("bar.sync %0, %1;" ::"r"(bar_id), "n"(kGroupThreads) : "memory");
      if (!ok) continue;
      float mraw = -INFINITY;
#pragma unroll
      for (int d2 = 0; d2 < R; ++d2)
#pragma unroll
        for (int s2 = 0; s2 < 2; ++s2) {
          const int w2 = sw_of(quad_of(d2), s2);
          mraw = fmaxf(mraw, bf16_bits_to_float(red_max[((q & 1) * kSoftWarps + w2) * 32 + lane]));
        }
      const float mt = mraw * a.scale_log2;     // the scale is positive
      // Each row decides for itself; the TMEM rescale of O is warp-collective,
      // so a warp rescales when any of its rows does (alpha = 1 for the rest).
      const bool rescale = m_ref != -INFINITY && mt > m_ref + kRescaleThreshold;
      const bool warp_rescale = __any_sync(0xffffffffu, rescale);
      // The P block of this pair is free once PV(q-2) is done (it lives in
      // the pair's own K sub-tiles for D = 128); O itself is only touched
      // (rescaled) after PV(q-1).
      const int wait_q = warp_rescale ? q - 1 : (kPInK ? -1 : q - 2);
      bool waited = wait_q < 0 || mbar_wait(&pv_done[wait_q & 1], (wait_q >> 1) & 1, a.err);
      if (!__all_sync(0xffffffffu, waited)) {
        ok = false;
        continue;
      }
      tc_fence_after();
      const float alpha = rescale ? exp2f(m_ref - mt) : 1.f;
      if (m_ref == -INFINITY) {
        m_ref = mt;
      } else if (rescale) {
        l *= alpha;
        m_ref = mt;
      }
      if (warp_rescale) {
        // the two sub-warps of a quadrant rescale half of its lanes' O each
#pragma unroll
        for (int c = sub * (D / 32); c < (sub + 1) * (D / 32); ++c) {
          uint32_t r[16];
          tc_ld16(tmem + lane_addr + o_col + c * 16, r);
          tc_wait_ld();
#pragma unroll
          for (int e = 0; e < 16; ++e) r[e] = __float_as_uint(__uint_as_float(r[e]) * alpha);
          tc_st16(tmem + lane_addr + o_col + c * 16, r);
        }
        tc_wait_st();
      }
      // P = 2^(scale * s - m_ref) as bf16 into this warp's columns of the
      // pair's P block, in row `lane_t` (R = 1: the packed row; R = 2: the
      // copy's row, whose keys are its tile's).  Rows past M are garbage
      // whose O rows are never read.
      const uint32_t pb = p_block(q) + (R == 1 ? half * kQBytes : 0);
      {
        const float nm = -m_ref;
        float psum[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int c = 0; c < kCW / 8; ++c) {
          float p[8];
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            p[e] = ex2_ftz(fmaf(s[c * 8 + e], a.scale_log2, nm));
            psum[e] += p[e];
          }
          st_shared_v4(swz(pb, lane_t, coff / 8 + c),
                       make_uint4(pack_bf16(p[0], p[1]), pack_bf16(p[2], p[3]),
                                  pack_bf16(p[4], p[5]), pack_bf16(p[6], p[7])));
        }
        l += ((psum[0] + psum[1]) + (psum[2] + psum[3])) + ((psum[4] + psum[5]) + (psum[6] + psum[7]));
      }
      fence_proxy_async_smem();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&p_full[q & 1]);
    }
    grid_dependents_launch();
    // ------------------------------------------------ epilogue
    // Row sums over the group, in a fixed order.  They reuse the buffer of
    // the maxima, whose slots of every group they overlap, and a slower
    // group may still be reading the last pair's maxima: all softmax warps
    // pass one barrier (id 5; the groups use 1-4) before any sum is written.
    asm volatile("bar.sync 5, %0;" ::"n"(kSoftWarps * 32) : "memory");
    red_l[sw * 32 + lane] = l;
    asm volatile("bar.sync %0, %1;" ::"r"(bar_id), "n"(kGroupThreads) : "memory");
    float lsum = 0.f;
#pragma unroll
    for (int d2 = 0; d2 < R; ++d2)
#pragma unroll
      for (int s2 = 0; s2 < 2; ++s2)
        lsum += red_l[sw_of(quad_of(d2), s2) * 32 + lane];
    const bool mine = owns_o && row < a.M;
    // the two sub-warps of a quadrant take half of the D columns each
    const int c_lo = sub * (D / 32), c_hi = (sub + 1) * (D / 32);
    bool final_ok = ok && np > 0 && mbar_wait(&pv_done[(np - 1) & 1], ((np - 1) >> 1) & 1, a.err);
    final_ok = __all_sync(0xffffffffu, final_ok);   // the reads below are warp-collective
    // R = 2: copy 1 hands its partial O to copy 0 through shared memory (the
    // ring, idle once the last PV is done: every load was consumed by an
    // MMA before it).  A split of one tile gave copy 1 no keys; its half of
    // O was never written and is left out.
    constexpr int kStageStride = D + 1;           // floats per staged row (bank spread)
    float* stage = reinterpret_cast<float*>(smem_raw + (kv_s - smem_u32(smem_raw)));
    const bool has_copy1 = R == 2 && n >= 2;
    // Cluster merge: this CTA's normalised partial rows and their log2-sum-
    // exps, 64 KB into the ring (past the copy-1 stage), read by every CTA of
    // the cluster after a cluster barrier.
    constexpr int kCStride = D + 4;             // floats per partial row (16-byte rows)
    float* cpart = reinterpret_cast<float*>(smem_raw + (kv_s + 65536u - smem_u32(smem_raw)));
    float* clse = cpart + kRows * kCStride;
    if constexpr (R == 2) {
      if (final_ok && dup == 1 && has_copy1) {
        tc_fence_after();
#pragma unroll
        for (int c = c_lo; c < c_hi; ++c) {
          uint32_t r[16];
          tc_ld16(tmem + lane_addr + o_col + c * 16, r);
          tc_wait_ld();
#pragma unroll
          for (int e = 0; e < 16; ++e) stage[row * kStageStride + c * 16 + e] = __uint_as_float(r[e]);
        }
      }
      asm volatile("bar.sync %0, %1;" ::"r"(bar_id), "n"(kGroupThreads) : "memory");
    }
    // Row `row` of O in columns [16 c, 16 c + 16): this lane's accumulator
    // plus, with R = 2, the other copy's.
    auto load_o = [&](int c, float (&o)[16]) {
      uint32_t r[16];
      tc_ld16(tmem + lane_addr + o_col + c * 16, r);
      tc_wait_ld();
#pragma unroll
      for (int e = 0; e < 16; ++e) o[e] = __uint_as_float(r[e]);
      if (has_copy1) {
#pragma unroll
        for (int e = 0; e < 16; ++e) o[e] += stage[row * kStageStride + c * 16 + e];
      }
    };
    if (final_ok && owns_o) {
      tc_fence_after();
      const float inv = lsum > 0.f ? 1.f / lsum : 0.f;
      if (a.splits == 1) {
        __nv_bfloat16* dst =
            mine ? a.out + (((size_t)b * a.k + row / a.G) * a.Hq + hkv * a.G + row % a.G) * D
                 : nullptr;
#pragma unroll
        for (int c = c_lo; c < c_hi; ++c) {
          float o[16];
          load_o(c, o);
          if (mine) {
            uint4 w0, w1;
            w0.x = pack_bf16(o[0] * inv, o[1] * inv);
            w0.y = pack_bf16(o[2] * inv, o[3] * inv);
            w0.z = pack_bf16(o[4] * inv, o[5] * inv);
            w0.w = pack_bf16(o[6] * inv, o[7] * inv);
            w1.x = pack_bf16(o[8] * inv, o[9] * inv);
            w1.y = pack_bf16(o[10] * inv, o[11] * inv);
            w1.z = pack_bf16(o[12] * inv, o[13] * inv);
            w1.w = pack_bf16(o[14] * inv, o[15] * inv);
            *reinterpret_cast<uint4*>(dst + c * 16) = w0;
            *reinterpret_cast<uint4*>(dst + c * 16 + 8) = w1;
          }
        }
      } else {
        const size_t prow = (((size_t)b * a.Hkv + hkv) * a.splits + split) * a.M + row;
        float* dst = mine ? (a.cluster ? cpart + row * kCStride : a.part_o + prow * D) : nullptr;
#pragma unroll
        for (int c = c_lo; c < c_hi; ++c) {
          float o[16];
          load_o(c, o);
          if (mine) {
#pragma unroll
            for (int e = 0; e < 16; e += 4)
              *reinterpret_cast<float4*>(dst + c * 16 + e) =
                  make_float4(o[e] * inv, o[e + 1] * inv, o[e + 2] * inv, o[e + 3] * inv);
          }
        }
        if (mine && sub == 0) {
          const float lse = lsum > 0.f ? m_ref + log2f(lsum) : -INFINITY;
          if (a.cluster) clse[row] = lse; else a.part_lse[prow] = lse;
        }
      }
    } else if (n == 0 && a.splits > 1 && mine) {
      // an empty split contributes nothing
      const size_t prow = (((size_t)b * a.Hkv + hkv) * a.splits + split) * a.M + row;
      float* dst = a.cluster ? cpart + row * kCStride : a.part_o + prow * D;
      for (int d = c_lo * 16; d < c_hi * 16; ++d) dst[d] = 0.f;
      if (sub == 0) {
        if (a.cluster) clse[row] = -INFINITY; else a.part_lse[prow] = -INFINITY;
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tc_dealloc(tmem, kTmemCols);
  }
  if (a.cluster) cluster_merge<D>(a, b, hkv, kv_s + 65536u, warp - 2, lane);
}

// ------------------------------------------------------------ wide row tiles
// More than 64 packed rows (M = 65..128, e.g. k = 32 with 4 query heads per
// KV head): every TMEM lane holds a distinct row, so the copy scheme of
// attn_tc_kernel has nothing to pair, and PV needs D / 16 ... keys / 16
// instructions of N = D.  What can still shrink is the score product and
// the ring's hold on K.  Keys go in triples of 64-key tiles:
//
//   S_t = Q K_t^T     A = Q (shared, K-major), B = the triple's K (shared,
//                     K-major), N = 192: D / 16 instructions per 192 keys
//                     instead of per 128;
//   O  += P_t V_t     A = P_t from tensor memory (tcgen05.mma with the A
//                     operand in TMEM; bf16 pairs written by the softmax
//                     warps with tcgen05.st), B = each tile's V (shared,
//                     MN-major), N = D: 12 instructions per triple.
//
// Tensor memory: S 192 | O D | P 2 x 96 columns.  With P there, shared
// memory holds Q and two separate rings: 2 triples of K, each freed as soon
// as its score product is done, and V tiles, each freed after its PV
// instructions.  S is a single buffer (S_{t+1} is issued once the softmax
// warps hold S_t in registers); P is double-buffered, so that the
// exponentials of triple t + 1 do not wait for PV_t.
//
// Warp roles: warp 0 loads K (TMA), warp 1 owns the tensor memory and
// issues the MMAs, warp 2 loads V (TMA; zeroes value rows past the cache
// length; copies the causal rows into the cache), warps 3-10 are the softmax
// (two per lane quadrant, 96 of a triple's 192 columns each, the row maximum
// agreed through shared memory).  Rescale rule, epilogue and cluster merge
// as in attn_tc_kernel.
constexpr int kTriTiles = 3;
constexpr int kTriKeys = kTriTiles * kTileKeys;          // 192
constexpr int kWideKSlots = 2;                           // K triples in the ring
// V tiles in the ring: what is left of the 227 KB next to Q and the K ring
template <int D> __host__ __device__ constexpr int wide_v_slots() { return D == 128 ? 6 : 8; }
constexpr int kWideThreads = 96 + 32 * kSoftWarps;       // K, MMA, V, softmax warps

__host__ __device__ constexpr int wide_tmem_o() { return kTriKeys; }              // 192
template <int D> __host__ __device__ constexpr int wide_tmem_p() { return kTriKeys + D; }

template <int D>
__global__ void __launch_bounds__(kWideThreads, 1)
attn_wide_kernel(const __grid_constant__ CUtensorMap tmap_k,
                 const __grid_constant__ CUtensorMap tmap_v,
                 const __grid_constant__ CUtensorMap tmap_kb,
                 const __grid_constant__ CUtensorMap tmap_vb, const TcArgs a) {
  constexpr int kSub = D / 64;                     // 128-B column sub-tiles of a key row
  constexpr int kKVSub = kTileKeys * 128;          // one tile's K or V sub-tile: 8 KB
  constexpr int kTriSub = kTriTiles * kKVSub;      // a triple's K sub-tile: 24 KB
  constexpr int kKSlotBytes = kSub * kTriSub;
  constexpr int kVSlotBytes = kSub * kKVSub;
  constexpr int kVSlots = wide_v_slots<D>();
  constexpr int kQBytes = kRows * 128;             // one Q sub-tile: 16 KB
  constexpr uint32_t kTmemCols = 512;
  constexpr uint32_t kOCol = wide_tmem_o();
  constexpr uint32_t kPCol = wide_tmem_p<D>();
  constexpr uint32_t kPStride = kTriKeys / 2;      // columns of one P buffer
  static_assert(kPCol + 2 * kPStride <= kTmemCols, "S, O and two P buffers fit the allocation");
  constexpr int kCW = kTriKeys / 2;                // columns per softmax warp: 96

  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t k_full[kWideKSlots], k_empty[kWideKSlots];
  __shared__ __align__(8) uint64_t v_full[kVSlots], v_empty[kVSlots];
  __shared__ __align__(8) uint64_t s_full, s_free, p_full[2], pv_done[2], q_ready, tail_bar;
  __shared__ uint32_t tmem_base_sh;
  __shared__ __align__(16) uint32_t red_buf[kSoftWarps * 32];
  uint16_t* red_max = reinterpret_cast<uint16_t*>(red_buf);
  float* red_l = reinterpret_cast<float*>(red_buf);
  __shared__ int b_pick;

  const uint32_t sbase = (smem_u32(smem_raw) + 1023u) & ~1023u;
  const uint32_t q_s = sbase;                                   // kSub x 16 KB
  const uint32_t k_s = q_s + kSub * kQBytes;                    // kWideKSlots x kKSlotBytes
  const uint32_t v_s = k_s + kWideKSlots * kKSlotBytes;         // kVSlots x kVSlotBytes
  // tile j of the split: K in triple slot (j / 3) mod 2, position j mod 3 of
  // every sub-tile (the triple's keys form one 192-row operand); V in tile
  // slot j mod kVSlots
  auto k_chunk = [&](int j, int h) -> uint32_t {
    return k_s + ((j / kTriTiles) % kWideKSlots) * kKSlotBytes + h * kTriSub + (j % kTriTiles) * kKVSub;
  };
  auto v_chunk = [&](int j, int h) -> uint32_t {
    return v_s + (j % kVSlots) * kVSlotBytes + h * kKVSub;
  };

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int split = blockIdx.x, hkv = blockIdx.y;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kWideKSlots; ++s) {
      mbar_init(&k_full[s], 1);
      mbar_init(&k_empty[s], 1);
    }
    for (int s = 0; s < kVSlots; ++s) {
      mbar_init(&v_full[s], 1);
      mbar_init(&v_empty[s], 1);
    }
    mbar_init(&s_full, 1);
    mbar_init(&s_free, kSoftWarps);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&p_full[i], kSoftWarps);
      mbar_init(&pv_done[i], 1);
    }
    mbar_init(&q_ready, kSoftWarps);
    mbar_init(&tail_bar, 1);
    fence_mbar_init();
  }
  grid_dependency_wait();
  if (a.order) {
    longest_first_pick(a.lens, a.B, a.Lmax, blockIdx.z, &b_pick);
    __syncthreads();
  }
  const int b = a.order ? b_pick : (int)blockIdx.z;
  if (warp == 1) tc_alloc(&tmem_base_sh, kTmemCols);

  int len = a.lens[b];
  if (len < 0 || len > a.Lmax) {
    if (threadIdx.x == 0 && split == 0 && hkv == 0) record_error(a.err, SBD_DEVERR_CACHE_LEN);
    len = len < 0 ? 0 : a.Lmax;
  }
  const int n_cache_tiles = (len + kTileKeys - 1) / kTileKeys;
  const int n_tiles = n_cache_tiles + 1;
  const int t_begin = (int)((long long)split * n_tiles / a.splits);
  const int t_end = (int)((long long)(split + 1) * n_tiles / a.splits);
  const int n = t_end - t_begin;                  // 64-key tiles of this split
  const int nt = (n + kTriTiles - 1) / kTriTiles; // triples (the last may be short)

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base_sh;

  if (warp == 0) {
    // ------------------------------------------------ K producer
    if (lane == 0) {
      tma_prefetch_desc(&tmap_k);
      if (t_end == n_tiles) tma_prefetch_desc(&tmap_kb);
      int issued = 0;
      for (int t = 0; t < nt; ++t) {
        const int slot = t % kWideKSlots;
        if (!mbar_wait(&k_empty[slot], ((t / kWideKSlots) & 1) ^ 1, a.err)) break;
        const int j0 = kTriTiles * t, ntl = min(kTriTiles, n - j0);
        mbar_arrive_expect_tx(&k_full[slot], ntl * kSub * kKVSub);
        for (int e = 0; e < ntl; ++e) {
          const int j = j0 + e, tg = t_begin + j;
          for (int h = 0; h < kSub; ++h) {
            uint8_t* dst = smem_raw + (k_chunk(j, h) - smem_u32(smem_raw));
            if (tg < n_cache_tiles)
              tma_load_4d(dst, &tmap_k, &k_full[slot], 64 * h, hkv, tg * kTileKeys, b);
            else   // the block keys; rows k..63 lie outside the block tensor: zeros
              tma_load_4d(dst, &tmap_kb, &k_full[slot], 64 * h, hkv, 0, b);
          }
        }
        issued = t + 1;
      }
      // copies still in flight land before the CTA exits (on every path the
      // consumer would have waited for them; this matters only after a
      // bounded wait gave up)
      for (int t = issued - kWideKSlots > 0 ? issued - kWideKSlots : 0; t < issued; ++t)
        mbar_wait(&k_full[t % kWideKSlots], (t / kWideKSlots) & 1, a.err);
    }
  } else if (warp == 2) {
    // ------------------------------------------------ V producer
    if (lane == 0) {
      tma_prefetch_desc(&tmap_v);
      if (t_end == n_tiles) tma_prefetch_desc(&tmap_vb);
    }
    int issued = 0;
    for (int j = 0; j < n; ++j) {
      const int slot = j % kVSlots, tg = t_begin + j;
      const bool freed = mbar_wait(&v_empty[slot], ((j / kVSlots) & 1) ^ 1, a.err);
      if (!__all_sync(0xffffffffu, freed)) break;
      issued = j + 1;
      if (tg < n_cache_tiles) {
        const int valid = min(kTileKeys, len - tg * kTileKeys);
        const bool tail = valid < kTileKeys;
        uint64_t* bar = tail ? &tail_bar : &v_full[slot];
        if (lane == 0) {
          mbar_arrive_expect_tx(bar, kSub * kKVSub);
          for (int h = 0; h < kSub; ++h)
            tma_load_4d(smem_raw + (v_chunk(j, h) - smem_u32(smem_raw)), &tmap_v, bar, 64 * h, hkv,
                        tg * kTileKeys, b);
        }
        if (tail) {
          // value rows past the length may hold anything (NaN): zero them so
          // that zero probabilities stay zero
          mbar_wait(&tail_bar, 0, a.err);
          for (int c = lane; c < (kTileKeys - valid) * kSub * 8; c += 32) {
            const int row = valid + c / (kSub * 8), h = (c / 8) % kSub, cc = c % 8;
            st_shared_v4(swz(v_chunk(j, h), row, cc), make_uint4(0, 0, 0, 0));
          }
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) mbar_arrive(&v_full[slot]);
        }
      } else {
        if (lane == 0) {
          mbar_arrive_expect_tx(&v_full[slot], kSub * kKVSub);
          for (int h = 0; h < kSub; ++h)
            tma_load_4d(smem_raw + (v_chunk(j, h) - smem_u32(smem_raw)), &tmap_vb, &v_full[slot],
                        64 * h, hkv, 0, b);
        }
        if (a.kc_app) {
          // first iteration of a block: the causal rows' keys and values also
          // enter the cache at len .. len + n_causal - 1 (see attn_tc_kernel)
          if (len + a.n_causal <= a.Lmax) {
            constexpr int kCpr = kSub * 8;
            constexpr int kBatch = 8;
            const int n_app = a.n_causal * kCpr;
            for (int c0 = 0; c0 < n_app; c0 += 32 * kBatch) {
              uint4 kv[kBatch], vv[kBatch];
#pragma unroll
              for (int e = 0; e < kBatch; ++e) {
                const int c = c0 + e * 32 + lane;
                if (c < n_app) {
                  const size_t off = (((size_t)b * a.k + c / kCpr) * a.Hkv + hkv) * D + (c % kCpr) * 8;
                  kv[e] = *reinterpret_cast<const uint4*>(a.kb + off);
                  vv[e] = *reinterpret_cast<const uint4*>(a.vb + off);
                }
              }
#pragma unroll
              for (int e = 0; e < kBatch; ++e) {
                const int c = c0 + e * 32 + lane;
                if (c < n_app) {
                  const size_t dst =
                      (((size_t)b * a.Lmax + len + c / kCpr) * a.Hkv + hkv) * D + (c % kCpr) * 8;
                  *reinterpret_cast<uint4*>(a.kc_app + dst) = kv[e];
                  *reinterpret_cast<uint4*>(a.vc_app + dst) = vv[e];
                }
              }
            }
          } else if (lane == 0) {
            record_error(a.err, SBD_DEVERR_CACHE_LEN);
          }
        }
      }
    }
    if (lane == 0)
      for (int j = issued - kVSlots > 0 ? issued - kVSlots : 0; j < issued; ++j)
        mbar_wait(&v_full[j % kVSlots], (j / kVSlots) & 1, a.err);
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer
    if (lane == 0 && n > 0) {
      const uint32_t id_o = idesc_bf16(kRows, D, true);
      bool ok = mbar_wait(&q_ready, 0, a.err);
      tc_fence_after();
      auto issue_s = [&](int t) -> bool {
        const int slot = t % kWideKSlots;
        if (!mbar_wait(&k_full[slot], (t / kWideKSlots) & 1, a.err)) return false;
        tc_fence_after();
        const int ntl = min(kTriTiles, n - kTriTiles * t);
        const uint32_t kb = k_chunk(kTriTiles * t, 0);
        const uint32_t id_s = idesc_bf16(kRows, ntl * kTileKeys, false);
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint64_t ad = sw128_desc(q_s + (kk / 4) * kQBytes + (kk % 4) * 32, 16, 1024);
          const uint64_t bd = sw128_desc(kb + (kk / 4) * kTriSub + (kk % 4) * 32, 16, 1024);
          tc_mma(tmem, ad, bd, id_s, kk > 0);
        }
        tc_commit(&s_full);
        tc_commit(&k_empty[slot]);
        return true;
      };
      if (ok) ok = issue_s(0);
      for (int t = 0; t < nt && ok; ++t) {
        // the next scores as soon as the softmax warps hold S_t in registers
        if (t + 1 < nt) {
          if (!mbar_wait(&s_free, t & 1, a.err)) break;
          if (!issue_s(t + 1)) break;
        }
        if (!mbar_wait(&p_full[t & 1], (t >> 1) & 1, a.err)) break;
        tc_fence_after();
        const int j0 = kTriTiles * t, ntl = min(kTriTiles, n - j0);
        for (int e = 0; e < ntl && ok; ++e) {
          const int j = j0 + e;
          if (!mbar_wait(&v_full[j % kVSlots], (j / kVSlots) & 1, a.err)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t vb = v_chunk(j, 0);
#pragma unroll
          for (int kk = 0; kk < 4; ++kk) {
            const uint64_t bd = sw128_desc(vb + kk * 16 * 128, kKVSub, 1024);
            tc_mma_ts(tmem + kOCol, tmem + kPCol + (t & 1) * kPStride + (4 * e + kk) * 8, bd, id_o,
                      (t > 0 || e > 0 || kk > 0) ? 1u : 0u);
          }
          tc_commit(&v_empty[j % kVSlots]);
        }
        if (ok) tc_commit(&pv_done[t & 1]);
      }
    }
  } else {
    // ------------------------------------------------ softmax warps
    const int sw = warp - 3;                     // 0..7
    const int quad = warp & 3;                   // TMEM lanes 32*quad .. +31
    const int sub = sw >> 2;                     // 0 or 1 within the quadrant
    const int row = quad * 32 + lane;            // packed row = TMEM lane
    const int cbase = kCW * sub;                 // this warp's columns of a triple
    const int bar_id = 1 + quad;                 // the two warps of a quadrant
    const uint32_t lane_addr = (uint32_t)(quad * 32) << 16;
    auto sw_of = [](int q_, int s_) { return 4 * s_ + ((q_ - 3) & 3); };
    // Q row -> shared (swizzled, K-major); each sub-warp copies half a row;
    // padding rows are zero.
    {
      const __nv_bfloat16* qrow =
          row < a.M ? a.q + (((size_t)b * a.k + row / a.G) * a.Hq + hkv * a.G + row % a.G) * D
                    : nullptr;
#pragma unroll
      for (int c = sub * (D / 16); c < (sub + 1) * (D / 16); ++c) {
        const uint4 v = qrow ? *reinterpret_cast<const uint4*>(qrow + c * 8) : make_uint4(0, 0, 0, 0);
        st_shared_v4(swz(q_s + (c / 8) * kQBytes, row, c % 8), v);
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(&q_ready);
    }
    float m_ref = -INFINITY, l = 0.f;
    bool ok = true;
    for (int t = 0; t < nt; ++t) {
      // valid keys of the two tiles this warp's 96 columns fall in (sub 0:
      // tile 0 and the first half of tile 1; sub 1: the second half of tile
      // 1 and tile 2), for this row
      auto valid_of = [&](int e) {
        const int j = kTriTiles * t + e, tg = t_begin + j;
        if (j >= n) return 0;
        if (tg < n_cache_tiles) return min(kTileKeys, len - tg * kTileKeys);
        return row / a.G < a.n_causal ? row / a.G + 1 : a.k;
      };
      const int valid_a = valid_of(sub), valid_b = valid_of(sub + 1);
      const int off0 = cbase & (kTileKeys - 1);    // key of column 0 within its tile
      if (ok && !mbar_wait(&s_full, t & 1, a.err)) ok = false;
      ok = __all_sync(0xffffffffu, ok);
      // the warp's 96 scores of this row, as raw fp32 bits
      uint32_t sr[kCW / 16][16];
      float mloc = -INFINITY;
      if (ok) {
        tc_fence_after();
        const uint32_t sa = tmem + lane_addr + (uint32_t)cbase;
#pragma unroll
        for (int h = 0; h < kCW / 16; ++h) tc_ld16(sa + 16 * h, sr[h]);
        tc_wait_ld();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&s_free);
        // column c is key off0 + c of the first tile while that is < 64, then
        // key c - (64 - off0) of the second; masked keys exist only in the
        // last cache tile, the block tile and past the split's last tile
        if (valid_a < kTileKeys || valid_b < kTileKeys) {
#pragma unroll
          for (int c = 0; c < kCW; ++c) {
            const bool first = c < kTileKeys - off0;
            const int key = first ? off0 + c : c - (kTileKeys - off0);
            if (key >= (first ? valid_a : valid_b)) sr[c / 16][c % 16] = __float_as_uint(-INFINITY);
          }
        }
        float mx[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) mx[e] = __uint_as_float(sr[0][e]);
#pragma unroll
        for (int c = 8; c < kCW; c += 8)
#pragma unroll
          for (int e = 0; e < 8; ++e) mx[e] = fmaxf(mx[e], __uint_as_float(sr[c / 16][c % 16 + e]));
        mloc = fmaxf(fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])),
                     fmaxf(fmaxf(mx[4], mx[5]), fmaxf(mx[6], mx[7])));
      }
      red_max[((t & 1) * kSoftWarps + sw) * 32 + lane] = bf16_bits_round_up(mloc);
      asm volatile("bar.sync %0, %1;" ::"r"(bar_id), "n"(64) : "memory");
      if (!ok) continue;
      float mraw = -INFINITY;
#pragma unroll
      for (int s2 = 0; s2 < 2; ++s2)
        mraw = fmaxf(mraw, bf16_bits_to_float(red_max[((t & 1) * kSoftWarps + sw_of(quad, s2)) * 32 + lane]));
      const float mt = mraw * a.scale_log2;
      const bool rescale = m_ref != -INFINITY && mt > m_ref + kRescaleThreshold;
      const bool warp_rescale = __any_sync(0xffffffffu, rescale);
      // P buffer t mod 2 is written after PV_{t-2}, O rescaled after PV_{t-1}
      const int wait_t = warp_rescale ? t - 1 : t - 2;
      bool waited = wait_t < 0 || mbar_wait(&pv_done[wait_t & 1], (wait_t >> 1) & 1, a.err);
      if (!__all_sync(0xffffffffu, waited)) {
        ok = false;
        continue;
      }
      tc_fence_after();
      const float alpha = rescale ? exp2f(m_ref - mt) : 1.f;
      if (m_ref == -INFINITY) {
        m_ref = mt;
      } else if (rescale) {
        l *= alpha;
        m_ref = mt;
      }
      if (warp_rescale) {
#pragma unroll
        for (int c = sub * (D / 32); c < (sub + 1) * (D / 32); ++c) {
          uint32_t r[16];
          tc_ld16(tmem + lane_addr + kOCol + c * 16, r);
          tc_wait_ld();
#pragma unroll
          for (int e = 0; e < 16; ++e) r[e] = __float_as_uint(__uint_as_float(r[e]) * alpha);
          tc_st16(tmem + lane_addr + kOCol + c * 16, r);
        }
      }
      // P = 2^(scale * s - m_ref) as bf16 pairs into tensor memory: this
      // warp's 96 keys are P columns cbase / 2 .. + 47
      {
        const float nm = -m_ref;
        float psum[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int h = 0; h < kCW / 32; ++h) {
          uint32_t r[16];
#pragma unroll
          for (int e = 0; e < 16; ++e) {
            const int c = 32 * h + 2 * e;
            const float p0 = ex2_ftz(fmaf(__uint_as_float(sr[c / 16][c % 16]), a.scale_log2, nm));
            const float p1 = ex2_ftz(fmaf(__uint_as_float(sr[(c + 1) / 16][(c + 1) % 16]), a.scale_log2, nm));
            psum[(2 * e) & 7] += p0;
            psum[(2 * e + 1) & 7] += p1;
            r[e] = pack_bf16(p0, p1);
          }
          tc_st16(tmem + lane_addr + kPCol + (t & 1) * kPStride + cbase / 2 + 16 * h, r);
        }
        l += ((psum[0] + psum[1]) + (psum[2] + psum[3])) + ((psum[4] + psum[5]) + (psum[6] + psum[7]));
      }
      tc_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&p_full[t & 1]);
    }
    grid_dependents_launch();
    // ------------------------------------------------ epilogue
    asm volatile("bar.sync 5, %0;" ::"n"(kSoftWarps * 32) : "memory");
    red_l[sw * 32 + lane] = l;
    asm volatile("bar.sync %0, %1;" ::"r"(bar_id), "n"(64) : "memory");
    const float lsum = red_l[sw_of(quad, 0) * 32 + lane] + red_l[sw_of(quad, 1) * 32 + lane];
    const bool mine = row < a.M;
    const int c_lo = sub * (D / 32), c_hi = (sub + 1) * (D / 32);
    bool final_ok = ok && nt > 0 && mbar_wait(&pv_done[(nt - 1) & 1], ((nt - 1) >> 1) & 1, a.err);
    final_ok = __all_sync(0xffffffffu, final_ok);
    constexpr int kCStride = D + 4;
    float* cpart = reinterpret_cast<float*>(smem_raw + (k_s - smem_u32(smem_raw)));
    float* clse = cpart + kRows * kCStride;
    if (final_ok) {
      tc_fence_after();
      const float inv = lsum > 0.f ? 1.f / lsum : 0.f;
      if (a.splits == 1) {
        __nv_bfloat16* dst =
            mine ? a.out + (((size_t)b * a.k + row / a.G) * a.Hq + hkv * a.G + row % a.G) * D
                 : nullptr;
#pragma unroll
        for (int c = c_lo; c < c_hi; ++c) {
          uint32_t r[16];
          tc_ld16(tmem + lane_addr + kOCol + c * 16, r);
          tc_wait_ld();
          if (mine) {
            uint4 w0, w1;
            w0.x = pack_bf16(__uint_as_float(r[0]) * inv, __uint_as_float(r[1]) * inv);
            w0.y = pack_bf16(__uint_as_float(r[2]) * inv, __uint_as_float(r[3]) * inv);
            w0.z = pack_bf16(__uint_as_float(r[4]) * inv, __uint_as_float(r[5]) * inv);
            w0.w = pack_bf16(__uint_as_float(r[6]) * inv, __uint_as_float(r[7]) * inv);
            w1.x = pack_bf16(__uint_as_float(r[8]) * inv, __uint_as_float(r[9]) * inv);
            w1.y = pack_bf16(__uint_as_float(r[10]) * inv, __uint_as_float(r[11]) * inv);
            w1.z = pack_bf16(__uint_as_float(r[12]) * inv, __uint_as_float(r[13]) * inv);
            w1.w = pack_bf16(__uint_as_float(r[14]) * inv, __uint_as_float(r[15]) * inv);
            *reinterpret_cast<uint4*>(dst + c * 16) = w0;
            *reinterpret_cast<uint4*>(dst + c * 16 + 8) = w1;
          }
        }
      } else {
        const size_t prow = (((size_t)b * a.Hkv + hkv) * a.splits + split) * a.M + row;
        float* dst = mine ? (a.cluster ? cpart + row * kCStride : a.part_o + prow * D) : nullptr;
#pragma unroll
        for (int c = c_lo; c < c_hi; ++c) {
          uint32_t r[16];
          tc_ld16(tmem + lane_addr + kOCol + c * 16, r);
          tc_wait_ld();
          if (mine) {
#pragma unroll
            for (int e = 0; e < 16; e += 4)
              *reinterpret_cast<float4*>(dst + c * 16 + e) =
                  make_float4(__uint_as_float(r[e]) * inv, __uint_as_float(r[e + 1]) * inv,
                              __uint_as_float(r[e + 2]) * inv, __uint_as_float(r[e + 3]) * inv);
          }
        }
        if (mine && sub == 0) {
          const float lse = lsum > 0.f ? m_ref + log2f(lsum) : -INFINITY;
          if (a.cluster) clse[row] = lse; else a.part_lse[prow] = lse;
        }
      }
    } else if (n == 0 && a.splits > 1 && mine) {
      const size_t prow = (((size_t)b * a.Hkv + hkv) * a.splits + split) * a.M + row;
      float* dst = a.cluster ? cpart + row * kCStride : a.part_o + prow * D;
      for (int d = c_lo * 16; d < c_hi * 16; ++d) dst[d] = 0.f;
      if (sub == 0) {
        if (a.cluster) clse[row] = -INFINITY; else a.part_lse[prow] = -INFINITY;
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tc_dealloc(tmem, kTmemCols);
  }
  if (a.cluster) cluster_merge<D>(a, b, hkv, k_s, warp - 3, lane);
}

}  // namespace

namespace sbd {

size_t attn_tc_smem_bytes(int D) {
  const int sub = D / 64;
  const bool p_in_k = D == 128;
  const int pairs = p_in_k ? 3 : 4;
  return 1024 + (size_t)sub * kRows * 128 + (p_in_k ? 0 : 4 * kRows * 128) +
         (size_t)pairs * 2 * sub * kPairKeys * 128;
}

static size_t attn_wide_smem_bytes(int D) {
  const int sub = D / 64;
  const int v_slots = D == 128 ? wide_v_slots<128>() : wide_v_slots<64>();
  return 1024 + (size_t)sub * kRows * 128 + (size_t)kWideKSlots * sub * kTriKeys * 128 +
         (size_t)v_slots * sub * kTileKeys * 128;
}

// The kernel for head dimension D and M packed rows: up to 64 rows
// attn_tc_kernel with every row copied into both lane halves, above that
// attn_wide_kernel.
struct TcKernel {
  const void* fn;
  int threads;
  size_t smem;
};
static TcKernel attn_tc_kernel_for(int D, int M) {
  if (M <= kRows / 2)
    return TcKernel{D == 128 ? (const void*)attn_tc_kernel<128, 2> : (const void*)attn_tc_kernel<64, 2>,
                    kThreads, attn_tc_smem_bytes(D)};
  return TcKernel{D == 128 ? (const void*)attn_wide_kernel<128> : (const void*)attn_wide_kernel<64>,
                  kWideThreads, attn_wide_smem_bytes(D)};
}

bool attn_tc_cluster_ok(const AttnPlan& p, int splits) {
  // Whether every (sequence, KV head)'s `splits` CTAs can run as one cluster,
  // all clusters at once.  The device's answer per (device, kernel, cluster
  // size) is kept; the call is on every launch's host path.
  struct Entry {
    int dev;
    const void* fn;
    int splits;
    int clusters;
  };
  static std::mutex mu;
  static Entry cache[32];
  static int n_cache = 0;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  const TcKernel kern = attn_tc_kernel_for(p.D, p.M);
  const void* fn = kern.fn;
  int clusters = -1;
  {
    std::lock_guard<std::mutex> lock(mu);
    for (int i = 0; i < n_cache; ++i)
      if (cache[i].dev == dev && cache[i].fn == fn && cache[i].splits == splits)
        clusters = cache[i].clusters;
  }
  if (clusters < 0) {
    clusters = max_active_clusters(fn, dim3(splits, p.Hkv, p.B), dim3(kern.threads), kern.smem,
                                   splits);
    std::lock_guard<std::mutex> lock(mu);
    if (n_cache < 32) cache[n_cache++] = Entry{dev, fn, splits, clusters};
  }
  return (long long)clusters >= (long long)p.B * p.Hkv;
}

sbd_status attn_tc_launch(const AttnPlan& p, const CUtensorMap& tk, const CUtensorMap& tv,
                          const void* q, const int32_t* lens, const void* kb, const void* vb,
                          void* out, float* part_o, float* part_lse, void* kc_app,
                          void* vc_app, cudaStream_t st) {
  TcArgs a;
  a.q = (const __nv_bfloat16*)q;
  a.kb = (const __nv_bfloat16*)kb;
  a.vb = (const __nv_bfloat16*)vb;
  a.lens = lens;
  a.out = (__nv_bfloat16*)out;
  a.part_o = part_o;
  a.part_lse = part_lse;
  a.err = device_error_word();
  a.B = p.B;
  a.k = p.k;
  a.Hq = p.Hq;
  a.Hkv = p.Hkv;
  a.G = p.G;
  a.M = p.M;
  a.Lmax = p.Lmax;
  a.splits = p.splits;
  a.n_causal = p.n_causal;
  a.order = p.order ? 1 : 0;
  a.kc_app = (__nv_bfloat16*)kc_app;
  a.vc_app = (__nv_bfloat16*)vc_app;
  a.scale_log2 = p.scale_log2;
  a.cluster = p.cluster ? 1 : 0;
  const TcKernel kern = attn_tc_kernel_for(p.D, p.M);
  const size_t smem = kern.smem;
  const void* fn = kern.fn;
  cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return cuda_fail(e, "cudaFuncSetAttribute(attn_tc_kernel)");
  // The block keys/values [B, k, Hkv, D] as 4-D tensors (D, Hkv, k, B), read
  // in the cache tiles' boxes (64 columns x 64 rows, 128-byte swizzle): the
  // rows past k are outside the tensor and arrive as zeros.
  CUtensorMap kb_map, vb_map;
  {
    const uint64_t dims[4] = {(uint64_t)p.D, (uint64_t)p.Hkv, (uint64_t)p.k, (uint64_t)p.B};
    const uint64_t strides[3] = {(uint64_t)p.D * 2, (uint64_t)p.Hkv * p.D * 2,
                                 (uint64_t)p.k * p.Hkv * p.D * 2};
    const uint32_t box[4] = {64, 1, (uint32_t)kTileKeys, 1};
    sbd_status s = encode_tensor_map(&kb_map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, (void*)kb, dims,
                                     strides, box, CU_TENSOR_MAP_SWIZZLE_128B);
    if (s != SBD_OK) return s;
    s = encode_tensor_map(&vb_map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, (void*)vb, dims, strides,
                          box, CU_TENSOR_MAP_SWIZZLE_128B);
    if (s != SBD_OK) return s;
  }
  CUtensorMap k_map = tk, v_map = tv;
  void* args[] = {(void*)&k_map, (void*)&v_map, (void*)&kb_map, (void*)&vb_map, (void*)&a};
  return launch_pdl(fn, dim3(p.splits, p.Hkv, p.B), dim3(kern.threads), smem, st, args,
                    "attn_tc_kernel launch", p.cluster ? p.splits : 1);
}

}  // namespace sbd

