// Block attention of one SBD forward (arXiv 2509.04185, Eq. 5; inference
// mask of Fig. 3): the k block queries of a sequence attend to its exact KV
// cache (all of it lies in their past) and bidirectionally to the k block
// keys.  Flash-decoding structure on sm_103a:
//
//   * one CTA per (KV split, KV head, sequence); the G = Hq/Hkv query heads
//     that share a KV head are packed with the k block rows into one
//     M = G*k row tile (row r = i*G + g), so each K/V byte is read once;
//   * a producer warp streams 64-key K/V tiles into a 4-stage shared-memory
//     ring with TMA (128-byte swizzle, completion on mbarriers); the block
//     keys/values (not cached, k <= 32 rows) are the last tile of the last
//     split and are copied in by the same warp;
//   * compute warps own 16 query rows each and, when M is small, a slice of
//     every key tile; S = Q K^T and O += P V run on bf16 mma.sync with fp32
//     accumulators in registers; the mask (cache key < L_b, block key < k,
//     block key j <= i for a causal block row i < n_causal) is applied to
//     the score registers; the online softmax keeps its row
//     max and sum per thread and reduces them across the 4 threads of a row
//     with shuffles;
//   * with more than one split, each CTA writes its normalised partial
//     output and log-sum-exp, merged by attn_combine_kernel.
//
// First iteration of a block after the previous one (Algorithm 3, "first
// iteration and t >= k"): the leading n_causal block rows are the previous
// block's tokens, causal among themselves, and their keys/values are written
// into the cache at L_b .. L_b + n_causal - 1 by the warp that copies the
// block tile in (one CTA per (KV head, sequence)).
//
// The fp32 variant (attn_f32_kernel) is a plain SIMT kernel with fp32 FMAs
// throughout, used for fp32 inputs.
#include <math.h>

#include "sbd_internal.cuh"

namespace {

using namespace sbd_dev;

constexpr int kTileKeys = 64;
constexpr int kMaxStages = 4;
// Ring depth cap (chosen by measurement).
constexpr int kStageCap = 3;
// Largest batch for which the CTAs of a multi-wave launch take the
// sequences longest first.
constexpr int kOrderMaxB = 128;
// bf16 attention runs on the tcgen05 kernel (block_attention_tc.cu) rather
// than the mma.sync kernel of this file from this many packed rows on.
constexpr int kTcMinRows = 17;
constexpr float kLog2e = 1.4426950408889634f;

// ------------------------------------------------------------ mma helpers
__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                        uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1,
                                          uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
// D = A(16x16 bf16, row) * B(16x8 bf16, col) + D, fp32 accumulate.
__device__ __forceinline__ void mma_bf16(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                         uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

// Address of (row, 16-byte chunk c) inside a [64 rows x 128 B] sub-tile laid
// out by TMA with the 128-byte swizzle (chunk index XOR row % 8).
__device__ __forceinline__ uint32_t swz(uint32_t base, int row, int chunk) {
  return base + row * 128 + (((chunk ^ (row & 7)) & 7) << 4);
}

struct AttnArgs {
  const __nv_bfloat16* q;
  const __nv_bfloat16* kb;
  const __nv_bfloat16* vb;
  const int32_t* lens;
  __nv_bfloat16* out;        // final output (splits == 1)
  float* part_o;             // [B, Hkv, S, M, D] (splits > 1)
  float* part_lse;           // [B, Hkv, S, M]
  int* err;
  __nv_bfloat16* kc_app;     // writable caches for the causal rows' keys/values, or NULL
  __nv_bfloat16* vc_app;
  int B, k, Hq, Hkv, G, M, Lmax, splits, MT, KG, stages, n_causal;
  int order;                 // blockIdx.z -> sequence by descending length
  float scale_log2;
};

template <int D, int NK>
__global__ void __launch_bounds__(288)
attn_bf16_kernel(const __grid_constant__ CUtensorMap tmap_k,
                 const __grid_constant__ CUtensorMap tmap_v, const AttnArgs a) {
  constexpr int kSub = D / 64;                       // 128-B column sub-tiles per row
  constexpr int kSubBytes = kTileKeys * 128;         // 8 KB
  constexpr int kStageBytes = 2 * kSub * kSubBytes;  // K then V
  constexpr int kDT = D / 8;                         // n-tiles of the output
  constexpr int kKS = D / 16;                        // k-steps of Q K^T
  constexpr int kNT = NK / 8;                        // score n-tiles per warp and tile

  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[kMaxStages];
  __shared__ __align__(8) uint64_t empty_bar[kMaxStages];

  const uint32_t smem_base = (smem_u32(smem_raw) + 1023u) & ~1023u;
  uint8_t* smem_gen = smem_raw + (smem_base - smem_u32(smem_raw));
  // The key-group merge reuses the ring once every tile has been consumed.
  float* merge_buf = reinterpret_cast<float*>(smem_gen);
  const int kStages = a.stages;

  const int NW = a.MT * a.KG;                        // compute warps
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int split = blockIdx.x, hkv = blockIdx.y;
  __shared__ int b_pick;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], NW);
    }
    fence_mbar_init();
  }
  // Everything below may read what the previous kernel on the stream wrote.
  grid_dependency_wait();
  if (a.order) {
    longest_first_pick(a.lens, a.B, a.Lmax, blockIdx.z, &b_pick);
    __syncthreads();
  }
  const int b = a.order ? b_pick : (int)blockIdx.z;

  int len = a.lens[b];
  if (len < 0 || len > a.Lmax) {
    if (threadIdx.x == 0 && split == 0 && hkv == 0) record_error(a.err, SBD_DEVERR_CACHE_LEN);
    len = len < 0 ? 0 : a.Lmax;
  }
  const int n_cache_tiles = (len + kTileKeys - 1) / kTileKeys;
  const int n_tiles = n_cache_tiles + 1;             // + the block tile
  const int t_begin = (int)((long long)split * n_tiles / a.splits);
  const int t_end = (int)((long long)(split + 1) * n_tiles / a.splits);
  __syncthreads();

  if (warp == NW) {
    // ------------------------------------------------ producer warp
    if (lane == 0) {
      tma_prefetch_desc(&tmap_k);
      tma_prefetch_desc(&tmap_v);
    }
    // The split that ends with the block tile asks for the block rows' keys
    // and values now (into L2); it copies them after its cache tiles.
    if (t_end == n_tiles)
      for (int c = lane; c < 2 * a.k * (D / 64); c += 32) {
        const int row = c / (2 * (D / 64)), part = c % (2 * (D / 64));
        const __nv_bfloat16* src = part < D / 64 ? a.kb : a.vb;
        prefetch_l2(src + (((size_t)b * a.k + row) * a.Hkv + hkv) * D + (part % (D / 64)) * 64);
      }
    int it = 0;
    for (int t = t_begin; t < t_end; ++t, ++it) {
      const int stage = it % kStages;
      const uint32_t ph = (it / kStages) & 1;
      if (!mbar_wait(&empty_bar[stage], ph ^ 1, a.err)) break;
      const uint32_t kbase = smem_base + stage * kStageBytes;
      const uint32_t vbase = kbase + kSub * kSubBytes;
      if (t < n_cache_tiles) {
        if (lane == 0) {
          mbar_arrive_expect_tx(&full_bar[stage], kStageBytes);
          for (int h = 0; h < kSub; ++h) {
            tma_load_4d(smem_gen + (kbase - smem_base) + h * kSubBytes, &tmap_k, &full_bar[stage],
                        64 * h, hkv, t * kTileKeys, b);
            tma_load_4d(smem_gen + (vbase - smem_base) + h * kSubBytes, &tmap_v, &full_bar[stage],
                        64 * h, hkv, t * kTileKeys, b);
          }
        }
      } else {
        // Block keys/values: rows j < k copied, rows k..63 zero.  Each batch
        // issues all of a lane's loads before its stores (shared stores are
        // volatile asm), so that it costs one memory round trip.
        constexpr int chunks_per_row = D / 8;                   // 16-byte chunks
        constexpr int kBatch = 8;                               // chunks per lane per batch
        const int n_valid = a.k * chunks_per_row;               // chunks of rows < k
        for (int c0 = 0; c0 < kTileKeys * chunks_per_row; c0 += 32 * kBatch) {
          uint4 kv[kBatch], vv[kBatch];
#pragma unroll
          for (int e = 0; e < kBatch; ++e) {
            const int c = c0 + e * 32 + lane;
            kv[e] = make_uint4(0, 0, 0, 0);
            vv[e] = make_uint4(0, 0, 0, 0);
            if (c < n_valid) {
              const size_t off =
                  (((size_t)b * a.k + c / chunks_per_row) * a.Hkv + hkv) * D + (c % chunks_per_row) * 8;
              kv[e] = *reinterpret_cast<const uint4*>(a.kb + off);
              vv[e] = *reinterpret_cast<const uint4*>(a.vb + off);
            }
          }
#pragma unroll
          for (int e = 0; e < kBatch; ++e) {
            const int c = c0 + e * 32 + lane;
            const int j = c / chunks_per_row, cc = c % chunks_per_row;
            if (a.kc_app && c < n_valid && j < a.n_causal && len + a.n_causal <= a.Lmax) {
              // a causal row enters the cache (positions >= len are read by
              // no split of this call, or masked and zeroed where they are)
              const size_t dst = (((size_t)b * a.Lmax + len + j) * a.Hkv + hkv) * D + cc * 8;
              *reinterpret_cast<uint4*>(a.kc_app + dst) = kv[e];
              *reinterpret_cast<uint4*>(a.vc_app + dst) = vv[e];
            }
            const int h = cc / 8, c8 = cc % 8;
            const uint32_t ka = swz(kbase + h * kSubBytes, j, c8);
            const uint32_t va = swz(vbase + h * kSubBytes, j, c8);
            asm volatile("st.shared.v4.b32 [%0], {%1,%2,%3,%4};" ::"r"(ka), "r"(kv[e].x),
                         "r"(kv[e].y), "r"(kv[e].z), "r"(kv[e].w)
                         : "memory");
            asm volatile("st.shared.v4.b32 [%0], {%1,%2,%3,%4};" ::"r"(va), "r"(vv[e].x),
                         "r"(vv[e].y), "r"(vv[e].z), "r"(vv[e].w)
                         : "memory");
          }
        }
        if (a.kc_app && lane == 0 && len + a.n_causal > a.Lmax)
          record_error(a.err, SBD_DEVERR_CACHE_LEN);
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(&full_bar[stage]);
      }
    }
    // Wait for this warp's copies still in flight before the CTA may exit.
    if (lane == 0) {
      const int issued = it;
      for (int q = issued - kStages > 0 ? issued - kStages : 0; q < issued; ++q)
        mbar_wait(&full_bar[q % kStages], (q / kStages) & 1, a.err);
    }
  } else if (warp < NW) {
    // ------------------------------------------------ compute warps
    const int rt = warp % a.MT, kg = warp / a.MT;    // NK keys of each tile per warp
    const int r0 = rt * 16 + (lane >> 2), r1 = r0 + 8;
    const int qc = (lane & 3) * 2;

    // Q fragments (A operand), rows r0/r1, zero for padding rows.
    uint32_t qa[kKS][4];
    {
      const __nv_bfloat16* q0 = nullptr;
      const __nv_bfloat16* q1 = nullptr;
      if (r0 < a.M)
        q0 = a.q + (((size_t)b * a.k + r0 / a.G) * a.Hq + hkv * a.G + r0 % a.G) * D;
      if (r1 < a.M)
        q1 = a.q + (((size_t)b * a.k + r1 / a.G) * a.Hq + hkv * a.G + r1 % a.G) * D;
#pragma unroll
      for (int ks = 0; ks < kKS; ++ks) {
        const int c = ks * 16 + qc;
        qa[ks][0] = q0 ? *reinterpret_cast<const uint32_t*>(q0 + c) : 0u;
        qa[ks][1] = q1 ? *reinterpret_cast<const uint32_t*>(q1 + c) : 0u;
        qa[ks][2] = q0 ? *reinterpret_cast<const uint32_t*>(q0 + c + 8) : 0u;
        qa[ks][3] = q1 ? *reinterpret_cast<const uint32_t*>(q1 + c + 8) : 0u;
      }
    }

    float o[kDT][4];
#pragma unroll
    for (int i = 0; i < kDT; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
    float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;

    // ldmatrix lane roles
    const int lm = lane >> 3, lr = lane & 7;

    int it = 0;
    bool ok = true;
    for (int t = t_begin; t < t_end; ++t, ++it) {
      const int stage = it % kStages;
      const uint32_t ph = (it / kStages) & 1;
      if (!mbar_wait(&full_bar[stage], ph, a.err)) {
        ok = false;
        break;
      }
      const bool block_tile = t >= n_cache_tiles;
      const int valid = block_tile ? a.k : min(kTileKeys, len - t * kTileKeys);
      // causal rows of the block see the block keys j <= i only
      int valid0 = valid, valid1 = valid;
      if (block_tile) {
        if (r0 / a.G < a.n_causal) valid0 = r0 / a.G + 1;
        if (r1 / a.G < a.n_causal) valid1 = r1 / a.G + 1;
      }
      const uint32_t kbase = smem_base + stage * kStageBytes;
      const uint32_t vbase = kbase + kSub * kSubBytes;
      const int key0 = kg * NK;

      // S = Q K^T over this warp's NK keys of the tile: NK/8 independent
      // accumulators per k-step.
      float s[kNT][4];
#pragma unroll
      for (int n = 0; n < kNT; ++n) s[n][0] = s[n][1] = s[n][2] = s[n][3] = 0.f;
#pragma unroll
      for (int ks = 0; ks < kKS; ++ks) {
#pragma unroll
        for (int np = 0; np < NK / 16; ++np) {
          const int key = key0 + np * 16 + ((lm >= 2) ? 8 : 0) + lr;
          const int d = ks * 16 + ((lm & 1) ? 8 : 0);
          uint32_t b0, b1, b2, b3;
          ldsm_x4(swz(kbase + (d >> 6) * kSubBytes, key, (d & 63) >> 3), b0, b1, b2, b3);
          mma_bf16(s[2 * np], qa[ks], b0, b1);
          mma_bf16(s[2 * np + 1], qa[ks], b2, b3);
        }
      }
      // scale + mask in registers, then one online-softmax update per tile
      float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
      for (int n = 0; n < kNT; ++n) {
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          const int key = key0 + n * 8 + qc + e;
          s[n][e] = key < valid0 ? s[n][e] * a.scale_log2 : -INFINITY;
          s[n][2 + e] = key < valid1 ? s[n][2 + e] * a.scale_log2 : -INFINITY;
          mx0 = fmaxf(mx0, s[n][e]);
          mx1 = fmaxf(mx1, s[n][2 + e]);
        }
      }
      mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
      mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
      mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
      mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
      const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);
      const float mu0 = (mn0 == -INFINITY) ? 0.f : mn0;
      const float mu1 = (mn1 == -INFINITY) ? 0.f : mn1;
      const float al0 = exp2f(m0 - mu0), al1 = exp2f(m1 - mu1);
      m0 = mn0;
      m1 = mn1;
      float ps0 = 0.f, ps1 = 0.f;
#pragma unroll
      for (int n = 0; n < kNT; ++n) {
        s[n][0] = ex2_ftz(s[n][0] - mu0);
        s[n][1] = ex2_ftz(s[n][1] - mu0);
        s[n][2] = ex2_ftz(s[n][2] - mu1);
        s[n][3] = ex2_ftz(s[n][3] - mu1);
        ps0 += s[n][0] + s[n][1];
        ps1 += s[n][2] + s[n][3];
      }
      l0 = l0 * al0 + ps0;
      l1 = l1 * al1 + ps1;
#pragma unroll
      for (int i = 0; i < kDT; ++i) {
        o[i][0] *= al0;
        o[i][1] *= al0;
        o[i][2] *= al1;
        o[i][3] *= al1;
      }
      // O += P V, 16 keys per k-step.  Value rows past `valid` are zeroed in
      // registers so that unused cache slots (possibly NaN) never meet a zero
      // probability.
#pragma unroll
      for (int kk = 0; kk < NK / 16; ++kk) {
        const int j0 = key0 + kk * 16;
        uint32_t pa[4];
        pa[0] = pack_bf16(s[2 * kk][0], s[2 * kk][1]);
        pa[1] = pack_bf16(s[2 * kk][2], s[2 * kk][3]);
        pa[2] = pack_bf16(s[2 * kk + 1][0], s[2 * kk + 1][1]);
        pa[3] = pack_bf16(s[2 * kk + 1][2], s[2 * kk + 1][3]);
        const bool sanitize = j0 + 16 > valid;
        const int ka = j0 + qc, kb8 = j0 + 8 + qc;
        const uint32_t m_a = (ka < valid ? 0xffffu : 0u) | (ka + 1 < valid ? 0xffff0000u : 0u);
        const uint32_t m_b = (kb8 < valid ? 0xffffu : 0u) | (kb8 + 1 < valid ? 0xffff0000u : 0u);
#pragma unroll
        for (int dp = 0; dp < kDT / 2; ++dp) {
          const int key = j0 + ((lm & 1) ? 8 : 0) + lr;
          const int d = dp * 16 + ((lm >= 2) ? 8 : 0);
          uint32_t b0, b1, b2, b3;
          ldsm_x4_t(swz(vbase + (d >> 6) * kSubBytes, key, (d & 63) >> 3), b0, b1, b2, b3);
          if (sanitize) {
            b0 &= m_a;
            b1 &= m_b;
            b2 &= m_a;
            b3 &= m_b;
          }
          mma_bf16(o[2 * dp], pa, b0, b1);
          mma_bf16(o[2 * dp + 1], pa, b2, b3);
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty_bar[stage]);
    }
    (void)ok;
    grid_dependents_launch();

    // Row sums across the 4 threads of a row.
    l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
    l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
    l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
    l1 += __shfl_xor_sync(0xffffffffu, l1, 2);

    // Merge the key groups of the same row tile through shared memory.
    if (a.KG > 1) {
      // layout per warp: [16 rows][D] o, then [16] m, [16] l
      float* mine = merge_buf + warp * (16 * D + 32);
      // every compute warp is done reading the ring before it is reused
      asm volatile("bar.sync 1, %0;" ::"r"(NW * 32) : "memory");
      if (kg > 0) {
#pragma unroll
        for (int i = 0; i < kDT; ++i) {
          const int c = i * 8 + qc;
          mine[(lane >> 2) * D + c] = o[i][0];
          mine[(lane >> 2) * D + c + 1] = o[i][1];
          mine[((lane >> 2) + 8) * D + c] = o[i][2];
          mine[((lane >> 2) + 8) * D + c + 1] = o[i][3];
        }
        if ((lane & 3) == 0) {
          mine[16 * D + (lane >> 2)] = m0;
          mine[16 * D + (lane >> 2) + 8] = m1;
          mine[16 * D + 16 + (lane >> 2)] = l0;
          mine[16 * D + 16 + (lane >> 2) + 8] = l1;
        }
      }
      asm volatile("bar.sync 1, %0;" ::"r"(NW * 32) : "memory");
      if (kg == 0) {
        for (int g2 = 1; g2 < a.KG; ++g2) {
          const float* other = merge_buf + (g2 * a.MT + rt) * (16 * D + 32);
          const float om0 = other[16 * D + (lane >> 2)];
          const float om1 = other[16 * D + (lane >> 2) + 8];
          const float ol0 = other[16 * D + 16 + (lane >> 2)];
          const float ol1 = other[16 * D + 16 + (lane >> 2) + 8];
          const float nm0 = fmaxf(m0, om0), nm1 = fmaxf(m1, om1);
          const float u0 = (nm0 == -INFINITY) ? 0.f : nm0;
          const float u1 = (nm1 == -INFINITY) ? 0.f : nm1;
          const float sa0 = exp2f(m0 - u0), sb0 = exp2f(om0 - u0);
          const float sa1 = exp2f(m1 - u1), sb1 = exp2f(om1 - u1);
#pragma unroll
          for (int i = 0; i < kDT; ++i) {
            const int c = i * 8 + qc;
            o[i][0] = o[i][0] * sa0 + other[(lane >> 2) * D + c] * sb0;
            o[i][1] = o[i][1] * sa0 + other[(lane >> 2) * D + c + 1] * sb0;
            o[i][2] = o[i][2] * sa1 + other[((lane >> 2) + 8) * D + c] * sb1;
            o[i][3] = o[i][3] * sa1 + other[((lane >> 2) + 8) * D + c + 1] * sb1;
          }
          l0 = l0 * sa0 + ol0 * sb0;
          l1 = l1 * sa1 + ol1 * sb1;
          m0 = nm0;
          m1 = nm1;
        }
      }
    }

    if (kg == 0) {
      const float inv0 = l0 > 0.f ? 1.f / l0 : 0.f;
      const float inv1 = l1 > 0.f ? 1.f / l1 : 0.f;
      if (a.splits == 1) {
#pragma unroll
        for (int rr = 0; rr < 2; ++rr) {
          const int r = rr ? r1 : r0;
          if (r >= a.M) continue;
          const float inv = rr ? inv1 : inv0;
          __nv_bfloat16* dst =
              a.out + (((size_t)b * a.k + r / a.G) * a.Hq + hkv * a.G + r % a.G) * D;
#pragma unroll
          for (int i = 0; i < kDT; ++i) {
            const int c = i * 8 + qc;
            *reinterpret_cast<uint32_t*>(dst + c) =
                pack_bf16(o[i][2 * rr] * inv, o[i][2 * rr + 1] * inv);
          }
        }
      } else {
        const size_t pbase = (((size_t)b * a.Hkv + hkv) * a.splits + split) * a.M;
#pragma unroll
        for (int rr = 0; rr < 2; ++rr) {
          const int r = rr ? r1 : r0;
          if (r >= a.M) continue;
          const float inv = rr ? inv1 : inv0;
          const float l = rr ? l1 : l0, m = rr ? m1 : m0;
          float* dst = a.part_o + (pbase + r) * D;
#pragma unroll
          for (int i = 0; i < kDT; ++i) {
            const int c = i * 8 + qc;
            *reinterpret_cast<float2*>(dst + c) =
                make_float2(o[i][2 * rr] * inv, o[i][2 * rr + 1] * inv);
          }
          if ((lane & 3) == 0) a.part_lse[pbase + r] = l > 0.f ? m + log2f(l) : -INFINITY;
        }
      }
    }
  }
}

// Merge of the split partials: O = sum_s 2^(lse_s - lse) O_s.  One warp per
// (packed row, KV head, sequence), kCombineRows rows per CTA: lane s holds
// the log-sum-exp of split s, and each lane owns D / 32 consecutive output
// columns.  The kernel is latency-bound: for each group of 32 splits a lane
// requests the log-sum-exp and its columns of all of them before it uses
// any, so that one memory round trip covers the group; groups merge online.
// (One 128-thread CTA per row instead took 12.6 us for 2048 CTAs at 4
// splits, its time growing with the CTA count.)
constexpr int kCombineRows = 4;

template <int D, typename OutT>
__global__ void __launch_bounds__(32 * kCombineRows)
attn_combine_kernel(const float* __restrict__ part_o, const float* __restrict__ part_lse,
                    OutT* __restrict__ out, int k, int Hq, int Hkv, int G, int M, int splits) {
  constexpr int kPer = D / 32;                 // columns per lane: 2 or 4
  grid_dependency_wait();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r = blockIdx.x * kCombineRows + warp, hkv = blockIdx.y, b = blockIdx.z;
  if (r >= M) return;
  const size_t pair = (size_t)b * Hkv + hkv;
  const float* lse = part_lse + pair * splits * M + r;
  const float* po = part_o + (pair * splits * M + r) * D + kPer * lane;
  const size_t po_stride = (size_t)M * D;
  float mx = -INFINITY, sum = 0.f, acc[kPer];
#pragma unroll
  for (int c = 0; c < kPer; ++c) acc[c] = 0.f;
  for (int s0 = 0; s0 < splits; s0 += 32) {
    const int n = min(32, splits - s0);
    const float l_lane = lane < n ? lse[(size_t)(s0 + lane) * M] : -INFINITY;
    float v[32][kPer];
#pragma unroll
    for (int e = 0; e < 32; ++e) {
      if (e < n) {
        const float* src = po + (size_t)(s0 + e) * po_stride;
        if constexpr (kPer == 4) {
          const float4 x = *reinterpret_cast<const float4*>(src);
          v[e][0] = x.x; v[e][1] = x.y; v[e][2] = x.z; v[e][3] = x.w;
        } else {
          const float2 x = *reinterpret_cast<const float2*>(src);
          v[e][0] = x.x; v[e][1] = x.y;
        }
      } else {
#pragma unroll
        for (int c = 0; c < kPer; ++c) v[e][c] = 0.f;
      }
    }
    const float gm = warp_max(l_lane);
    if (gm == -INFINITY) continue;               // every split of the group is empty
    if (gm > mx) {
      const float c = exp2f(mx - gm);            // 0 while mx = -inf
      sum *= c;
#pragma unroll
      for (int e = 0; e < kPer; ++e) acc[e] *= c;
      mx = gm;
    }
#pragma unroll
    for (int e = 0; e < 32; ++e) {
      const float wt = exp2f(__shfl_sync(0xffffffffu, l_lane, e) - mx);   // 0 past n
      sum += wt;
      if (wt > 0.f) {
#pragma unroll
        for (int c = 0; c < kPer; ++c) acc[c] = fmaf(wt, v[e][c], acc[c]);
      }
    }
  }
  const float inv = sum > 0.f ? 1.f / sum : 0.f;
  const size_t o = (((size_t)b * k + r / G) * Hq + hkv * G + r % G) * D + kPer * lane;
  if constexpr (sizeof(OutT) == 2) {
    if constexpr (kPer == 4) {
      uint2 w;
      w.x = pack_bf16(acc[0] * inv, acc[1] * inv);
      w.y = pack_bf16(acc[2] * inv, acc[3] * inv);
      *reinterpret_cast<uint2*>(out + o) = w;
    } else {
      *reinterpret_cast<uint32_t*>(out + o) = pack_bf16(acc[0] * inv, acc[1] * inv);
    }
  } else {
#pragma unroll
    for (int c = 0; c < kPer; ++c) out[o + c] = acc[c] * inv;
  }
}

// ------------------------------------------------------------ fp32 variant
// One CTA per (query row i, query head, sequence); keys in chunks of 128
// with an online softmax; every product and sum in fp32 FMAs.
__global__ void __launch_bounds__(128)
attn_f32_kernel(const float* __restrict__ q, const float* __restrict__ kc,
                const float* __restrict__ vc, const int32_t* __restrict__ lens,
                const float* __restrict__ kb, const float* __restrict__ vb,
                float* __restrict__ out, int* err, int k, int Hq, int Hkv, int D, int Lmax,
                float scale_log2, int n_causal, float* __restrict__ kc_app,
                float* __restrict__ vc_app) {
  __shared__ float qs[128];
  __shared__ float ps[128];
  __shared__ float red[4];
  grid_dependency_wait();
  const int i = blockIdx.x, hq = blockIdx.y, b = blockIdx.z;
  const int G = Hq / Hkv, hkv = hq / G;
  const int tid = threadIdx.x;
  int len = lens[b];
  if (len < 0 || len > Lmax) {
    if (tid == 0) sbd_dev::record_error(err, SBD_DEVERR_CACHE_LEN);
    len = len < 0 ? 0 : Lmax;
  }
  const float* qrow = q + (((size_t)b * k + i) * Hq + hq) * D;
  if (tid < D) qs[tid] = qrow[tid];
  // The first CTA of each KV head writes a causal row's key and value into
  // the cache; the attention below reads cache positions < len only.
  if (kc_app && i < n_causal && hq % G == 0 && tid < D) {
    if (len + n_causal <= Lmax) {
      const size_t dst = (((size_t)b * Lmax + len + i) * Hkv + hkv) * D + tid;
      const size_t src = (((size_t)b * k + i) * Hkv + hkv) * D + tid;
      kc_app[dst] = kb[src];
      vc_app[dst] = vb[src];
    } else if (tid == 0 && i == 0) {
      sbd_dev::record_error(err, SBD_DEVERR_CACHE_LEN);
    }
  }
  __syncthreads();
  // causal rows of the block see the block keys j <= i only
  const int total = len + (i < n_causal ? i + 1 : k);
  float m = -INFINITY, l = 0.f, acc = 0.f;   // acc: output element d = tid
  for (int c0 = 0; c0 < total; c0 += 128) {
    const int u = c0 + tid;
    float s = -INFINITY;
    if (u < total) {
      const float* key = (u < len) ? kc + (((size_t)b * Lmax + u) * Hkv + hkv) * D
                                   : kb + (((size_t)b * k + (u - len)) * Hkv + hkv) * D;
      float dot = 0.f;
      for (int d = 0; d < D; ++d) dot = fmaf(qs[d], key[d], dot);
      s = dot * scale_log2;
    }
    // block max
    float mx = sbd_dev::warp_max(s);
    if ((tid & 31) == 0) red[tid >> 5] = mx;
    __syncthreads();
    mx = fmaxf(fmaxf(red[0], red[1]), fmaxf(red[2], red[3]));
    __syncthreads();
    const float mn = fmaxf(m, mx);
    const float alpha = (m == -INFINITY) ? 0.f : exp2f(m - mn);
    const float p = (s == -INFINITY) ? 0.f : exp2f(s - mn);
    ps[tid] = p;
    float psum = sbd_dev::warp_sum(p);
    if ((tid & 31) == 0) red[tid >> 5] = psum;
    __syncthreads();
    psum = (red[0] + red[1]) + (red[2] + red[3]);
    l = l * alpha + psum;
    m = mn;
    if (tid < D) {
      acc *= alpha;
      const int n = min(128, total - c0);
      for (int j = 0; j < n; ++j) {
        const int uu = c0 + j;
        const float* val = (uu < len) ? vc + (((size_t)b * Lmax + uu) * Hkv + hkv) * D
                                      : vb + (((size_t)b * k + (uu - len)) * Hkv + hkv) * D;
        acc = fmaf(ps[j], val[tid], acc);
      }
    }
    __syncthreads();
  }
  if (tid < D) out[(((size_t)b * k + i) * Hq + hq) * D + tid] = acc / l;
}

}  // namespace

namespace sbd {

// KV splits per (sequence, KV head): one wave of CTAs, each as long as
// possible.  A CTA pays a fixed start (tensor memory, barriers, Q, the first
// loads' latency) and drain; measured on the long-cache workloads, filling
// further waves with shorter CTAs loses more than the idle SMs of one wave.
static int choose_splits(int pairs, int n_tiles_max, int sms) {
  int s = pairs >= sms ? 1 : sms / pairs;
  int max_s = n_tiles_max / 2;
  if (max_s < 1) max_s = 1;
  if (max_s > 32) max_s = 32;
  return s < max_s ? s : max_s;
}

AttnPlan attn_plan(const sbd_attn_desc& d) {
  AttnPlan p;
  p.B = d.batch;
  p.k = d.block_k;
  p.Hq = d.n_q_heads;
  p.Hkv = d.n_kv_heads;
  p.G = d.n_q_heads / d.n_kv_heads;
  p.D = d.head_dim;
  p.Lmax = d.max_cache_len;
  p.M = p.G * p.k;
  p.bf16 = d.dtype == SBD_DTYPE_BF16;
  p.n_causal = 0;
  const float scale = d.scale != 0.f ? d.scale : 1.0f / sqrtf((float)d.head_dim);
  p.scale_log2 = scale * kLog2e;
  const int tiles = (p.Lmax + kTileKeys - 1) / kTileKeys + 1;
  if (!p.bf16) {
    p.splits = 1;
  } else if (d.num_splits > 0) {
    p.splits = d.num_splits;
  } else {
    p.splits = choose_splits(p.B * p.Hkv, tiles, num_sms());
  }
  // tcgen05 path: the splits of a (sequence, KV head) merge in shared memory
  // as one thread-block cluster (at most 16 CTAs) when the device can hold
  // all the clusters at once.  An automatic split count is lowered, down to
  // 3/5 of it, to the largest cluster size that fits (GB300, one 227 KB CTA
  // per SM: 36 clusters of 4, 15 of 8, 7 of 16); at batch 1, Llama-8B, 4096
  // cached keys, 12 splits in clusters took 12.9 us against 13.9 us for 19
  // splits merged by attn_combine_kernel.  Otherwise the partials go through
  // the workspace and attn_combine_kernel.
  p.cluster = false;
  if (p.bf16 && p.M >= kTcMinRows && p.B > 0 && p.splits >= 2) {
    const int hi = p.splits < 16 ? p.splits : 16;
    const int lo = d.num_splits > 0 ? p.splits : (3 * p.splits + 4) / 5;
    for (int s = hi; s >= lo && s >= 2; --s) {
      if (attn_tc_cluster_ok(p, s)) {
        p.splits = s;
        p.cluster = true;
        break;
      }
    }
  }
  // With more CTAs than one wave, the CTAs take the sequences longest first
  // (the pick costs B^2 comparisons per CTA, hence the batch limit).
  p.order = p.bf16 && p.B > 1 && p.B <= kOrderMaxB &&
            (long long)p.B * p.Hkv * p.splits > num_sms();
  // Ring depth: as many stages as a split has tiles, between 2 and 4.
  const int per_split = (tiles + p.splits - 1) / p.splits;
  const int cap = kStageCap < kMaxStages ? kStageCap : kMaxStages;
  p.stages = per_split < 2 ? 2 : (per_split > cap ? cap : per_split);
  // Row tiles of 16 packed rows; small tiles also split every key tile
  // between key groups so that at least 4 (up to 8) warps share the work.
  p.MT = (p.M + 15) / 16;
  p.KG = p.MT >= 5 ? 1 : (p.MT == 4 ? 1 : (p.MT == 3 ? 2 : 4));
  if (p.MT == 1) p.KG = 4;
  return p;
}

size_t attn_workspace_bytes(const AttnPlan& p) {
  if (p.splits <= 1 || p.cluster) return 0;
  const size_t n = (size_t)p.B * p.Hkv * p.splits * p.M;
  return align_up(n * p.D * sizeof(float), 256) + align_up(n * sizeof(float), 256);
}

static size_t attn_smem_bytes(const AttnPlan& p) {
  const size_t ring = (size_t)p.stages * 2 * (p.D / 64) * kTileKeys * 128;
  const size_t merge = p.KG > 1 ? (size_t)p.MT * p.KG * (16 * p.D + 32) * sizeof(float) : 0;
  return 1024 + (ring > merge ? ring : merge);
}

sbd_status attn_launch(const AttnPlan& p, const void* q, const void* kc, const void* vc,
                       const int32_t* lens, const void* kb, const void* vb, void* out, void* ws,
                       void* kc_app, void* vc_app, cudaStream_t st) {
  if (p.B == 0) return SBD_OK;
  int* err = device_error_word();
  if (!p.bf16) {
    const float *qf = (const float*)q, *kcf = (const float*)kc, *vcf = (const float*)vc;
    const float *kbf = (const float*)kb, *vbf = (const float*)vb;
    float* of = (float*)out;
    int k = p.k, Hq = p.Hq, Hkv = p.Hkv, D = p.D, Lmax = p.Lmax;
    float sl2 = p.scale_log2;
    int nc = p.n_causal;
    float* kca = (float*)kc_app;
    float* vca = (float*)vc_app;
    void* args[] = {(void*)&qf,  (void*)&kcf, (void*)&vcf,  (void*)&lens, (void*)&kbf,
                    (void*)&vbf, (void*)&of,  (void*)&err,  (void*)&k,    (void*)&Hq,
                    (void*)&Hkv, (void*)&D,   (void*)&Lmax, (void*)&sl2,  (void*)&nc,
                    (void*)&kca, (void*)&vca};
    return launch_pdl((const void*)attn_f32_kernel, dim3(p.k, p.Hq, p.B), dim3(128), 0, st, args,
                      "attn_f32_kernel launch");
  }

  // 4-D tensor maps over the caches: dims (D, Hkv, Lmax, B), 64x64 boxes.
  CUtensorMap tk, tv;
  const uint64_t dims[4] = {(uint64_t)p.D, (uint64_t)p.Hkv, (uint64_t)p.Lmax, (uint64_t)p.B};
  const uint64_t strides[3] = {(uint64_t)p.D * 2, (uint64_t)p.Hkv * p.D * 2,
                               (uint64_t)p.Lmax * p.Hkv * p.D * 2};
  const uint32_t box[4] = {64, 1, (uint32_t)kTileKeys, 1};
  sbd_status s = encode_tensor_map(&tk, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, (void*)kc, dims,
                                   strides, box, CU_TENSOR_MAP_SWIZZLE_128B);
  if (s != SBD_OK) return s;
  s = encode_tensor_map(&tv, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, (void*)vc, dims, strides, box,
                        CU_TENSOR_MAP_SWIZZLE_128B);
  if (s != SBD_OK) return s;

  AttnArgs a;
  a.q = (const __nv_bfloat16*)q;
  a.kb = (const __nv_bfloat16*)kb;
  a.vb = (const __nv_bfloat16*)vb;
  a.lens = lens;
  a.out = (__nv_bfloat16*)out;
  a.err = err;
  a.B = p.B;
  a.k = p.k;
  a.Hq = p.Hq;
  a.Hkv = p.Hkv;
  a.G = p.G;
  a.M = p.M;
  a.Lmax = p.Lmax;
  a.splits = p.splits;
  a.MT = p.MT;
  a.KG = p.KG;
  a.stages = p.stages;
  a.n_causal = p.n_causal;
  a.order = p.order ? 1 : 0;
  a.kc_app = (__nv_bfloat16*)kc_app;
  a.vc_app = (__nv_bfloat16*)vc_app;
  a.scale_log2 = p.scale_log2;
  const size_t n = (size_t)p.B * p.Hkv * p.splits * p.M;
  const bool use_ws = p.splits > 1 && !p.cluster;
  a.part_o = use_ws ? (float*)ws : nullptr;
  a.part_lse = use_ws ? (float*)((char*)ws + align_up(n * p.D * sizeof(float), 256)) : nullptr;

  // Up to 16 packed rows the mma.sync kernel measures faster (the tcgen05
  // kernel pads every tile to 128 rows); from 17 on, tcgen05, with every row
  // copied into 4, 2 or 1 TMEM lane quadrants so that all SM sub-partitions
  // share the softmax.  Batch 16, KV 8192: 32 rows (k = 8) 115 -> 110 us;
  // 16 rows (k = 4) 104 us on mma.sync against 108 us on tcgen05.
  if (p.M >= kTcMinRows) {
    s = attn_tc_launch(p, tk, tv, q, lens, kb, vb, out, a.part_o, a.part_lse, kc_app, vc_app,
                       st);
    if (s != SBD_OK) return s;
  } else {
  const int NW = a.MT * a.KG;
  const size_t smem = attn_smem_bytes(p);
  const void* fn;
  if (p.D == 128)
    fn = p.KG == 1 ? (const void*)attn_bf16_kernel<128, 64>
                   : (p.KG == 2 ? (const void*)attn_bf16_kernel<128, 32>
                                : (const void*)attn_bf16_kernel<128, 16>);
  else
    fn = p.KG == 1 ? (const void*)attn_bf16_kernel<64, 64>
                   : (p.KG == 2 ? (const void*)attn_bf16_kernel<64, 32>
                                : (const void*)attn_bf16_kernel<64, 16>);
  cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return cuda_fail(e, "cudaFuncSetAttribute(attn_bf16_kernel)");
  {
    void* args[] = {(void*)&tk, (void*)&tv, (void*)&a};
    s = launch_pdl(fn, dim3(p.splits, p.Hkv, p.B), dim3(32 * (NW + 1)), smem, st, args,
                   "attn_bf16_kernel launch");
    if (s != SBD_OK) return s;
  }
  }
  if (use_ws) {
    const float* po = a.part_o;
    const float* pl = a.part_lse;
    __nv_bfloat16* o = (__nv_bfloat16*)out;
    int k = p.k, Hq = p.Hq, Hkv = p.Hkv, G = p.G, M = p.M, S = p.splits;
    void* args[] = {(void*)&po, (void*)&pl, (void*)&o, (void*)&k, (void*)&Hq, (void*)&Hkv,
                    (void*)&G,  (void*)&M,  (void*)&S};
    const void* fn = p.D == 128 ? (const void*)attn_combine_kernel<128, __nv_bfloat16>
                                : (const void*)attn_combine_kernel<64, __nv_bfloat16>;
    s = launch_pdl(fn, dim3((p.M + kCombineRows - 1) / kCombineRows, p.Hkv, p.B),
                   dim3(32 * kCombineRows), 0, st, args, "attn_combine_kernel launch");
    if (s != SBD_OK) return s;
  }
  return SBD_OK;
}

}  // namespace sbd
