// Block attention of one SBD forward (arXiv 2509.04185, Eq. 5; inference
// mask of Fig. 3): the k block queries of a sequence attend to its exact KV
// cache (all of it lies in their past) and bidirectionally to the k block
// keys.  This file holds the plan (KV splits per (sequence, KV head), the
// in-cluster merge or the workspace), the launch, the split merge kernel
// for plans whose splits do not form a cluster, and the fp32 variant; the
// bf16 kernels are the tcgen05 ones of block_attention_tc.cu:
//
//   * one CTA per (KV split, KV head, sequence); the G = Hq/Hkv query heads
//     that share a KV head are packed with the k block rows into one
//     M = G*k row tile (row r = i*G + g), so each K/V byte is read once;
//   * with more than one split, each CTA's normalised partial output and
//     log-sum-exp are merged inside its thread-block cluster, or written to
//     the workspace and merged by attn_combine_kernel.
//
// First iteration of a block after the previous one (Algorithm 3, "first
// iteration and t >= k"): the leading n_causal block rows are the previous
// block's tokens, causal among themselves, and their keys/values are written
// into the cache at L_b .. L_b + n_causal - 1 by the warp that brings the
// block tile in.
//
// The fp32 variant (attn_f32_kernel) is a plain SIMT kernel with fp32 FMAs
// throughout, used for fp32 inputs.
#include <math.h>

#include "sbd_internal.cuh"

namespace {

using namespace sbd_dev;

constexpr int kTileKeys = 64;
// Largest batch for which the CTAs of a multi-wave launch take the
// sequences longest first.
constexpr int kOrderMaxB = 128;
constexpr float kLog2e = 1.4426950408889634f;

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
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
  if (p.bf16 && p.B > 0 && p.splits >= 2) {
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
  return p;
}

size_t attn_workspace_bytes(const AttnPlan& p) {
  if (p.splits <= 1 || p.cluster) return 0;
  const size_t n = (size_t)p.B * p.Hkv * p.splits * p.M;
  return align_up(n * p.D * sizeof(float), 256) + align_up(n * sizeof(float), 256);
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

  // partials of a split that does not merge inside a cluster
  const size_t n = (size_t)p.B * p.Hkv * p.splits * p.M;
  const bool use_ws = p.splits > 1 && !p.cluster;
  float* part_o = use_ws ? (float*)ws : nullptr;
  float* part_lse = use_ws ? (float*)((char*)ws + align_up(n * p.D * sizeof(float), 256)) : nullptr;

  // Every bf16 shape runs on the tcgen05 kernels (block_attention_tc.cu).
  // Up to 16 packed rows a mma.sync kernel had measured faster than the
  // first tcgen05 form; against the current one it lost at every row count
  // (16 rows, batch 16, KV 8192: 91.2 against 88.9 us; batch 1, KV 4096,
  // 4 rows: 25.4 against 21.3 us) and was removed.
  s = attn_tc_launch(p, tk, tv, q, lens, kb, vb, out, part_o, part_lse, kc_app, vc_app, st);
  if (s != SBD_OK) return s;
  if (use_ws) {
    const float* po = part_o;
    const float* pl = part_lse;
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
