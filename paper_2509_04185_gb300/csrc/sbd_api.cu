// C ABI of libsbd: argument validation, workspace sizing, error reporting and
// dispatch to the kernels of block_attention.cu, lm_head.cu and eb_select.cu.
#include <cudaTypedefs.h>
#include <math.h>
#include <stdarg.h>
#include <stdio.h>

#include <mutex>

#include "sbd_internal.cuh"

namespace {

thread_local char g_last_error[512] = "";

constexpr int kMaxDevices = 64;
__device__ int g_device_error = 0;

// Per device: the SM count and the device address of the error word, set
// once both queries have succeeded (a failed query is retried on the next
// call instead of being kept).
struct DeviceCache {
  std::mutex mu;
  bool ready[kMaxDevices] = {false};
  int sms[kMaxDevices] = {0};
  int* err_word[kMaxDevices] = {nullptr};
};
DeviceCache& cache() {
  static DeviceCache c;
  return c;
}

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
std::once_flag g_encode_once;

// The current device's ordinal; an error status (with the reason recorded)
// when it cannot be read or is beyond the table.
sbd_status current_device(int* dev) {
  cudaError_t e = cudaGetDevice(dev);
  if (e != cudaSuccess) return sbd::cuda_fail(e, "cudaGetDevice");
  if (*dev < 0 || *dev >= kMaxDevices)
    return sbd::fail(SBD_ERR_UNSUPPORTED, "device ordinal %d >= %d", *dev, kMaxDevices);
  return SBD_OK;
}

}  // namespace

namespace sbd {

sbd_status device_ready() {
  int dev = 0;
  const sbd_status st = current_device(&dev);
  if (st != SBD_OK) return st;
  DeviceCache& c = cache();
  std::lock_guard<std::mutex> lock(c.mu);
  if (c.ready[dev]) return SBD_OK;
  int sms = 0;
  cudaError_t e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess || sms <= 0) {
    cudaGetLastError();
    return e != cudaSuccess ? cuda_fail(e, "cudaDeviceGetAttribute(MultiProcessorCount)")
                            : fail(SBD_ERR_CUDA, "device %d reports %d SMs", dev, sms);
  }
  void* p = nullptr;
  e = cudaGetSymbolAddress(&p, g_device_error);
  if (e != cudaSuccess) {
    cudaGetLastError();
    return cuda_fail(e, "cudaGetSymbolAddress(device error word)");
  }
  c.sms[dev] = sms;
  c.err_word[dev] = static_cast<int*>(p);
  c.ready[dev] = true;
  return SBD_OK;
}

sbd_status fail(sbd_status st, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_last_error, sizeof(g_last_error), fmt, ap);
  va_end(ap);
  return st;
}

sbd_status cuda_fail(cudaError_t e, const char* what) {
  return fail(SBD_ERR_CUDA, "%s: %s (%s)", what, cudaGetErrorName(e), cudaGetErrorString(e));
}

// Both below are called only after device_ready() succeeded on this thread's
// current device (every launching entry point checks it first).
int num_sms() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return 1;
  std::lock_guard<std::mutex> lock(cache().mu);
  return cache().ready[dev] ? cache().sms[dev] : 1;
}

int* device_error_word() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  std::lock_guard<std::mutex> lock(cache().mu);
  return cache().ready[dev] ? cache().err_word[dev] : nullptr;
}

sbd_status encode_tensor_map(CUtensorMap* map, CUtensorMapDataType dtype, uint32_t rank,
                             void* base, const uint64_t* dims, const uint64_t* strides_bytes,
                             const uint32_t* box, CUtensorMapSwizzle swizzle) {
  std::call_once(g_encode_once, [] {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000,
                                         cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    else
      cudaGetLastError();
  });
  if (!g_encode) return fail(SBD_ERR_CUDA, "cuTensorMapEncodeTiled is not available");
  cuuint64_t d[5];
  cuuint64_t s[4];
  cuuint32_t bx[5], es[5];
  for (uint32_t i = 0; i < rank; ++i) {
    d[i] = dims[i];
    bx[i] = box[i];
    es[i] = 1;
    if (i + 1 < rank) s[i] = strides_bytes[i];
  }
  CUresult r = g_encode(map, dtype, rank, base, d, s, bx, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        swizzle, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(SBD_ERR_CUDA, "cuTensorMapEncodeTiled failed (CUresult %d)", (int)r);
  return SBD_OK;
}

sbd_status launch_pdl(const void* fn, dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                      void** args, const char* what, int cluster_x) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (cluster_x > 1) {
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = (unsigned)cluster_x;
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    cfg.numAttrs = 2;
  }
  cudaError_t e = cudaLaunchKernelExC(&cfg, fn, args);
  if (e != cudaSuccess) return cuda_fail(e, what);
  return SBD_OK;
}

int max_active_clusters(const void* fn, dim3 grid, dim3 block, size_t smem, int cluster_x) {
  if (cluster_x > 8 &&
      cudaFuncSetAttribute(fn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  if (cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) !=
      cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)cluster_x;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, fn, &cfg) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  return n;
}

}  // namespace sbd

using sbd::aligned16;
using sbd::fail;

namespace {

sbd_status check_attn_desc(const sbd_attn_desc* d) {
  if (!d) return fail(SBD_ERR_INVALID_ARG, "desc is NULL");
  if (d->batch < 0 || d->block_k < 1 || d->n_q_heads < 1 || d->n_kv_heads < 1 ||
      d->head_dim < 1 || d->max_cache_len < 0)
    return fail(SBD_ERR_INVALID_ARG,
                "bad sizes: batch=%d block_k=%d n_q_heads=%d n_kv_heads=%d head_dim=%d "
                "max_cache_len=%d",
                d->batch, d->block_k, d->n_q_heads, d->n_kv_heads, d->head_dim,
                d->max_cache_len);
  if (d->dtype != SBD_DTYPE_F32 && d->dtype != SBD_DTYPE_BF16)
    return fail(SBD_ERR_INVALID_ARG, "unknown dtype %d", d->dtype);
  if (!(isfinite(d->scale) && d->scale >= 0.f))
    return fail(SBD_ERR_INVALID_ARG, "scale must be finite and >= 0 (0 = 1/sqrt(D))");
  if (d->n_q_heads % d->n_kv_heads != 0)
    return fail(SBD_ERR_INVALID_ARG, "n_q_heads (%d) must be a multiple of n_kv_heads (%d)",
                d->n_q_heads, d->n_kv_heads);
  if (d->num_splits < 0) return fail(SBD_ERR_INVALID_ARG, "num_splits must be >= 0");
  if (d->block_k > 32) return fail(SBD_ERR_UNSUPPORTED, "block_k %d > 32", d->block_k);
  if (d->head_dim != 64 && d->head_dim != 128)
    return fail(SBD_ERR_UNSUPPORTED, "head_dim %d not in {64, 128}", d->head_dim);
  if (d->dtype == SBD_DTYPE_BF16) {
    const int M = (d->n_q_heads / d->n_kv_heads) * d->block_k;
    if (M > 128)
      return fail(SBD_ERR_UNSUPPORTED, "(Hq/Hkv) * block_k = %d > 128", M);
    if (d->num_splits > 64) return fail(SBD_ERR_UNSUPPORTED, "num_splits %d > 64", d->num_splits);
    if (d->max_cache_len > (1 << 30) / 64)
      return fail(SBD_ERR_UNSUPPORTED, "max_cache_len %d too large", d->max_cache_len);
  }
  return SBD_OK;
}

sbd_status check_head_desc(const sbd_head_desc* d) {
  if (!d) return fail(SBD_ERR_INVALID_ARG, "desc is NULL");
  if (d->batch < 0 || d->block_k < 1 || d->hidden < 1 || d->vocab < 1)
    return fail(SBD_ERR_INVALID_ARG, "bad sizes: batch=%d block_k=%d hidden=%d vocab=%d",
                d->batch, d->block_k, d->hidden, d->vocab);
  if (d->dtype != SBD_DTYPE_F32 && d->dtype != SBD_DTYPE_BF16)
    return fail(SBD_ERR_INVALID_ARG, "unknown dtype %d", d->dtype);
  if ((long long)d->batch * d->block_k > 512)
    return fail(SBD_ERR_UNSUPPORTED, "batch * block_k = %lld > 512",
                (long long)d->batch * d->block_k);
  if (d->dtype == SBD_DTYPE_BF16 && d->hidden % 64 != 0)
    return fail(SBD_ERR_UNSUPPORTED, "hidden %d is not a multiple of 64", d->hidden);
  if (d->dtype == SBD_DTYPE_F32 && d->hidden % 4 != 0)
    return fail(SBD_ERR_UNSUPPORTED, "hidden %d is not a multiple of 4", d->hidden);
  return SBD_OK;
}

sbd_status attn_call(const sbd_attn_desc* desc, int n_causal, const void* q, const void* k_cache,
                     const void* v_cache, const int32_t* cache_len, const void* k_blk,
                     const void* v_blk, void* out, void* workspace, size_t workspace_bytes,
                     void* kc_app, void* vc_app, void* stream) {
  sbd_status s = check_attn_desc(desc);
  if (s != SBD_OK) return s;
  if (desc->batch == 0) return SBD_OK;
  const void* ptrs[] = {q, k_cache, v_cache, cache_len, k_blk, v_blk, out};
  const char* names[] = {"q", "k_cache", "v_cache", "cache_len", "k_blk", "v_blk", "out"};
  for (int i = 0; i < 7; ++i) {
    if (!ptrs[i]) return fail(SBD_ERR_INVALID_ARG, "%s is NULL", names[i]);
    if (!aligned16(ptrs[i])) return fail(SBD_ERR_INVALID_ARG, "%s is not 16-byte aligned", names[i]);
  }
  s = sbd::device_ready();
  if (s != SBD_OK) return s;
  sbd::AttnPlan p = sbd::attn_plan(*desc);
  p.n_causal = n_causal;
  const size_t need = sbd::attn_workspace_bytes(p);
  if (need > 0) {
    if (!workspace || workspace_bytes < need)
      return fail(SBD_ERR_WORKSPACE, "workspace of %zu bytes needed, %zu given", need,
                  workspace ? workspace_bytes : (size_t)0);
    if (!aligned16(workspace)) return fail(SBD_ERR_INVALID_ARG, "workspace is not 16-byte aligned");
  }
  return sbd::attn_launch(p, q, k_cache, v_cache, cache_len, k_blk, v_blk, out, workspace, kc_app,
                          vc_app, (cudaStream_t)stream);
}

}  // namespace

extern "C" {

size_t sbd_block_attention_workspace_size(const sbd_attn_desc* desc) {
  if (check_attn_desc(desc) != SBD_OK || sbd::device_ready() != SBD_OK) return 0;
  return sbd::attn_workspace_bytes(sbd::attn_plan(*desc));
}

sbd_status sbd_block_attention(const sbd_attn_desc* desc, const void* q, const void* k_cache,
                               const void* v_cache, const int32_t* cache_len, const void* k_blk,
                               const void* v_blk, void* out, void* workspace,
                               size_t workspace_bytes, void* stream) {
  return attn_call(desc, 0, q, k_cache, v_cache, cache_len, k_blk, v_blk, out, workspace,
                   workspace_bytes, nullptr, nullptr, stream);
}

sbd_status sbd_block_attention_causal_prefix(const sbd_attn_desc* desc, int32_t n_causal,
                                             const void* q, void* k_cache, void* v_cache,
                                             const int32_t* cache_len, const void* k_blk,
                                             const void* v_blk, void* out, void* workspace,
                                             size_t workspace_bytes, void* stream) {
  if (desc && (n_causal < 0 || n_causal > desc->block_k))
    return fail(SBD_ERR_INVALID_ARG, "n_causal %d outside [0, block_k = %d]", n_causal,
                desc->block_k);
  return attn_call(desc, n_causal, q, k_cache, v_cache, cache_len, k_blk, v_blk, out, workspace,
                   workspace_bytes, n_causal > 0 ? k_cache : nullptr,
                   n_causal > 0 ? v_cache : nullptr, stream);
}

size_t sbd_head_entropy_sample_workspace_size(const sbd_head_desc* desc) {
  if (check_head_desc(desc) != SBD_OK || sbd::device_ready() != SBD_OK) return 0;
  return sbd::head_workspace_bytes(sbd::head_plan(*desc));
}

}  // extern "C"

namespace {

sbd_status head_call(const sbd_head_desc* desc, const void* hidden, const void* w,
                     const uint8_t* masked, const float* gumbel, float tau, float* entropy,
                     float* confidence, int32_t* token, void* workspace, size_t workspace_bytes,
                     void* stream, const sbd::PhiloxNoise* philox = nullptr) {
  sbd_status s = check_head_desc(desc);
  if (s != SBD_OK) return s;
  if (!(isfinite(tau) && tau >= 0.f))
    return fail(SBD_ERR_INVALID_ARG, "tau must be finite and >= 0");
  if (desc->batch == 0) return SBD_OK;
  const void* ptrs[] = {hidden, w, masked, entropy, token};
  const char* names[] = {"hidden", "w", "masked", "entropy", "token"};
  for (int i = 0; i < 5; ++i) {
    if (!ptrs[i]) return fail(SBD_ERR_INVALID_ARG, "%s is NULL", names[i]);
    if (!aligned16(ptrs[i])) return fail(SBD_ERR_INVALID_ARG, "%s is not 16-byte aligned", names[i]);
  }
  if (confidence && !aligned16(confidence))
    return fail(SBD_ERR_INVALID_ARG, "confidence is not 16-byte aligned");
  if (tau != 0.f && !gumbel && !philox)
    return fail(SBD_ERR_INVALID_ARG, "gumbel is NULL but tau != 0");
  if (gumbel && !aligned16(gumbel))
    return fail(SBD_ERR_INVALID_ARG, "gumbel is not 16-byte aligned");
  s = sbd::device_ready();
  if (s != SBD_OK) return s;
  const sbd::HeadPlan p = sbd::head_plan(*desc);
  const size_t need = sbd::head_workspace_bytes(p);
  if (!workspace || workspace_bytes < need)
    return fail(SBD_ERR_WORKSPACE, "workspace of %zu bytes needed, %zu given", need,
                workspace ? workspace_bytes : (size_t)0);
  if (!aligned16(workspace)) return fail(SBD_ERR_INVALID_ARG, "workspace is not 16-byte aligned");
  return sbd::head_launch(p, hidden, w, masked, tau == 0.f ? nullptr : gumbel, tau, entropy,
                          confidence, token, workspace, (cudaStream_t)stream, philox);
}

sbd_status select_call(int32_t rule, int32_t batch, int32_t block_k, const float* entropy,
                       const float* confidence, const int32_t* token, float threshold,
                       uint8_t* masked, int32_t* block_tokens, int32_t* n_unmasked,
                       void* stream) {
  if (rule < SBD_SELECT_EB_ENTROPY || rule > SBD_SELECT_FACTOR_COMPLEMENT)
    return fail(SBD_ERR_INVALID_ARG, "unknown selection rule %d", rule);
  if (batch < 0 || block_k < 1)
    return fail(SBD_ERR_INVALID_ARG, "bad sizes: batch=%d block_k=%d", batch, block_k);
  if (block_k > 32) return fail(SBD_ERR_UNSUPPORTED, "block_k %d > 32", block_k);
  if (!(isfinite(threshold) && threshold >= 0.f))
    return fail(SBD_ERR_INVALID_ARG, "%s must be finite and >= 0",
                rule <= SBD_SELECT_EB_CONFIDENCE ? "gamma" : "f");
  if (batch == 0) return SBD_OK;
  const void* ptrs[] = {entropy, token, masked, block_tokens};
  const char* names[] = {"entropy", "token", "masked", "block_tokens"};
  for (int i = 0; i < 4; ++i)
    if (!ptrs[i]) return fail(SBD_ERR_INVALID_ARG, "%s is NULL", names[i]);
  if (rule != SBD_SELECT_EB_ENTROPY && !confidence)
    return fail(SBD_ERR_INVALID_ARG, "confidence is NULL but rule %d orders by confidence", rule);
  const sbd_status s = sbd::device_ready();
  if (s != SBD_OK) return s;
  return sbd::select_launch(rule, batch, block_k, entropy, confidence, token, threshold, masked,
                            block_tokens, n_unmasked, (cudaStream_t)stream);
}

}  // namespace

extern "C" {

sbd_status sbd_head_entropy_sample(const sbd_head_desc* desc, const void* hidden, const void* w,
                                   const uint8_t* masked, const float* gumbel, float tau,
                                   float* entropy, int32_t* token, void* workspace,
                                   size_t workspace_bytes, void* stream) {
  return head_call(desc, hidden, w, masked, gumbel, tau, entropy, nullptr, token, workspace,
                   workspace_bytes, stream);
}

sbd_status sbd_head_entropy_confidence_sample(const sbd_head_desc* desc, const void* hidden,
                                              const void* w, const uint8_t* masked,
                                              const float* gumbel, float tau, float* entropy,
                                              float* confidence, int32_t* token,
                                              void* workspace, size_t workspace_bytes,
                                              void* stream) {
  if (!confidence) return fail(SBD_ERR_INVALID_ARG, "confidence is NULL");
  return head_call(desc, hidden, w, masked, gumbel, tau, entropy, confidence, token, workspace,
                   workspace_bytes, stream);
}

sbd_status sbd_head_entropy_sample_philox(const sbd_head_desc* desc, const void* hidden,
                                          const void* w, const uint8_t* masked, uint64_t seed,
                                          uint64_t offset, float tau, float* entropy,
                                          int32_t* token, void* workspace,
                                          size_t workspace_bytes, void* stream) {
  const sbd::PhiloxNoise noise{seed, offset};
  return head_call(desc, hidden, w, masked, nullptr, tau, entropy, nullptr, token, workspace,
                   workspace_bytes, stream, &noise);
}

}  // extern "C"

namespace {

sbd_status check_linear_desc(const sbd_linear_desc* desc) {
  if (!desc) return fail(SBD_ERR_INVALID_ARG, "desc is NULL");
  if (desc->rows < 0 || desc->in_features < 1 || desc->out_features < 1)
    return fail(SBD_ERR_INVALID_ARG, "bad sizes: rows=%d in_features=%d out_features=%d",
                desc->rows, desc->in_features, desc->out_features);
  if (desc->dtype != SBD_DTYPE_F32 && desc->dtype != SBD_DTYPE_BF16)
    return fail(SBD_ERR_INVALID_ARG, "unknown dtype %d", desc->dtype);
  if (desc->dtype != SBD_DTYPE_BF16) return fail(SBD_ERR_UNSUPPORTED, "sbd_linear is bf16 only");
  if (desc->rows > 512) return fail(SBD_ERR_UNSUPPORTED, "rows %d > 512", desc->rows);
  if (desc->in_features % 64 != 0)
    return fail(SBD_ERR_UNSUPPORTED, "in_features %d is not a multiple of 64",
                desc->in_features);
  return SBD_OK;
}

}  // namespace

extern "C" {

size_t sbd_linear_workspace_size(const sbd_linear_desc* desc) {
  if (check_linear_desc(desc) != SBD_OK) return 0;
  return sbd::linear_workspace_bytes(desc->rows, desc->in_features, desc->out_features);
}

sbd_status sbd_linear(const sbd_linear_desc* desc, const void* x, const void* w, void* y,
                      void* workspace, size_t workspace_bytes, void* stream) {
  sbd_status s = check_linear_desc(desc);
  if (s != SBD_OK) return s;
  if (desc->rows == 0) return SBD_OK;
  const void* ptrs[] = {x, w, y};
  const char* names[] = {"x", "w", "y"};
  for (int i = 0; i < 3; ++i) {
    if (!ptrs[i]) return fail(SBD_ERR_INVALID_ARG, "%s is NULL", names[i]);
    if (!aligned16(ptrs[i])) return fail(SBD_ERR_INVALID_ARG, "%s is not 16-byte aligned", names[i]);
  }
  const size_t need = sbd::linear_workspace_bytes(desc->rows, desc->in_features,
                                                  desc->out_features);
  if (need > 0 && (!workspace || workspace_bytes < need))
    return fail(SBD_ERR_WORKSPACE, "workspace of %zu bytes needed, %zu given", need,
                workspace ? workspace_bytes : (size_t)0);
  if (need > 0 && !aligned16(workspace))
    return fail(SBD_ERR_INVALID_ARG, "workspace is not 16-byte aligned");
  s = sbd::device_ready();
  if (s != SBD_OK) return s;
  return sbd::linear_launch(desc->rows, desc->in_features, desc->out_features, x, w, y,
                            workspace, (cudaStream_t)stream);
}

sbd_status sbd_gumbel_philox(int32_t n_rows, const int32_t* row_ids, int32_t vocab,
                             uint64_t seed, uint64_t offset, float* out, void* stream) {
  if (n_rows < 0 || vocab < 0)
    return fail(SBD_ERR_INVALID_ARG, "bad sizes: n_rows=%d vocab=%d", n_rows, vocab);
  if (n_rows > 65535) return fail(SBD_ERR_UNSUPPORTED, "n_rows %d > 65535", n_rows);
  if (n_rows == 0 || vocab == 0) return SBD_OK;
  if (!row_ids) return fail(SBD_ERR_INVALID_ARG, "row_ids is NULL");
  if (!out) return fail(SBD_ERR_INVALID_ARG, "out is NULL");
  const sbd_status s = sbd::device_ready();
  if (s != SBD_OK) return s;
  return sbd::gumbel_fill_launch(n_rows, row_ids, vocab, seed, offset, out, (cudaStream_t)stream);
}

sbd_status sbd_eb_select(int32_t batch, int32_t block_k, const float* entropy,
                         const int32_t* token, float gamma, uint8_t* masked,
                         int32_t* block_tokens, int32_t* n_unmasked, void* stream) {
  return select_call(SBD_SELECT_EB_ENTROPY, batch, block_k, entropy, nullptr, token, gamma,
                     masked, block_tokens, n_unmasked, stream);
}

sbd_status sbd_select(int32_t rule, int32_t batch, int32_t block_k, const float* entropy,
                      const float* confidence, const int32_t* token, float threshold,
                      uint8_t* masked, int32_t* block_tokens, int32_t* n_unmasked,
                      void* stream) {
  return select_call(rule, batch, block_k, entropy, confidence, token, threshold, masked,
                     block_tokens, n_unmasked, stream);
}

const char* sbd_status_string(sbd_status status) {
  switch (status) {
    case SBD_OK: return "SBD_OK";
    case SBD_ERR_INVALID_ARG: return "SBD_ERR_INVALID_ARG";
    case SBD_ERR_UNSUPPORTED: return "SBD_ERR_UNSUPPORTED";
    case SBD_ERR_WORKSPACE: return "SBD_ERR_WORKSPACE";
    case SBD_ERR_CUDA: return "SBD_ERR_CUDA";
  }
  return "SBD_ERR_UNKNOWN";
}

const char* sbd_last_error(void) { return g_last_error; }

sbd_status sbd_device_error(int32_t* code) {
  if (!code) return fail(SBD_ERR_INVALID_ARG, "code is NULL");
  int v = 0;
  cudaError_t e = cudaMemcpyFromSymbol(&v, g_device_error, sizeof(int));
  if (e != cudaSuccess) return sbd::cuda_fail(e, "reading the device error word");
  const int zero = 0;
  e = cudaMemcpyToSymbol(g_device_error, &zero, sizeof(int));
  if (e != cudaSuccess) return sbd::cuda_fail(e, "clearing the device error word");
  *code = v;
  return SBD_OK;
}

int32_t sbd_version(void) { return 100; }

}  // extern "C"
