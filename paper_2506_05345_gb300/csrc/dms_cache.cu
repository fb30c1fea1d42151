// Host side of the C ABI declared in include/dms.h: argument checks, cache
// memory, dispatch to the append and decode kernels, statistics.
#include <math.h>
#include <stdlib.h>
#include <string.h>

#include <algorithm>
#include <new>
#include <vector>

#include "dms_internal.cuh"

struct dms_cache {
  dms::Cache c;
};

namespace {

using dms::Cache;

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

void free_device(Cache& c) {
  cudaFree(c.pool);
  cudaFree(c.pos);
  cudaFree(c.page_table);
  cudaFree(c.counts);
  cudaFree(c.rings);
  cudaFree(c.ctrl);
  cudaFree(c.freed);
  cudaFree(c.pieces);
  cudaFree(c.piece_counters);
  cudaFree(c.head_flags);
  c.head_flags = nullptr;
  c.pool = nullptr;
  c.pos = c.page_table = c.counts = c.ctrl = c.freed = c.piece_counters = nullptr;
  c.rings = nullptr;
  c.pieces = nullptr;
}

void free_host(Cache& c) {
  free(c.lengths);
  c.lengths = nullptr;
  free(c.flag_seq);
  c.flag_seq = nullptr;
  free(c.flag_valid);
  c.flag_valid = nullptr;
}

template <typename T>
cudaError_t alloc(T** p, size_t count) {
  return cudaMalloc(reinterpret_cast<void**>(p), count * sizeof(T) > 0 ? count * sizeof(T) : 16);
}

}  // namespace

extern "C" {

const char* dms_status_string(dms_status s) {
  switch (s) {
    case DMS_OK: return "ok";
    case DMS_ERR_INVALID_ARGUMENT: return "invalid argument";
    case DMS_ERR_OUT_OF_MEMORY: return "out of device memory";
    case DMS_ERR_CAPACITY: return "capacity exceeded (sequence length or page pool)";
    case DMS_ERR_CUDA: return "CUDA runtime error";
    case DMS_ERR_TIMEOUT: return "bounded device wait timed out";
    case DMS_ERR_STATE: return "invalid cache state";
  }
  return "unknown status";
}

dms_status dms_cache_create(int32_t layers, int32_t kv_heads, int32_t head_dim, int32_t window,
                            int64_t capacity, const dms_options* opt, dms_cache** out) {
  if (out == nullptr) return DMS_ERR_INVALID_ARGUMENT;
  *out = nullptr;
  if (opt == nullptr || layers < 1 || kv_heads < 1 || head_dim != dms::kHeadDim || window < 0 ||
      capacity < 1 || capacity > dms::kMaxCapacity || opt->batch < 1)
    return DMS_ERR_INVALID_ARGUMENT;
  if (opt->page_tokens != 0 && opt->page_tokens != dms::kPageTokens) return DMS_ERR_INVALID_ARGUMENT;
  if (opt->pool_tokens < 0 || opt->decode_kernel < 0 || opt->decode_kernel > DMS_DECODE_CLUSTER ||
      opt->ctas_per_sm < 0 || opt->ctas_per_sm > dms::kMaxCtasPerSm || opt->min_pages_per_cta < 0 ||
      opt->eviction_policy < DMS_EVICT_DELAYED || opt->eviction_policy > DMS_EVICT_IMMEDIATE ||
      opt->kv_format < DMS_KV_BF16 || opt->kv_format > DMS_KV_FP8_E4M3)
    return DMS_ERR_INVALID_ARGUMENT;
  if (opt->kv_format == DMS_KV_FP8_E4M3 && opt->decode_kernel == DMS_DECODE_SIMPLE)
    return DMS_ERR_INVALID_ARGUMENT;  // only the tiled kernel reads fp8 pages
  for (int i = 0; i < 3; ++i)
    if (opt->reserved[i] != 0) return DMS_ERR_INVALID_ARGUMENT;
  const int64_t heads = (int64_t)opt->batch * kv_heads;
  if (heads > dms::kMaxHeads) return DMS_ERR_INVALID_ARGUMENT;

  dms_cache* h = new (std::nothrow) dms_cache();
  if (h == nullptr) return DMS_ERR_OUT_OF_MEMORY;
  Cache& c = h->c;
  c.layers = layers;
  c.kv_heads = kv_heads;
  c.head_dim = head_dim;
  c.window = window;
  c.batch = opt->batch;
  c.capacity = capacity;
  c.heads = (int32_t)heads;
  c.ring_len = (int32_t)std::min<int64_t>(dms::ring_period(window), capacity);
  c.max_pages = (int32_t)((capacity + dms::kPageTokens - 1) / dms::kPageTokens);
  // Default: the dense worst case, every head of every layer at full capacity.
  c.pool_pages = opt->pool_tokens > 0
                     ? (opt->pool_tokens + dms::kPageTokens - 1) / dms::kPageTokens
                     : (int64_t)layers * heads * c.max_pages;
  c.decode_kernel = opt->decode_kernel;
  c.eviction_policy = opt->eviction_policy;
  c.kv_format = opt->kv_format;
  c.ctas_per_sm = opt->ctas_per_sm > 0 ? opt->ctas_per_sm : 1;
  c.min_pages_per_cta = opt->min_pages_per_cta > 0 ? opt->min_pages_per_cta : 2;
  if (c.pool_pages < 1 || c.pool_pages > 0x7fffffffLL) {
    delete h;
    return DMS_ERR_INVALID_ARGUMENT;
  }

  if (cudaGetDevice(&c.device) != cudaSuccess ||
      cudaDeviceGetAttribute(&c.num_sms, cudaDevAttrMultiProcessorCount, c.device) != cudaSuccess) {
    delete h;
    return DMS_ERR_CUDA;
  }
  c.piece_capacity = (int64_t)c.num_sms * dms::kMaxCtasPerSm + heads;
  c.lengths = static_cast<int64_t*>(calloc((size_t)layers, sizeof(int64_t)));
  c.flag_seq = static_cast<uint32_t*>(calloc((size_t)layers, sizeof(uint32_t)));
  c.flag_valid = static_cast<uint8_t*>(calloc((size_t)layers, sizeof(uint8_t)));
  if (c.lengths == nullptr || c.flag_seq == nullptr || c.flag_valid == nullptr) {
    free_host(c);
    delete h;
    return DMS_ERR_OUT_OF_MEMORY;
  }

  cudaError_t e = cudaSuccess;
  if (e == cudaSuccess) e = alloc(&c.pool, (size_t)c.pool_pages * (size_t)c.page_bytes());
  if (e == cudaSuccess) e = alloc(&c.pos, (size_t)c.pool_pages * dms::kPageTokens);
  if (e == cudaSuccess) e = alloc(&c.page_table, (size_t)layers * heads * c.max_pages);
  if (e == cudaSuccess) e = alloc(&c.counts, (size_t)layers * 2 * heads);
  if (e == cudaSuccess) e = alloc(&c.rings, (size_t)layers * heads * c.ring_len);
  if (e == cudaSuccess) e = alloc(&c.ctrl, (size_t)dms::kCtrlWords);
  if (e == cudaSuccess) e = alloc(&c.freed, (size_t)heads * c.ring_len);
  if (e == cudaSuccess) e = alloc(&c.pieces, (size_t)c.piece_capacity * dms::kPieceFloats);
  if (e == cudaSuccess) e = alloc(&c.piece_counters, (size_t)heads);
  if (e == cudaSuccess) e = alloc(&c.head_flags, (size_t)layers * heads);
  if (e == cudaSuccess) e = cudaMemset(c.head_flags, 0, sizeof(uint32_t) * (size_t)layers * heads);
  if (e == cudaSuccess) e = cudaMemset(c.counts, 0, sizeof(int32_t) * (size_t)layers * 2 * heads);
  if (e == cudaSuccess) e = cudaMemset(c.ctrl, 0, sizeof(int32_t) * dms::kCtrlWords);
  if (e == cudaSuccess) e = cudaMemset(c.piece_counters, 0, sizeof(int32_t) * (size_t)heads);
  if (e == cudaSuccess) e = dms::prepare_decode(c);
  if (e == cudaSuccess) e = dms::prepare_cluster_decode(c);
  if (e == cudaSuccess) e = cudaDeviceSynchronize();
  if (e != cudaSuccess) {
    const bool oom = (e == cudaErrorMemoryAllocation);
    cudaGetLastError();
    free_device(c);
    free_host(c);
    delete h;
    return oom ? DMS_ERR_OUT_OF_MEMORY : DMS_ERR_CUDA;
  }
  *out = h;
  return DMS_OK;
}

dms_status dms_cache_destroy(dms_cache* h) {
  if (h == nullptr) return DMS_OK;
  cudaDeviceSynchronize();
  free_device(h->c);
  free_host(h->c);
  delete h;
  return DMS_OK;
}

dms_status dms_cache_reset(dms_cache* h, void* stream) {
  if (h == nullptr) return DMS_ERR_INVALID_ARGUMENT;
  Cache& c = h->c;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  // Remember the high-water mark before the pool is handed back.
  int32_t next = 0;
  if (cudaMemcpyAsync(&next, c.ctrl + dms::kCtrlPoolNext, sizeof(int32_t), cudaMemcpyDeviceToHost,
                      st) != cudaSuccess ||
      cudaStreamSynchronize(st) != cudaSuccess)
    return DMS_ERR_CUDA;
  c.peak_pages = std::max<int64_t>(c.peak_pages, std::min<int64_t>(next, c.pool_pages));
  if (cudaMemsetAsync(c.counts, 0, sizeof(int32_t) * (size_t)c.layers * 2 * c.heads, st) !=
          cudaSuccess ||
      cudaMemsetAsync(c.ctrl, 0, sizeof(int32_t) * dms::kCtrlWords, st) != cudaSuccess ||
      cudaMemsetAsync(c.piece_counters, 0, sizeof(int32_t) * (size_t)c.heads, st) != cudaSuccess)
    return DMS_ERR_CUDA;
  for (int l = 0; l < c.layers; ++l) {
    c.lengths[l] = 0;
    c.flag_valid[l] = 0;
  }
  c.last_layer = -1;
  c.last_full_tiled = false;
  return DMS_OK;
}

}  // extern "C"

namespace {

// Shared bodies of the plain and the borrowed-decision entry points: the decision logit
// of entry i sits at logit[i * logit_stride]; zero_first makes the attention take
// element 0 of every group's first query head as 0.
dms_status append_impl(dms_cache* h, int32_t layer, const void* k, const void* v,
                       const void* logit, int64_t logit_stride, int32_t n_tokens, void* stream) {
  if (h == nullptr) return DMS_ERR_INVALID_ARGUMENT;
  Cache& c = h->c;
  if (layer < 0 || layer >= c.layers || n_tokens < 1 || k == nullptr || v == nullptr ||
      logit == nullptr || !aligned16(k) || !aligned16(v))
    return DMS_ERR_INVALID_ARGUMENT;
  if ((reinterpret_cast<uintptr_t>(logit) & 1u) != 0) return DMS_ERR_INVALID_ARGUMENT;
  const int64_t t0 = c.lengths[layer];
  if (t0 + n_tokens > c.capacity) return DMS_ERR_CAPACITY;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  c.flag_valid[layer] = 0;  // this append publishes no completion flags
  const cudaError_t e =
      (n_tokens == 1)
          ? dms::launch_append_one(c, layer, k, v, logit, logit_stride, t0, st)
          : dms::launch_append_bulk(c, layer, k, v, logit, logit_stride, t0, n_tokens, st);
  if (e != cudaSuccess) return DMS_ERR_CUDA;
  c.lengths[layer] = t0 + n_tokens;
  c.last_layer = layer;
  c.last_full_tiled = false;
  return DMS_OK;
}

dms_status decode_impl(dms_cache* h, int32_t layer, const void* q, void* out, int32_t gqa_group,
                       float sm_scale, bool zero_first, void* stream) {
  if (h == nullptr) return DMS_ERR_INVALID_ARGUMENT;
  Cache& c = h->c;
  if (layer < 0 || layer >= c.layers || q == nullptr || out == nullptr || !aligned16(q) ||
      !aligned16(out) || gqa_group < 1 || gqa_group > dms::kMaxGroup || !(sm_scale == sm_scale))
    return DMS_ERR_INVALID_ARGUMENT;
  const float scale = sm_scale > 0.f ? sm_scale : 1.0f / sqrtf((float)dms::kHeadDim);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  cudaError_t e;
  if (c.decode_kernel == DMS_DECODE_SIMPLE)
    e = dms::launch_decode_simple(c, layer, q, out, gqa_group, scale, zero_first, st);
  else
    e = dms::launch_decode_tiled(c, layer, q, out, gqa_group, scale * 1.4426950408889634f,
                                 zero_first, st);
  if (e != cudaSuccess) return DMS_ERR_CUDA;
  const bool cluster = c.decode_kernel != DMS_DECODE_SIMPLE &&
                       dms::decode_cluster_size(c, gqa_group, c.lengths[layer]) > 0;
  if (cluster && c.flag_test_layer == layer) c.flag_test_layer = -1;  // the self-test ran
  c.last_layer = layer;
  c.last_full_tiled = c.decode_kernel != DMS_DECODE_SIMPLE && dms::tiled_one_cta_per_sm(c) &&
                      !cluster;
  return DMS_OK;
}

dms_status append_decode_impl(dms_cache* h, int32_t layer, const void* k, const void* v,
                              const void* logit, int64_t logit_stride, const void* q, void* out,
                              int32_t gqa_group, float sm_scale, bool zero_first, void* stream) {
  if (h == nullptr) return DMS_ERR_INVALID_ARGUMENT;
  Cache& c = h->c;
  if (layer < 0 || layer >= c.layers || k == nullptr || v == nullptr || logit == nullptr ||
      q == nullptr || out == nullptr || !aligned16(k) || !aligned16(v) || !aligned16(q) ||
      !aligned16(out) || (reinterpret_cast<uintptr_t>(logit) & 1u) != 0 ||
      gqa_group < 1 || gqa_group > dms::kMaxGroup || !(sm_scale == sm_scale))
    return DMS_ERR_INVALID_ARGUMENT;
  const int64_t t0 = c.lengths[layer];
  if (t0 + 1 > c.capacity) return DMS_ERR_CAPACITY;
  if (!dms::append_decode_fusable(c)) {
    const dms_status st = append_impl(h, layer, k, v, logit, logit_stride, 1, stream);
    if (st != DMS_OK) return st;
    return decode_impl(h, layer, q, out, gqa_group, sm_scale, zero_first, stream);
  }
  const float scale = sm_scale > 0.f ? sm_scale : 1.0f / sqrtf((float)dms::kHeadDim);
  const bool cluster = dms::decode_cluster_size(c, gqa_group, t0 + 1) > 0;
  const cudaError_t e = dms::launch_append_decode(
      c, layer, k, v, logit, logit_stride, q, out, gqa_group, scale * 1.4426950408889634f,
      zero_first, static_cast<cudaStream_t>(stream));
  // A cluster launch publishes the next sequence number in the layer's completion flags.
  c.flag_valid[layer] = (e == cudaSuccess && cluster) ? 1 : 0;
  if (e != cudaSuccess) return DMS_ERR_CUDA;
  if (cluster) c.flag_seq[layer] = dms::next_flag_seq(c.flag_seq[layer]);
  if (cluster && c.flag_test_layer == layer) c.flag_test_layer = -1;  // the self-test ran
  c.lengths[layer] = t0 + 1;
  c.last_layer = layer;
  c.last_full_tiled = !cluster;
  return DMS_OK;
}

}  // namespace

extern "C" {

dms_status dms_append_and_evict(dms_cache* h, int32_t layer, const void* k, const void* v,
                                const void* decision_logit, int32_t n_tokens, void* stream) {
  return append_impl(h, layer, k, v, decision_logit, 1, n_tokens, stream);
}

dms_status dms_decode_attention(dms_cache* h, int32_t layer, const void* q, void* out,
                                int32_t gqa_group, float sm_scale, void* stream) {
  return decode_impl(h, layer, q, out, gqa_group, sm_scale, false, stream);
}

dms_status dms_append_and_decode(dms_cache* h, int32_t layer, const void* k, const void* v,
                                 const void* decision_logit, const void* q, void* out,
                                 int32_t gqa_group, float sm_scale, void* stream) {
  return append_decode_impl(h, layer, k, v, decision_logit, 1, q, out, gqa_group, sm_scale, false,
                            stream);
}

dms_status dms_append_shared_prefix(dms_cache* h, int32_t layer, const void* k, const void* v,
                                    const void* decision_logit, int32_t n_tokens, void* stream) {
  if (h == nullptr) return DMS_ERR_INVALID_ARGUMENT;
  Cache& c = h->c;
  if (layer < 0 || layer >= c.layers || n_tokens < 1 || k == nullptr || v == nullptr ||
      decision_logit == nullptr || !aligned16(k) || !aligned16(v) ||
      (reinterpret_cast<uintptr_t>(decision_logit) & 1u) != 0)
    return DMS_ERR_INVALID_ARGUMENT;
  if (c.lengths[layer] != 0) return DMS_ERR_STATE;  // a shared prompt starts the sequences
  if (n_tokens > c.capacity) return DMS_ERR_CAPACITY;
  c.flag_valid[layer] = 0;
  const cudaError_t e = dms::launch_append_shared_prefix(c, layer, k, v, decision_logit, n_tokens,
                                                         static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return DMS_ERR_CUDA;
  c.lengths[layer] = n_tokens;
  c.last_layer = layer;
  c.last_full_tiled = false;
  return DMS_OK;
}

// App. B: the decision logit of (sequence b, KV head h) at token t is element 0 of query
// head h * G, i.e. q + ((b * n + t) * kv_heads + h) * G * 128 for q of [B, n, kv_heads * G, 128].
dms_status dms_append_and_evict_borrowed(dms_cache* h, int32_t layer, const void* k,
                                         const void* v, const void* q, int32_t n_tokens,
                                         int32_t gqa_group, void* stream) {
  if (gqa_group < 1 || gqa_group > dms::kMaxGroup || q == nullptr || !aligned16(q))
    return DMS_ERR_INVALID_ARGUMENT;
  return append_impl(h, layer, k, v, q, (int64_t)gqa_group * dms::kHeadDim, n_tokens, stream);
}

dms_status dms_decode_attention_borrowed(dms_cache* h, int32_t layer, const void* q, void* out,
                                         int32_t gqa_group, float sm_scale, void* stream) {
  return decode_impl(h, layer, q, out, gqa_group, sm_scale, true, stream);
}

dms_status dms_append_and_decode_borrowed(dms_cache* h, int32_t layer, const void* k,
                                          const void* v, const void* q, void* out,
                                          int32_t gqa_group, float sm_scale, void* stream) {
  if (gqa_group < 1 || gqa_group > dms::kMaxGroup) return DMS_ERR_INVALID_ARGUMENT;
  return append_decode_impl(h, layer, k, v, q, (int64_t)gqa_group * dms::kHeadDim, q, out,
                            gqa_group, sm_scale, true, stream);
}

dms_status dms_cache_stats(dms_cache* h, dms_stats* out, int32_t* counts, void* stream) {
  if (h == nullptr || out == nullptr) return DMS_ERR_INVALID_ARGUMENT;
  Cache& c = h->c;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const size_t n = (size_t)c.layers * c.heads;
  std::vector<int32_t> both(2 * n), host(n);
  int32_t ctrl[dms::kCtrlWords];
  if (cudaMemcpyAsync(both.data(), c.counts, 2 * n * sizeof(int32_t), cudaMemcpyDeviceToHost, st) !=
          cudaSuccess ||
      cudaMemcpyAsync(ctrl, c.ctrl, sizeof(ctrl), cudaMemcpyDeviceToHost, st) != cudaSuccess ||
      cudaStreamSynchronize(st) != cudaSuccess)
    return DMS_ERR_CUDA;
  for (int l = 0; l < c.layers; ++l) {
    const int32_t* src = both.data() + ((size_t)l * 2 + (c.lengths[l] & 1)) * c.heads;
    memcpy(host.data() + (size_t)l * c.heads, src, sizeof(int32_t) * c.heads);
  }
  memset(out, 0, sizeof(*out));
  int64_t total = 0;
  int32_t mx = 0, mn = n ? host[0] : 0;
  for (size_t i = 0; i < n; ++i) {
    total += host[i];
    mx = std::max(mx, host[i]);
    mn = std::min(mn, host[i]);
  }
  int64_t appended = 0;
  for (int l = 0; l < c.layers; ++l) appended += c.lengths[l] * c.heads;
  out->total_retained = total;
  out->total_appended = appended;
  out->total_evicted = appended - total;
  out->pages_in_use = std::min<int64_t>(ctrl[dms::kCtrlPoolNext], c.pool_pages);
  out->pool_pages = c.pool_pages;
  c.peak_pages = std::max(c.peak_pages, out->pages_in_use);
  out->peak_pages = c.peak_pages;
  out->max_retained = mx;
  out->min_retained = mn;
  out->device_error = ctrl[dms::kCtrlError];
  if (counts != nullptr) memcpy(counts, host.data(), n * sizeof(int32_t));
  return ctrl[dms::kCtrlError] != 0 ? static_cast<dms_status>(ctrl[dms::kCtrlError]) : DMS_OK;
}

dms_status dms_cache_export_positions(dms_cache* h, int32_t layer, int32_t* host_pos,
                                      void* stream) {
  if (h == nullptr || host_pos == nullptr) return DMS_ERR_INVALID_ARGUMENT;
  Cache& c = h->c;
  if (layer < 0 || layer >= c.layers) return DMS_ERR_INVALID_ARGUMENT;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const size_t n = (size_t)c.heads * (size_t)c.capacity;
  int32_t* dev = nullptr;
  if (cudaMalloc(&dev, n * sizeof(int32_t)) != cudaSuccess) {
    cudaGetLastError();
    return DMS_ERR_OUT_OF_MEMORY;
  }
  cudaError_t e = dms::launch_export_positions(c, layer, dev, st);
  if (e == cudaSuccess) e = cudaMemcpyAsync(host_pos, dev, n * sizeof(int32_t), cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  cudaFree(dev);
  return e == cudaSuccess ? DMS_OK : DMS_ERR_CUDA;
}

dms_status dms_cache_export_kv(dms_cache* h, int32_t layer, void* host_k, void* host_v,
                               float* host_scales, void* stream) {
  if (h == nullptr || host_k == nullptr || host_v == nullptr) return DMS_ERR_INVALID_ARGUMENT;
  Cache& c = h->c;
  if (layer < 0 || layer >= c.layers || (c.fp8() && host_scales == nullptr))
    return DMS_ERR_INVALID_ARGUMENT;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const int64_t heads = c.heads, cap = c.capacity, D = dms::kHeadDim;
  std::vector<int32_t> cnt((size_t)heads), pt((size_t)heads * c.max_pages);
  if (cudaMemcpyAsync(cnt.data(), c.counts_at(layer, c.lengths[layer]), heads * sizeof(int32_t),
                      cudaMemcpyDeviceToHost, st) != cudaSuccess ||
      cudaMemcpyAsync(pt.data(), c.page_table + (int64_t)layer * heads * c.max_pages,
                      pt.size() * sizeof(int32_t), cudaMemcpyDeviceToHost, st) != cudaSuccess ||
      cudaStreamSynchronize(st) != cudaSuccess)
    return DMS_ERR_CUDA;
  const size_t esize = c.fp8() ? 1 : 2;
  memset(host_k, 0, (size_t)heads * cap * D * esize);
  memset(host_v, 0, (size_t)heads * cap * D * esize);
  if (c.fp8()) memset(host_scales, 0, (size_t)heads * cap * 2 * sizeof(float));
  std::vector<uint8_t> page((size_t)c.page_bytes());
  for (int64_t bh = 0; bh < heads; ++bh) {
    const int32_t n = cnt[(size_t)bh];
    if (n < 0 || n > cap) return DMS_ERR_STATE;
    for (int32_t pg = 0; pg * dms::kPageTokens < n; ++pg) {
      const int32_t id = pt[(size_t)bh * c.max_pages + pg];
      if (id < 0 || id >= c.pool_pages) return DMS_ERR_STATE;
      if (cudaMemcpy(page.data(), c.pool + (int64_t)id * c.page_bytes(), page.size(),
                     cudaMemcpyDeviceToHost) != cudaSuccess)
        return DMS_ERR_CUDA;
      float sc[2 * dms::kPageTokens];  // fp8: the page's key and value row scales
      if (c.fp8()) memcpy(sc, page.data() + dms::kPageCodesBytesFp8, sizeof(sc));
      for (int32_t r = 0; r < dms::kPageTokens && pg * dms::kPageTokens + r < n; ++r) {
        const int64_t slot = (int64_t)pg * dms::kPageTokens + r;
        const size_t row = ((size_t)bh * cap + slot) * D;
        if (c.fp8()) {
          uint8_t* ko = static_cast<uint8_t*>(host_k) + row;
          uint8_t* vo = static_cast<uint8_t*>(host_v) + row;
          for (uint32_t d = 0; d < (uint32_t)D; ++d) {
            ko[d] = page[dms::k8_offset((uint32_t)r, d)];
            vo[d] = page[dms::vt8_offset((uint32_t)r, d)];
          }
          host_scales[((size_t)bh * cap + slot) * 2] = sc[r];
          host_scales[((size_t)bh * cap + slot) * 2 + 1] = sc[dms::kPageTokens + r];
        } else {
          uint16_t* ko = static_cast<uint16_t*>(host_k) + row;
          uint16_t* vo = static_cast<uint16_t*>(host_v) + row;
          for (uint32_t ch = 0; ch < 16; ++ch) {
            memcpy(ko + 8 * ch, page.data() + dms::swizzled_offset((uint32_t)r, ch), 16);
            memcpy(vo + 8 * ch, page.data() + dms::kHalfPageBytes + dms::swizzled_offset((uint32_t)r, ch), 16);
          }
        }
      }
    }
  }
  return DMS_OK;
}

dms_status dms_selftest_bounded_wait(int32_t arrive, int64_t limit_ns, void* stream) {
  if (limit_ns < 1000 || limit_ns > 10000000000LL) return DMS_ERR_INVALID_ARGUMENT;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  int32_t* dev = nullptr;
  int32_t host[dms::kCtrlWords] = {0};
  if (cudaMalloc(&dev, sizeof(host)) != cudaSuccess) {
    cudaGetLastError();
    return DMS_ERR_OUT_OF_MEMORY;
  }
  cudaError_t e = cudaMemsetAsync(dev, 0, sizeof(host), st);
  if (e == cudaSuccess) e = dms::launch_bounded_wait_probe(arrive != 0, limit_ns, dev, st);
  if (e == cudaSuccess) e = cudaMemcpyAsync(host, dev, sizeof(host), cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  cudaFree(dev);
  if (e != cudaSuccess) return DMS_ERR_CUDA;
  if (host[dms::kCtrlError] != 0) return static_cast<dms_status>(host[dms::kCtrlError]);
  return host[dms::kCtrlError + 1] == 1 ? DMS_OK : DMS_ERR_STATE;
}

dms_status dms_cache_layer_length(const dms_cache* h, int32_t layer, int64_t* out) {
  if (h == nullptr || out == nullptr || layer < 0 || layer >= h->c.layers)
    return DMS_ERR_INVALID_ARGUMENT;
  *out = h->c.lengths[layer];
  return DMS_OK;
}

dms_status dms_selftest_stale_flag(dms_cache* h, int32_t layer, int64_t limit_ns) {
  if (h == nullptr || layer < 0 || layer >= h->c.layers || limit_ns < 1000 ||
      limit_ns > 10000000000LL)
    return DMS_ERR_INVALID_ARGUMENT;
  Cache& c = h->c;
  // a value above every number published so far (they only grow): no launch stores it
  c.flag_seq[layer] = dms::next_flag_seq(c.flag_seq[layer] + 1000u);
  c.flag_valid[layer] = 1;
  c.flag_test_layer = layer;
  c.flag_test_wait_ns = limit_ns;
  return DMS_OK;
}

dms_status dms_decode_plan(const dms_cache* h, int32_t layer, int32_t gqa_group, int32_t* kernel,
                           int32_t* ctas, int32_t* cluster_size) {
  if (h == nullptr || kernel == nullptr || ctas == nullptr || cluster_size == nullptr ||
      gqa_group < 1 || gqa_group > dms::kMaxGroup || layer < 0 || layer >= h->c.layers)
    return DMS_ERR_INVALID_ARGUMENT;
  const Cache& c = h->c;
  *cluster_size = 0;
  if (c.decode_kernel == DMS_DECODE_SIMPLE) {
    *kernel = DMS_DECODE_SIMPLE;
    *ctas = c.heads;
    return DMS_OK;
  }
  const int cs = dms::decode_cluster_size(c, gqa_group, c.lengths[layer] + 1);
  if (cs > 0) {
    *kernel = DMS_DECODE_CLUSTER;
    *ctas = c.heads * cs;
    *cluster_size = cs;
    return DMS_OK;
  }
  *kernel = DMS_DECODE_SPLIT;
  *ctas = c.num_sms * (!c.fp8() && c.ctas_per_sm >= 2 ? c.ctas_per_sm : 1);
  return DMS_OK;
}

}  // extern "C"
