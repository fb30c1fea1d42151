// Fused append + delayed eviction (arXiv 2506.05345, Sec. 3.1 "Delayed Eviction via
// Sliding Window" and Sec. 3.2 "Inference").
//
// State per (layer, sequence, KV head): n_h retained tokens in slots [0, n_h), a
// page list, and a ring holding (slot, alpha) of the last window+1 positions.
// Appending position j: the token j - window - 1 leaves the window now; if its
// decision was alpha = 1 it is dropped and the new token takes over its slot,
// otherwise the new token gets the fresh slot n_h (Sec. 3.2: evicted tokens are
// overwritten by incoming ones).  One token enters and at most one leaves, so the
// slots stay dense and n_h never decreases; pages are only ever added.
#include "dms_internal.cuh"

namespace dms {
namespace {

// Programmatic dependent launch (see the decode kernel): no-ops without it.
__device__ __forceinline__ void pdl_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
__device__ __forceinline__ void pdl_wait_prerequisites() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
}

struct AppendParams {
  uint8_t* pool;
  int32_t fp8;          // the cache's pages hold fp8 E4M3 rows
  int32_t* pos;
  int32_t* page_table;  // this layer: [heads][max_pages]
  const int32_t* counts_cur;  // this layer, current buffer: [heads]
  int32_t* counts_next;       // this layer, buffer after the append: [heads]
  uint32_t* ring;       // this layer: [heads][ring_len]
  int32_t* ctrl;
  int32_t* freed;       // [heads][ring_len]
  const uint16_t* k;
  const uint16_t* v;
  const uint16_t* logit;
  int64_t logit_stride;  // elements between consecutive decision logits
  int64_t t0;           // position of the first appended token
  int64_t window;
  int64_t decider;       // the eviction bit of token i is the decision of token i + decider
  int64_t pool_pages;
  int32_t n;            // tokens appended by this call
  int32_t heads, kv_heads, max_pages, ring_len;
};

// Copy one 256-byte K row and one V row into `row` of `page`, applying the chunk
// permutation of the pool layout.  Lanes 0-15 move K, lanes 16-31 move V.
__device__ __forceinline__ void store_row(uint8_t* pool, int32_t page, uint32_t row, int lane,
                                          uint4 val) {
  const uint32_t chunk = lane & 15;
  uint8_t* dst = pool + (int64_t)page * kPageBytes + (lane >= 16 ? kHalfPageBytes : 0) +
                 swizzled_offset(row, chunk);
  *reinterpret_cast<uint4*>(dst) = val;
}

// fp8 E4M3 page format: the warp's K row (lanes 0-15, elements 8 l .. 8 l + 7 of
// chunk l = lane & 15) and V row (lanes 16-31) are quantised with one scale per row,
// scale = amax / 448 (IEEE fp32 division), code = E4M3(x / scale), round to nearest
// even, saturated; a row of zeros gets scale 0 and zero codes.  K codes go to the
// K rows of the page, V codes to the slot's column of V^T (k8_offset / vt8_offset),
// the two scales to the page's scale words (page_scales_fp8).
__device__ __forceinline__ void store_row_fp8(uint8_t* pool, int32_t page, uint32_t row, int lane,
                                              uint4 val) {
  const uint32_t w[4] = {val.x, val.y, val.z, val.w};
  float x[8];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    x[2 * i] = __uint_as_float(w[i] << 16);
    x[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
  }
  float a = 0.f;
#pragma unroll
  for (int i = 0; i < 8; ++i) a = fmaxf(a, fabsf(x[i]));
#pragma unroll
  for (int off = 1; off < 16; off <<= 1) a = fmaxf(a, __shfl_xor_sync(0xffffffffu, a, off));
  const float scale = a == 0.f ? 0.f : __fdiv_rn(a, 448.f);
  uint8_t* pg = pool + (int64_t)page * kPageBytesFp8;
  const uint32_t d0 = 8u * (uint32_t)(lane & 15);
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    const float lo = scale == 0.f ? 0.f : __fdiv_rn(x[2 * e], scale);
    const float hi = scale == 0.f ? 0.f : __fdiv_rn(x[2 * e + 1], scale);
    uint16_t pair;  // code of lo in the low byte, of hi in the high byte
    asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(pair) : "f"(hi), "f"(lo));
    const uint32_t d = d0 + 2u * (uint32_t)e;
    if (lane < 16) {
      // d even: the pair (d, d + 1) is 2 consecutive bytes of the thread's word
      *reinterpret_cast<uint16_t*>(pg + k8_offset(row, d)) = pair;
    } else {
      pg[vt8_offset(row, d)] = (uint8_t)(pair & 0xffu);
      pg[vt8_offset(row, d + 1)] = (uint8_t)(pair >> 8);
    }
  }
  if ((lane & 15) == 0) page_scales_fp8(pool, page)[(lane >= 16 ? kPageTokens : 0) + row] = scale;
}

// One K and V row into `row` of `page` in the cache's format (the whole warp calls it).
__device__ __forceinline__ void store_kv_row(const AppendParams& p, int32_t page, uint32_t row,
                                             int lane, uint4 val) {
  if (p.fp8)
    store_row_fp8(p.pool, page, row, lane, val);
  else
    store_row(p.pool, page, row, lane, val);
}

__device__ __forceinline__ uint4 load_row_chunk(const uint16_t* k, const uint16_t* v,
                                                int64_t row_elem, int lane) {
  const uint16_t* src = (lane >= 16 ? v : k) + row_elem + (lane & 15) * 8;
  return __ldg(reinterpret_cast<const uint4*>(src));
}

// n = 1: one warp per head.  Lane 0 runs the ring/slot logic, the warp moves the
// 512 bytes of K and V.
__global__ void __launch_bounds__(256) append_one_kernel(const AppendParams p) {
  pdl_launch_dependents();
  pdl_wait_prerequisites();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int bh = blockIdx.x * (blockDim.x >> 5) + warp;
  if (bh >= p.heads) return;
  const int b = bh / p.kv_heads, hk = bh - b * p.kv_heads;
  const int64_t row_elem = ((int64_t)b * p.kv_heads + hk) * kHeadDim;  // [B,1,Hkv,D]
  const uint4 val = load_row_chunk(p.k, p.v, row_elem, lane);

  int32_t slot = 0, page = 0, ok = 1;
  if (lane == 0) {
    const int64_t j = p.t0;
    const int64_t R = p.window + 1, RP = ring_period(p.window);
    const uint32_t alpha = decision_from_bf16(p.logit[((int64_t)b * p.kv_heads + hk) * p.logit_stride]);
    uint32_t* ring = p.ring + (int64_t)bh * p.ring_len;
    int32_t* pt = p.page_table + (int64_t)bh * p.max_pages;
    int32_t n = p.counts_cur[bh];
    slot = -1;
    if (j >= R) {  // token j - window - 1 leaves the window now
      const uint32_t e = ring[(j - R) % RP];
      if (e & kAlphaBit) slot = (int32_t)(e & kSlotMask);  // evicted: reuse its slot
    }
    if (slot < 0) {
      slot = n;
      if ((slot & (kPageTokens - 1)) == 0) {
        const int32_t np = atomicAdd(p.ctrl + kCtrlPoolNext, 1);
        if ((int64_t)np >= p.pool_pages) {
          set_device_error(p.ctrl, DMS_ERR_CAPACITY);
          ok = 0;
        } else {
          pt[slot / kPageTokens] = np;
        }
      }
      n += ok;
    }
    p.counts_next[bh] = n;  // unchanged if the page pool ran out
    if (ok) {
      // This token's decision: its own eviction bit (delayed), or that of token
      // j - decider (immediate-eviction ablation; its entry is still in the ring).
      ring[j % RP] = (uint32_t)slot | ((p.decider == 0 ? alpha : 0u) << 31);
      if (p.decider > 0 && j >= p.decider) ring[(j - p.decider) % RP] |= alpha << 31;
      page = pt[slot / kPageTokens];
      if (page < 0) ok = 0;  // a fused step could not open this slot's page
      else p.pos[(int64_t)page * kPageTokens + (slot & (kPageTokens - 1))] = (int32_t)j;
    }
  }
  ok = __shfl_sync(0xffffffffu, ok, 0);
  if (!ok) return;
  slot = __shfl_sync(0xffffffffu, slot, 0);
  page = __shfl_sync(0xffffffffu, page, 0);
  store_kv_row(p, page, (uint32_t)(slot & (kPageTokens - 1)), lane, val);
}

constexpr int kBulkThreads = 512;
constexpr int kBulkWarps = kBulkThreads / 32;

// Block-wide exclusive scan of 0/1 flags; returns the prefix, writes the total.
__device__ __forceinline__ int block_scan_flags(int flag, int* s_warp, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const unsigned ballot = __ballot_sync(0xffffffffu, flag);
  const int in_warp = __popc(ballot & ((1u << lane) - 1u));
  if (lane == 0) s_warp[warp] = __popc(ballot);
  __syncthreads();
  int before = 0, sum = 0;
  for (int w = 0; w < kBulkWarps; ++w) {
    const int c = s_warp[w];
    before += (w < warp) ? c : 0;
    sum += c;
  }
  __syncthreads();
  *total = sum;
  return before + in_warp;
}

// n >= 1 tokens per call (prefill): one CTA per head.  Produces the same retained
// set as n single-token appends; slots freed by tokens that leave during the call
// are refilled first (in order), further kept tokens extend [0, n_h).
__global__ void __launch_bounds__(kBulkThreads) append_bulk_kernel(const AppendParams p) {
  pdl_launch_dependents();
  pdl_wait_prerequisites();
  __shared__ int s_warp[kBulkWarps];
  __shared__ int32_t s_slot[kBulkThreads];
  __shared__ int32_t s_misc[4];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int bh = blockIdx.x;
  const int b = bh / p.kv_heads, hk = bh - b * p.kv_heads;
  const int64_t R = p.window + 1, RP = ring_period(p.window), t0 = p.t0, n = p.n;
  uint32_t* ring = p.ring + (int64_t)bh * p.ring_len;
  int32_t* F = p.freed + (int64_t)bh * p.ring_len;
  int32_t* pt = p.page_table + (int64_t)bh * p.max_pages;
  const int32_t nh = p.counts_cur[bh];

  // Decision of new token li (local index), 0 past the call.
  auto alpha_new = [&](int64_t li) -> uint32_t {
    return li < n ? decision_from_bf16(p.logit[(((int64_t)b * n + li) * p.kv_heads + hk) * p.logit_stride])
                  : 0u;
  };
  const int64_t dec = p.decider;
  // 0. Immediate-eviction ablation: old tokens still in the window whose deciding
  //    token (i + decider) arrives in this call receive their eviction bit now.
  if (dec > 0) {
    const int64_t a = t0 - dec > 0 ? t0 - dec : 0;
    for (int64_t i = a + tid; i < t0; i += kBulkThreads) {
      const int64_t li = i + dec - t0;
      if (li < n) ring[i % RP] |= alpha_new(li) << 31;
    }
    __syncthreads();
  }

  // 1. Old tokens leaving the window during this call: positions [lo, hi], all < t0.
  const int64_t lo = t0 - R > 0 ? t0 - R : 0;
  const int64_t hi = (t0 - 1) < (t0 + n - R - 1) ? (t0 - 1) : (t0 + n - R - 1);
  const int64_t len_old = hi >= lo ? hi - lo + 1 : 0;
  int nf = 0;
  for (int64_t base = 0; base < len_old; base += kBulkThreads) {
    int flag = 0;
    uint32_t e = 0;
    if (base + tid < len_old) {
      e = ring[(lo + base + tid) % RP];
      flag = (e & kAlphaBit) ? 1 : 0;
    }
    int total;
    const int r = block_scan_flags(flag, s_warp, &total);
    if (flag) F[nf + r] = (int32_t)(e & kSlotMask);
    nf += total;
  }

  // 2. New tokens that also leave within this call (local index < n - R) and are
  //    flagged (their deciding token, li + decider < n - 1, is in the call) are never
  //    stored.
  const int64_t n_leave_new = n - R > 0 ? n - R : 0;
  int evicted_new = 0;
  for (int64_t base = 0; base < n_leave_new; base += kBulkThreads) {
    int flag = 0;
    if (base + tid < n_leave_new) flag = (int)alpha_new(base + tid + dec);
    int total;
    block_scan_flags(flag, s_warp, &total);
    evicted_new += total;
  }
  const int64_t kept_total = n - evicted_new;
  const int64_t new_n = nh + kept_total - nf;

  // 3. Pages for the slots [nh, new_n).
  const int32_t old_pages = (nh + kPageTokens - 1) / kPageTokens;
  const int32_t new_pages = (int32_t)((new_n + kPageTokens - 1) / kPageTokens);
  const int32_t add = new_pages - old_pages;
  if (tid == 0) {
    int32_t base = 0, ok = 1;
    if (add > 0) {
      base = atomicAdd(p.ctrl + kCtrlPoolNext, add);
      if ((int64_t)base + add > p.pool_pages) {
        set_device_error(p.ctrl, DMS_ERR_CAPACITY);
        ok = 0;
      }
    }
    s_misc[0] = base;
    s_misc[1] = ok;
  }
  __syncthreads();
  if (!s_misc[1]) {  // page pool ran out: the head keeps its state
    if (tid == 0) p.counts_next[bh] = nh;
    return;
  }
  for (int i = tid; i < add; i += kBulkThreads) pt[old_pages + i] = s_misc[0] + i;
  __syncthreads();

  // 4. Slot assignment, ring update for the final window, row copies.
  int64_t kept_before = 0;
  for (int64_t base = 0; base < n; base += kBulkThreads) {
    const int64_t li = base + tid;
    const bool valid = li < n;
    // eviction bit of token li: the decision of token li + decider if it is in the call
    const uint32_t alpha = valid ? alpha_new(li + dec) : 0u;
    const int kept = (valid && !(alpha && li < n_leave_new)) ? 1 : 0;
    int total;
    const int r = block_scan_flags(kept, s_warp, &total);
    int32_t slot = -1;
    if (kept) {
      const int64_t rank = kept_before + r;
      slot = rank < nf ? F[rank] : (int32_t)(nh + (rank - nf));
    }
    s_slot[tid] = slot;
    if (valid && li >= n - R) ring[(t0 + li) % RP] = (uint32_t)slot | (alpha << 31);
    kept_before += total;
    __syncthreads();
    // Each warp moves 4 rows at a time (loads first, then stores).
    const int64_t chunk_n = (n - base) < kBulkThreads ? (n - base) : kBulkThreads;
    for (int t = warp * 4; t < chunk_n; t += kBulkWarps * 4) {
      uint4 val[4];
      int32_t sl[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        sl[u] = (t + u < chunk_n) ? s_slot[t + u] : -1;
        if (sl[u] >= 0) {
          const int64_t row_elem = (((int64_t)b * n + base + t + u) * p.kv_heads + hk) * kHeadDim;
          val[u] = load_row_chunk(p.k, p.v, row_elem, lane);
        }
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        if (sl[u] >= 0) {
          const int32_t page = pt[sl[u] / kPageTokens];
          const uint32_t row = (uint32_t)(sl[u] & (kPageTokens - 1));
          if (page >= 0) {  // -1: a fused step could not open this slot's page
            store_kv_row(p, page, row, lane, val[u]);
            if (lane == 0) p.pos[(int64_t)page * kPageTokens + row] = (int32_t)(t0 + base + t + u);
          }
        }
      }
    }
    __syncthreads();
  }
  if (tid == 0) p.counts_next[bh] = (int32_t)new_n;
}

// Shared prompt (a prefix identical in every sequence), after the bulk append has
// filled sequence 0 of an empty layer: every other sequence b gets sequence 0's state.
// Slots below s_min = n_h - min(window + 1, n) hold tokens that have already left the
// window: they are kept for good and no later append writes them (reused slots belong to
// tokens still in the window, fresh slots start at n_h).  The pages entirely below s_min
// are therefore mapped read-only into every sequence's page table; the pages from
// s_min / 64 on are copied per sequence.  One CTA per (sequence b >= 1, KV head).
__global__ void __launch_bounds__(256) share_prefix_kernel(const AppendParams p) {
  const int h = blockIdx.x % p.kv_heads, b = 1 + blockIdx.x / p.kv_heads;
  const int src = h, dst = b * p.kv_heads + h;
  const int tid = threadIdx.x;
  __shared__ int32_t s_base, s_ok;
  const int32_t nh = p.counts_next[src];
  const int64_t R = p.window + 1;
  const int64_t smin = nh - (p.n < R ? p.n : R);
  const int32_t pages = (nh + kPageTokens - 1) / kPageTokens;
  const int32_t shared = smin > 0 ? (int32_t)(smin / kPageTokens) : 0;
  const int32_t own = pages - shared;
  if (tid == 0) {
    int32_t base = 0, ok = 1;
    if (own > 0) {
      base = atomicAdd(p.ctrl + kCtrlPoolNext, own);
      if ((int64_t)base + own > p.pool_pages) {
        set_device_error(p.ctrl, DMS_ERR_CAPACITY);
        ok = 0;
      }
    }
    s_base = base;
    s_ok = ok;
    p.counts_next[dst] = ok ? nh : 0;  // pool exhausted: the sequence stays empty
  }
  __syncthreads();
  if (!s_ok) return;
  const int32_t* pt_src = p.page_table + (int64_t)src * p.max_pages;
  int32_t* pt_dst = p.page_table + (int64_t)dst * p.max_pages;
  for (int i = tid; i < shared; i += blockDim.x) pt_dst[i] = pt_src[i];
  for (int i = tid; i < own; i += blockDim.x) pt_dst[shared + i] = s_base + i;
  for (int i = tid; i < p.ring_len; i += blockDim.x)
    p.ring[(int64_t)dst * p.ring_len + i] = p.ring[(int64_t)src * p.ring_len + i];
  // private copies of the pages that may still change (rows, scales and positions)
  const int64_t page_bytes = p.fp8 ? kPageBytesFp8 : kPageBytes;
  for (int i = 0; i < own; ++i) {
    const int32_t from = pt_src[shared + i], to = s_base + i;
    const uint4* a = reinterpret_cast<const uint4*>(p.pool + (int64_t)from * page_bytes);
    uint4* c = reinterpret_cast<uint4*>(p.pool + (int64_t)to * page_bytes);
    for (int e = tid; e < page_bytes / 16; e += blockDim.x) c[e] = a[e];
    for (int e = tid; e < kPageTokens; e += blockDim.x)
      p.pos[(int64_t)to * kPageTokens + e] = p.pos[(int64_t)from * kPageTokens + e];
  }
}

__global__ void export_positions_kernel(const int32_t* counts, const int32_t* page_table,
                                        const int32_t* pos, int32_t max_pages, int64_t capacity,
                                        int32_t* out) {
  const int bh = blockIdx.x;
  const int32_t n = counts[bh];
  const int32_t* pt = page_table + (int64_t)bh * max_pages;
  int32_t* o = out + (int64_t)bh * capacity;
  for (int64_t s = threadIdx.x; s < capacity; s += blockDim.x) {
    int32_t val = -1;
    if (s < n) {
      const int32_t page = pt[s / kPageTokens];  // -1: a page the pool could not give
      val = page < 0 ? -1 : pos[(int64_t)page * kPageTokens + (s & (kPageTokens - 1))];
    }
    o[s] = val;
  }
}

AppendParams make_params(const Cache& c, int32_t layer, const void* k, const void* v,
                         const void* logit, int64_t logit_stride, int64_t t0, int32_t n) {
  AppendParams p;
  p.pool = c.pool;
  p.fp8 = c.fp8() ? 1 : 0;
  p.pos = c.pos;
  p.page_table = c.page_table + (int64_t)layer * c.heads * c.max_pages;
  p.counts_cur = c.counts_at(layer, t0);
  p.counts_next = c.counts_at(layer, t0 + n);
  p.ring = c.rings + (int64_t)layer * c.heads * c.ring_len;
  p.ctrl = c.ctrl;
  p.freed = c.freed;
  p.k = static_cast<const uint16_t*>(k);
  p.v = static_cast<const uint16_t*>(v);
  p.logit = static_cast<const uint16_t*>(logit);
  p.logit_stride = logit_stride;
  p.t0 = t0;
  p.window = c.window;
  p.decider = c.decider();
  p.pool_pages = c.pool_pages;
  p.n = n;
  p.heads = c.heads;
  p.kv_heads = c.kv_heads;
  p.max_pages = c.max_pages;
  p.ring_len = c.ring_len;
  return p;
}

}  // namespace

cudaError_t launch_append_one(const Cache& c, int32_t layer, const void* k, const void* v,
                              const void* logit, int64_t logit_stride, int64_t t0,
                              cudaStream_t stream) {
  const AppendParams p = make_params(c, layer, k, v, logit, logit_stride, t0, 1);
  const int threads = 256, per_block = threads / 32;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.gridDim = dim3((c.heads + per_block - 1) / per_block);
  cfg.blockDim = dim3(threads);
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, append_one_kernel, p);
}

cudaError_t launch_append_bulk(const Cache& c, int32_t layer, const void* k, const void* v,
                               const void* logit, int64_t logit_stride, int64_t t0, int32_t n,
                               cudaStream_t stream) {
  const AppendParams p = make_params(c, layer, k, v, logit, logit_stride, t0, n);
  append_bulk_kernel<<<c.heads, kBulkThreads, 0, stream>>>(p);
  return cudaGetLastError();
}

// Shared prompt of n tokens into an empty layer: the bulk append of sequence 0 (its
// inputs are [1, n, kv_heads, 128]), then every other sequence shares its frozen pages.
cudaError_t launch_append_shared_prefix(const Cache& c, int32_t layer, const void* k, const void* v,
                                        const void* logit, int32_t n, cudaStream_t stream) {
  AppendParams p = make_params(c, layer, k, v, logit, 1, 0, n);
  append_bulk_kernel<<<c.kv_heads, kBulkThreads, 0, stream>>>(p);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess || c.batch == 1) return e;
  share_prefix_kernel<<<(c.batch - 1) * c.kv_heads, 256, 0, stream>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_export_positions(const Cache& c, int32_t layer, int32_t* dev_out,
                                    cudaStream_t stream) {
  export_positions_kernel<<<c.heads, 256, 0, stream>>>(
      c.counts_at(layer, c.lengths[layer]), c.page_table + (int64_t)layer * c.heads * c.max_pages,
      c.pos, c.max_pages, c.capacity, dev_out);
  return cudaGetLastError();
}

}  // namespace dms
