// Decode attention over the per-head retained sets (arXiv 2506.05345, Sec. 3.2
// "Inference" and Sec. 4 GQA): every query head of a group attends, with plain
// softmax, to the tokens its KV head still holds in slots [0, n_h).
//
// Tiled kernel (default).  The work is the flat list of all pages of all heads of
// the layer, split into equal contiguous ranges, one per CTA (page-balanced
// split-K: ragged heads cost nothing extra and every SM streams the same number
// of bytes).  Per CTA:
//   * one producer warp walks its page range and stages each page's valid K rows,
//     V rows (and, at the first page of a head, the group's queries) into a
//     shared-memory ring of NST stages with 1-D bulk async copies (TMA engine)
//     completing on mbarriers;
//   * four consumer warps each own 16 tokens of every page: S = Q K^T and O += P V
//     on the tensor cores (mma.sync m16n8k16 bf16 -> fp32, G query heads padded to
//     16 rows), fp32 online softmax in the exp2 domain, quad shuffles for the row
//     reductions;
//   * at the end of each head segment the four warp states are merged in shared
//     memory; a head covered by one CTA is written directly, otherwise the CTA
//     writes a partial record (m, l, O) and the last CTA to arrive on the head's
//     counter merges all records (log-sum-exp combine) and writes the output.
// Arithmetic intensity is G flop per byte of K/V, far below the tensor-core ridge:
// the kernel is HBM-bound and the tensor cores only keep the issue slots free.
//
// Simple kernel (DMS_DECODE_SIMPLE): one CTA per (sequence, KV head), one warp per
// query head, scalar fp32 dot products with warp shuffles.  A cross-check path.
#include <math.h>

#include "dms_internal.cuh"

namespace dms {
namespace {

constexpr int kConsumerWarps = 4;
constexpr int kThreads = (kConsumerWarps + 1) * 32;
constexpr int kConsumerThreads = kConsumerWarps * 32;
constexpr int kQBytes = kMaxGroup * kRowBytes;                 // 4096
constexpr int kStageBytes = 2 * kHalfPageBytes + kQBytes;      // 36864
constexpr int kMergeOBytes = kConsumerWarps * kMaxGroup * kHeadDim * 4;  // 32768
constexpr int kMergeMLBytes = kConsumerWarps * kMaxGroup * 2 * 4;         // 512
constexpr int kStages = 4;

struct DecodeParams {
  const uint8_t* pool;
  const int32_t* page_table;  // this layer
  const int32_t* counts;      // this layer
  const __nv_bfloat16* q;
  __nv_bfloat16* out;
  float* pieces;
  int32_t* piece_counters;
  int32_t* ctrl;
  int32_t heads, kv_heads, group, max_pages, min_pages;
  float scale_log2;  // sm_scale * log2(e)
};

// ---------------------------------------------------------------- PTX wrappers

__device__ __forceinline__ uint32_t smem_addr(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count)
               : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)),
               "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(bar)) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t done;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(done)
      : "r"(smem_addr(bar)), "r"(parity)
      : "memory");
  return done != 0;
}

__device__ __forceinline__ unsigned long long global_timer_ns() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Wait for the phase of `bar` with the given parity to complete.  Gives up after
// kWaitLimitNs, or at once when another thread of the CTA has already given up
// (*abort != 0); then records DMS_ERR_TIMEOUT and returns false.  Callers keep
// their control flow unchanged on failure, so no barrier is ever left waiting.
__device__ __noinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, volatile int* abort,
                                       int32_t* ctrl) {
  if (mbar_try_wait(bar, parity)) return true;
  const unsigned long long t0 = global_timer_ns();
  for (uint32_t it = 1;; ++it) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((it & 31u) == 0u) {
      if (*abort) return false;
      if (global_timer_ns() - t0 > kWaitLimitNs) {
        *abort = 1;
        set_device_error(ctrl, DMS_ERR_TIMEOUT);
        return false;
      }
    }
  }
}

__device__ __forceinline__ void bulk_copy_g2s(void* dst, const void* src, uint32_t bytes,
                                              uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::
          "r"(smem_addr(dst)),
      "l"(src), "r"(bytes), "r"(smem_addr(bar))
      : "memory");
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                        uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr)
               : "memory");
}

__device__ __forceinline__ void ldsm_x4_trans(uint32_t addr, uint32_t& r0, uint32_t& r1,
                                              uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr)
               : "memory");
}

// D += A (16x16 bf16, row) * B (16x8 bf16, col), fp32 accumulators.
__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                               uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
      "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&v);
}

__device__ __forceinline__ void named_barrier_consumers() {
  asm volatile("bar.sync 1, %0;" ::"n"(kConsumerThreads) : "memory");
}

// ---------------------------------------------------------------- partition helpers

// Flat page x belongs to CTA ceil((x + 1) * P / N) - 1 when CTA k owns pages
// [floor(k N / P), floor((k + 1) N / P)).
__device__ __forceinline__ int cta_of_page(int64_t x, int64_t P, int64_t N) {
  return (int)(((x + 1) * P + N - 1) / N - 1);
}

// Last head h with pstart[h] <= x (x < pstart[heads]).
__device__ __forceinline__ int head_of_page(const int32_t* pstart, int heads, int64_t x) {
  int lo = 0, hi = heads;
  while (lo < hi) {
    const int mid = (lo + hi) >> 1;
    if (pstart[mid] > x) hi = mid; else lo = mid + 1;
  }
  return lo - 1;
}

size_t tiled_smem_bytes(int heads) {
  return (size_t)kStages * kStageBytes + kMergeOBytes + kMergeMLBytes +
         2 * kStages * sizeof(uint64_t) + 64 + (size_t)(2 * heads + 1) * sizeof(int32_t);
}

// ---------------------------------------------------------------- tiled kernel

__global__ void __launch_bounds__(kThreads, 1) decode_tiled_kernel(const DecodeParams p) {
  extern __shared__ __align__(128) uint8_t smem[];
  uint8_t* stages = smem;
  float* merge_o = reinterpret_cast<float*>(smem + kStages * kStageBytes);  // [4][16][128]
  float* merge_m = merge_o + kConsumerWarps * kMaxGroup * kHeadDim;           // [4][16]
  float* merge_l = merge_m + kConsumerWarps * kMaxGroup;                      // [4][16]
  uint64_t* full_bar = reinterpret_cast<uint64_t*>(merge_l + kConsumerWarps * kMaxGroup);
  uint64_t* empty_bar = full_bar + kStages;
  int* s_misc = reinterpret_cast<int*>(empty_bar + kStages);  // [0] abort [1] last flag [2..7] warp sums
  int32_t* s_cnt = s_misc + 16;                                // [heads]
  int32_t* s_pstart = s_cnt + p.heads;                         // [heads + 1]

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int heads = p.heads, G = p.group, Hq = p.kv_heads * p.group;
  volatile int* abort_flag = s_misc;

  // ---- prologue: per-head counts, page prefix, CTA range
  for (int h = tid; h < heads; h += kThreads) s_cnt[h] = p.counts[h];
  if (tid == 0) {
    s_misc[0] = 0;
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], kConsumerWarps);
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();
  {
    const int per = (heads + kThreads - 1) / kThreads;
    const int beg = min(tid * per, heads), end = min(beg + per, heads);
    int local = 0;
    for (int i = beg; i < end; ++i) local += (s_cnt[i] + kPageTokens - 1) / kPageTokens;
    int x = local;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, x, off);
      if (lane >= off) x += y;
    }
    if (lane == 31) s_misc[2 + warp] = x;
    __syncthreads();
    int run = x - local;
    for (int w = 0; w < warp; ++w) run += s_misc[2 + w];
    for (int i = beg; i < end; ++i) {
      s_pstart[i] = run;
      run += (s_cnt[i] + kPageTokens - 1) / kPageTokens;
    }
    if (tid == kThreads - 1) s_pstart[heads] = run;
  }
  __syncthreads();
  const int64_t N = s_pstart[heads];

  // Heads with no tokens yet produce zeros (spread over the CTAs).
  for (int h = blockIdx.x; h < heads; h += gridDim.x) {
    if (s_cnt[h] != 0) continue;
    const int b = h / p.kv_heads, hk = h - b * p.kv_heads;
    __nv_bfloat16* o = p.out + ((int64_t)b * Hq + (int64_t)hk * G) * kHeadDim;
    for (int i = tid; i < G * kHeadDim; i += kThreads) o[i] = __float2bfloat16_rn(0.f);
  }
  if (N == 0) return;
  int64_t P = N / (p.min_pages > 0 ? p.min_pages : 1);
  if (P < 1) P = 1;
  if (P > gridDim.x) P = gridDim.x;
  const int k = blockIdx.x;
  if (k >= P) return;
  const int64_t pbeg = (int64_t)k * N / P, pend = (int64_t)(k + 1) * N / P;
  const int niters = (int)(pend - pbeg);
  const int h_first = head_of_page(s_pstart, heads, pbeg);

  if (warp == kConsumerWarps) {
    // ================================================================ producer warp
    int issued = 0;
    for (int it0 = 0; it0 < niters; it0 += 32) {
      const int it = it0 + lane;
      int hh = 0, pg = 0, nv = 0, page = 0;
      if (it < niters) {
        const int64_t x = pbeg + it;
        hh = head_of_page(s_pstart, heads, x);
        pg = (int)(x - s_pstart[hh]);
        nv = min(kPageTokens, s_cnt[hh] - pg * kPageTokens);
        page = __ldg(p.page_table + (int64_t)hh * p.max_pages + pg);
      }
      const int nb = min(32, niters - it0);
      for (int i = 0; i < nb; ++i) {
        const int h_i = __shfl_sync(0xffffffffu, hh, i);
        const int pg_i = __shfl_sync(0xffffffffu, pg, i);
        const int nv_i = __shfl_sync(0xffffffffu, nv, i);
        const int page_i = __shfl_sync(0xffffffffu, page, i);
        if (lane == 0) {
          const int itg = it0 + i;
          const int s = itg % kStages;
          const int use = itg / kStages;
          if (use > 0) mbar_wait(&empty_bar[s], (use - 1) & 1, abort_flag, p.ctrl);
          const bool seg_start = (itg == 0) || (pg_i == 0);
          const uint32_t kv_bytes = (uint32_t)nv_i * kRowBytes;
          const uint32_t q_bytes = seg_start ? (uint32_t)G * kRowBytes : 0u;
          uint8_t* st = stages + s * kStageBytes;
          mbar_arrive_expect_tx(&full_bar[s], 2 * kv_bytes + q_bytes);
          const uint8_t* src = p.pool + (int64_t)page_i * kPageBytes;
          bulk_copy_g2s(st, src, kv_bytes, &full_bar[s]);
          bulk_copy_g2s(st + kHalfPageBytes, src + kHalfPageBytes, kv_bytes, &full_bar[s]);
          if (seg_start) {
            const int b = h_i / p.kv_heads, hk = h_i - b * p.kv_heads;
            const __nv_bfloat16* qsrc = p.q + ((int64_t)b * Hq + (int64_t)hk * G) * kHeadDim;
            bulk_copy_g2s(st + 2 * kHalfPageBytes, qsrc, q_bytes, &full_bar[s]);
          }
          ++issued;
        }
      }
    }
    // Drain: do not leave while a bulk copy may still be writing shared memory.
    if (lane == 0) {
      for (int s = 0; s < kStages && s < issued; ++s) {
        const int last_it = s + ((issued - 1 - s) / kStages) * kStages;
        mbar_wait(&full_bar[s], (last_it / kStages) & 1, abort_flag, p.ctrl);
      }
    }
    return;
  }

  // ================================================================ consumer warps
  const int g = lane >> 2, c4 = lane & 3;
  const int tb = warp * 16;  // this warp's first token within a page
  uint32_t qa[8][4];
  float o[16][4];
  float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
  int h = h_first;
  int pg = (int)(pbeg - s_pstart[h]);

  for (int it = 0; it < niters; ++it) {
    const int s = it % kStages;
    const int use = it / kStages;
    const int pc = s_pstart[h + 1] - s_pstart[h];
    const int nvalid = min(kPageTokens, s_cnt[h] - pg * kPageTokens);
    const bool seg_start = (it == 0) || (pg == 0);
    const bool seg_end = (it == niters - 1) || (pg == pc - 1);
    uint8_t* st = stages + s * kStageBytes;
    mbar_wait(&full_bar[s], use & 1, abort_flag, p.ctrl);

    if (seg_start) {
      const uint32_t qbase = smem_addr(st + 2 * kHalfPageBytes);
      const int mi = lane >> 3;
      const int row = (mi & 1) * 8 + (lane & 7);
#pragma unroll
      for (int kk = 0; kk < 8; ++kk) {
        const int chunk = 2 * kk + (mi >> 1);
        ldsm_x4(qbase + row * kRowBytes + chunk * 16, qa[kk][0], qa[kk][1], qa[kk][2], qa[kk][3]);
        if (g >= G) { qa[kk][0] = 0u; qa[kk][2] = 0u; }
        if (g + 8 >= G) { qa[kk][1] = 0u; qa[kk][3] = 0u; }
      }
#pragma unroll
      for (int j = 0; j < 16; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;
      m0 = m1 = -INFINITY;
      l0 = l1 = 0.f;
    }

    if (tb < nvalid) {
      // ---- S = Q K^T for tokens tb .. tb+15 (two n8 tiles)
      float sc[2][4];
#pragma unroll
      for (int nt = 0; nt < 2; ++nt) sc[nt][0] = sc[nt][1] = sc[nt][2] = sc[nt][3] = 0.f;
      const uint32_t kbase = smem_addr(st);
      {
        const int mi = lane >> 3;
        const uint32_t row = (uint32_t)(tb + (mi >> 1) * 8 + (lane & 7));
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
          uint32_t b00, b01, b10, b11;
          ldsm_x4(kbase + swizzled_offset(row, (uint32_t)(2 * kk + (mi & 1))), b00, b01, b10, b11);
          mma_bf16_16816(sc[0], qa[kk], b00, b01);
          mma_bf16_16816(sc[1], qa[kk], b10, b11);
        }
      }
      // ---- mask tokens past n_valid, online softmax (exp2 domain)
#pragma unroll
      for (int nt = 0; nt < 2; ++nt)
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int t = tb + nt * 8 + 2 * c4 + (e & 1);
          sc[nt][e] = (t < nvalid) ? sc[nt][e] * p.scale_log2 : -INFINITY;
        }
      float mx0 = fmaxf(fmaxf(sc[0][0], sc[0][1]), fmaxf(sc[1][0], sc[1][1]));
      float mx1 = fmaxf(fmaxf(sc[0][2], sc[0][3]), fmaxf(sc[1][2], sc[1][3]));
      mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
      mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
      mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
      mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
      const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);
      const float corr0 = exp2f(m0 - mn0), corr1 = exp2f(m1 - mn1);
      m0 = mn0;
      m1 = mn1;
      float pr[2][4];
#pragma unroll
      for (int nt = 0; nt < 2; ++nt) {
        pr[nt][0] = exp2f(sc[nt][0] - mn0);
        pr[nt][1] = exp2f(sc[nt][1] - mn0);
        pr[nt][2] = exp2f(sc[nt][2] - mn1);
        pr[nt][3] = exp2f(sc[nt][3] - mn1);
      }
      l0 = l0 * corr0 + (pr[0][0] + pr[0][1]) + (pr[1][0] + pr[1][1]);
      l1 = l1 * corr1 + (pr[0][2] + pr[0][3]) + (pr[1][2] + pr[1][3]);
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        o[j][0] *= corr0;
        o[j][1] *= corr0;
        o[j][2] *= corr1;
        o[j][3] *= corr1;
      }
      uint32_t pa[4];
      pa[0] = pack_bf16x2(pr[0][0], pr[0][1]);
      pa[1] = pack_bf16x2(pr[0][2], pr[0][3]);
      pa[2] = pack_bf16x2(pr[1][0], pr[1][1]);
      pa[3] = pack_bf16x2(pr[1][2], pr[1][3]);

      // ---- O += P V (16 n8 tiles over head_dim)
      const uint32_t vbase = smem_addr(st + kHalfPageBytes);
      const bool partial = tb + 16 > nvalid;
      uint32_t mk0 = 0xffffffffu, mk1 = 0xffffffffu;
      if (partial) {
        const int t = tb + 2 * c4;
        mk0 = (t < nvalid ? 0x0000ffffu : 0u) | (t + 1 < nvalid ? 0xffff0000u : 0u);
        mk1 = (t + 8 < nvalid ? 0x0000ffffu : 0u) | (t + 9 < nvalid ? 0xffff0000u : 0u);
      }
      {
        const int mi = lane >> 3;
        const uint32_t row = (uint32_t)(tb + (mi & 1) * 8 + (lane & 7));
#pragma unroll
        for (int jj = 0; jj < 8; ++jj) {
          uint32_t v0, v1, v2, v3;
          ldsm_x4_trans(vbase + swizzled_offset(row, (uint32_t)(2 * jj + (mi >> 1))), v0, v1, v2,
                        v3);
          v0 &= mk0;
          v1 &= mk1;
          v2 &= mk0;
          v3 &= mk1;
          mma_bf16_16816(o[2 * jj], pa, v0, v1);
          mma_bf16_16816(o[2 * jj + 1], pa, v2, v3);
        }
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&empty_bar[s]);

    if (seg_end) {
      // ---- merge the four warp states of this head segment
      float lt0 = l0 + __shfl_xor_sync(0xffffffffu, l0, 1);
      lt0 += __shfl_xor_sync(0xffffffffu, lt0, 2);
      float lt1 = l1 + __shfl_xor_sync(0xffffffffu, l1, 1);
      lt1 += __shfl_xor_sync(0xffffffffu, lt1, 2);
      if (c4 == 0) {
        merge_m[warp * kMaxGroup + g] = m0;
        merge_m[warp * kMaxGroup + g + 8] = m1;
        merge_l[warp * kMaxGroup + g] = lt0;
        merge_l[warp * kMaxGroup + g + 8] = lt1;
      }
      float* mo = merge_o + warp * kMaxGroup * kHeadDim;
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        *reinterpret_cast<float2*>(mo + g * kHeadDim + 8 * j + 2 * c4) = make_float2(o[j][0], o[j][1]);
        *reinterpret_cast<float2*>(mo + (g + 8) * kHeadDim + 8 * j + 2 * c4) =
            make_float2(o[j][2], o[j][3]);
      }
      named_barrier_consumers();

      const int b = h / p.kv_heads, hk = h - b * p.kv_heads;
      const int64_t first = s_pstart[h], last = s_pstart[h] + pc - 1;
      const int k_lo = cta_of_page(first, P, N), k_hi = cta_of_page(last, P, N);
      const bool single = (k_lo == k_hi);
      __nv_bfloat16* out_h = p.out + ((int64_t)b * Hq + (int64_t)hk * G) * kHeadDim;
      float* rec = p.pieces + (int64_t)(k + h) * kPieceFloats;  // m[16] l[16] o[16][128]
      const int d = tid;  // 0..127
      for (int r = 0; r < G; ++r) {
        float M = merge_m[r];
#pragma unroll
        for (int w = 1; w < kConsumerWarps; ++w) M = fmaxf(M, merge_m[w * kMaxGroup + r]);
        float L = 0.f, O = 0.f;
#pragma unroll
        for (int w = 0; w < kConsumerWarps; ++w) {
          const float wt = exp2f(merge_m[w * kMaxGroup + r] - M);
          L += wt * merge_l[w * kMaxGroup + r];
          O += wt * merge_o[(w * kMaxGroup + r) * kHeadDim + d];
        }
        if (single) {
          out_h[r * kHeadDim + d] = __float2bfloat16_rn(O / L);
        } else {
          rec[2 * kMaxGroup + r * kHeadDim + d] = O;
          if (d == 0) {
            rec[r] = M;
            rec[kMaxGroup + r] = L;
          }
        }
      }
      if (!single) {
        __threadfence();
        named_barrier_consumers();
        if (tid == 0) {
          const int prev = atomicAdd(p.piece_counters + h, 1);
          s_misc[1] = (prev == k_hi - k_lo) ? 1 : 0;
        }
        named_barrier_consumers();
        if (s_misc[1]) {
          // Last CTA of this head: log-sum-exp merge of all records, in CTA order.
          __threadfence();
          for (int r = 0; r < G; ++r) {
            float M = -INFINITY;
            for (int kk = k_lo; kk <= k_hi; ++kk)
              M = fmaxf(M, __ldcg(p.pieces + (int64_t)(kk + h) * kPieceFloats + r));
            float L = 0.f, O = 0.f;
            for (int kk = k_lo; kk <= k_hi; ++kk) {
              const float* rk = p.pieces + (int64_t)(kk + h) * kPieceFloats;
              const float wt = exp2f(__ldcg(rk + r) - M);
              L += wt * __ldcg(rk + kMaxGroup + r);
              O += wt * __ldcg(rk + 2 * kMaxGroup + r * kHeadDim + d);
            }
            out_h[r * kHeadDim + d] = __float2bfloat16_rn(O / L);
          }
          if (tid == 0) p.piece_counters[h] = 0;
        }
      }
      named_barrier_consumers();  // merge buffers are reused by the next segment
    }

    // ---- advance to the next page of the flat list
    if (++pg == pc) {
      pg = 0;
      do { ++h; } while (h < heads && s_pstart[h + 1] == s_pstart[h]);
      if (h >= heads) h = heads - 1;  // only reached after the last iteration
    }
  }
}

// ---------------------------------------------------------------- simple kernel

__global__ void __launch_bounds__(128) decode_simple_kernel(const uint8_t* pool,
                                                            const int32_t* page_table,
                                                            const int32_t* counts,
                                                            const __nv_bfloat16* q,
                                                            __nv_bfloat16* out, int32_t kv_heads,
                                                            int32_t group, int32_t max_pages,
                                                            float scale) {
  const int bh = blockIdx.x;
  const int b = bh / kv_heads, hk = bh - b * kv_heads;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n = counts[bh];
  const int32_t* pt = page_table + (int64_t)bh * max_pages;
  const int Hq = kv_heads * group;
  for (int gq = warp; gq < group; gq += blockDim.x >> 5) {
    const int64_t qrow = ((int64_t)b * Hq + (int64_t)hk * group + gq) * kHeadDim;
    float qv[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) qv[e] = __bfloat162float(q[qrow + lane * 4 + e]);
    float m = -INFINITY, l = 0.f, acc[4] = {0.f, 0.f, 0.f, 0.f};
    for (int s = 0; s < n; ++s) {
      const int32_t page = pt[s / kPageTokens];
      const uint32_t row = (uint32_t)(s & (kPageTokens - 1));
      const uint8_t* kp = pool + (int64_t)page * kPageBytes;
      // elements 4*lane .. 4*lane+3 live in logical chunk lane/2, half lane&1
      const uint32_t off = swizzled_offset(row, (uint32_t)(lane >> 1)) + (lane & 1) * 8;
      const __nv_bfloat16* kr = reinterpret_cast<const __nv_bfloat16*>(kp + off);
      const __nv_bfloat16* vr = reinterpret_cast<const __nv_bfloat16*>(kp + kHalfPageBytes + off);
      float dot = 0.f;
#pragma unroll
      for (int e = 0; e < 4; ++e) dot += qv[e] * __bfloat162float(kr[e]);
#pragma unroll
      for (int off2 = 16; off2 > 0; off2 >>= 1) dot += __shfl_xor_sync(0xffffffffu, dot, off2);
      const float sc = dot * scale;
      const float mn = fmaxf(m, sc);
      const float corr = expf(m - mn);
      const float pexp = expf(sc - mn);
      l = l * corr + pexp;
#pragma unroll
      for (int e = 0; e < 4; ++e) acc[e] = acc[e] * corr + pexp * __bfloat162float(vr[e]);
      m = mn;
    }
#pragma unroll
    for (int e = 0; e < 4; ++e)
      out[qrow + lane * 4 + e] = __float2bfloat16_rn(n > 0 ? acc[e] / l : 0.f);
  }
}

}  // namespace

cudaError_t prepare_decode(const Cache& c) {
  (void)c;
  // Sized for the largest head count any cache may have, so that caches of
  // different sizes never lower the limit under one another.
  return cudaFuncSetAttribute(decode_tiled_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)tiled_smem_bytes(kMaxHeads));
}

cudaError_t launch_decode_tiled(const Cache& c, int32_t layer, const void* q, void* out,
                                int32_t group, float scale_log2, cudaStream_t stream) {
  DecodeParams p;
  p.pool = c.pool;
  p.page_table = c.page_table + (int64_t)layer * c.heads * c.max_pages;
  p.counts = c.counts + (int64_t)layer * c.heads;
  p.q = static_cast<const __nv_bfloat16*>(q);
  p.out = static_cast<__nv_bfloat16*>(out);
  p.pieces = c.pieces;
  p.piece_counters = c.piece_counters;
  p.ctrl = c.ctrl;
  p.heads = c.heads;
  p.kv_heads = c.kv_heads;
  p.group = group;
  p.max_pages = c.max_pages;
  p.min_pages = c.min_pages_per_cta;
  p.scale_log2 = scale_log2;
  const int grid = c.num_sms * c.ctas_per_sm;
  decode_tiled_kernel<<<grid, kThreads, tiled_smem_bytes(c.heads), stream>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_decode_simple(const Cache& c, int32_t layer, const void* q, void* out,
                                 int32_t group, float scale, cudaStream_t stream) {
  decode_simple_kernel<<<c.heads, 128, 0, stream>>>(
      c.pool, c.page_table + (int64_t)layer * c.heads * c.max_pages,
      c.counts + (int64_t)layer * c.heads, static_cast<const __nv_bfloat16*>(q),
      static_cast<__nv_bfloat16*>(out), c.kv_heads, group, c.max_pages, scale);
  return cudaGetLastError();
}

}  // namespace dms

// ============================================================================
// Allocation-free decode over caller-owned pages.
//
// Some callers cannot call cudaMalloc at all: for example a plugin living inside
// a host application whose device memory is entirely owned by that application's
// own allocator (a framework caching allocator or a fixed-budget arena reserved
// at start-up), where a direct cudaMalloc would bypass the budget or fail.  Such a
// caller owns the paged KV arrays and the query/output buffers itself.  The only
// extra memory the tiled decode kernel needs is its split-K scratch (partial
// records and per-head arrival counters); here it lives in one file-scope device
// array that every GPU loading the library holds until the process exits.
// ============================================================================

#include <mutex>

namespace {

// Partial records the static scratch can hold; a launch needs (CTAs + heads).
constexpr int kStaticRecords = 1024;
constexpr int kStaticCounters = kStaticRecords;  // per-head arrival counters (int32)
constexpr int kStaticCtrl = dms::kCtrlWords;     // error word of the kernel (int32)
constexpr size_t kStaticScratchWords =
    (size_t)kStaticRecords * dms::kPieceFloats + kStaticCounters + kStaticCtrl;
constexpr int kMaxDevices = 64;

struct StaticDeviceState {
  bool ready = false;
  float* scratch = nullptr;  // device address of g_decode_scratch on this device
  int num_sms = 0;
};
std::mutex g_static_mu;
StaticDeviceState g_static_state[kMaxDevices];

}  // namespace

// 32-bit words: [records][kPieceFloats] floats, then counters, then the error word.
static __device__ __align__(256) float g_decode_scratch[kStaticScratchWords];

extern "C" dms_status dms_decode_attention_paged_noalloc(
    const void* pool, const int32_t* page_table, const int32_t* counts, int32_t batch,
    int32_t kv_heads, int32_t max_pages, const void* q, void* out, int32_t gqa_group,
    float sm_scale, void* stream) {
  using namespace dms;
  auto misaligned = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) != 0; };
  if (pool == nullptr || page_table == nullptr || counts == nullptr || q == nullptr ||
      out == nullptr || misaligned(pool) || misaligned(q) || misaligned(out) || batch < 1 ||
      kv_heads < 1 || max_pages < 1 || gqa_group < 1 || gqa_group > kMaxGroup ||
      !(sm_scale == sm_scale))
    return DMS_ERR_INVALID_ARGUMENT;
  const int64_t heads = (int64_t)batch * kv_heads;
  if (heads > kMaxHeads) return DMS_ERR_INVALID_ARGUMENT;

  // One-time set-up per device, with that device current: the device address of
  // the scratch array (the host-side name is only a stand-in), the kernel's
  // shared-memory limit and the SM count.
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return DMS_ERR_CUDA;
  StaticDeviceState st;
  {
    std::lock_guard<std::mutex> lock(g_static_mu);
    StaticDeviceState& s = g_static_state[dev];
    if (!s.ready) {
      void* ptr = nullptr;
      if (cudaGetSymbolAddress(&ptr, g_decode_scratch) != cudaSuccess) {
        cudaGetLastError();
        return DMS_ERR_CUDA;
      }
      int sms = 0;
      if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
          cudaFuncSetAttribute(decode_tiled_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               (int)tiled_smem_bytes(kMaxHeads)) != cudaSuccess) {
        cudaGetLastError();
        return DMS_ERR_CUDA;
      }
      s.scratch = static_cast<float*>(ptr);
      s.num_sms = sms;
      s.ready = true;
    }
    st = s;
  }
  const int grid = st.num_sms;
  if (grid + heads > kStaticRecords) return DMS_ERR_CAPACITY;  // scratch too small for this batch

  int32_t* counters = reinterpret_cast<int32_t*>(st.scratch + (size_t)kStaticRecords * kPieceFloats);
  int32_t* ctrl = counters + kStaticCounters;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // The array keeps whatever the previous call left: the arrival counters and the
  // error word must start at zero.
  if (cudaMemsetAsync(counters, 0, sizeof(int32_t) * (size_t)(kStaticCounters + kStaticCtrl), s) !=
      cudaSuccess)
    return DMS_ERR_CUDA;

  DecodeParams p;
  p.pool = static_cast<const uint8_t*>(pool);
  p.page_table = page_table;
  p.counts = counts;
  p.q = static_cast<const __nv_bfloat16*>(q);
  p.out = static_cast<__nv_bfloat16*>(out);
  p.pieces = st.scratch;
  p.piece_counters = counters;
  p.ctrl = ctrl;
  p.heads = (int32_t)heads;
  p.kv_heads = kv_heads;
  p.group = gqa_group;
  p.max_pages = max_pages;
  p.min_pages = 2;
  const float scale = sm_scale > 0.f ? sm_scale : 1.0f / sqrtf((float)kHeadDim);
  p.scale_log2 = scale * 1.4426950408889634f;
  decode_tiled_kernel<<<grid, kThreads, tiled_smem_bytes((int)heads), s>>>(p);
  return cudaGetLastError() == cudaSuccess ? DMS_OK : DMS_ERR_CUDA;
}
