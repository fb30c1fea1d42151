// Decode attention over the per-head retained sets (arXiv 2506.05345, Sec. 3.2
// "Inference" and Sec. 4 GQA): every query head of a group attends, with plain
// softmax, to the tokens its KV head still holds in slots [0, n_h).
//
// Tiled kernel (default).  The work is the flat list of all pages of all heads of
// the layer, split into equal contiguous ranges, one per CTA (page-balanced
// split-K: ragged heads cost nothing extra and every SM streams the same number
// of bytes).  Per CTA, three warp roles:
//   * a producer warp walks the CTA's pages and stages each page's valid K rows,
//     V rows (and, at the first page of a head, the group's queries) into a
//     shared-memory ring of kStages stages with 1-D bulk async copies (TMA engine)
//     completing on mbarriers;
//   * four consumer warps each own 16 tokens of every page.  With the tokens and
//     head_dim in the M dimension of the tensor-core tiles and the group's <= 8
//     query heads in N (16 with two n-tiles), one page costs each warp
//     S^T = K Q^T (8 mma.sync m16n8k16, two independent accumulation chains) and
//     O^T += V^T P^T (8 mma.sync); P^T is formed from S^T in registers with
//     movmatrix.  fp32 online softmax in the exp2 domain; S^T and O^T share their
//     column (head) layout, so the running rescale needs no shuffles;
//   * an epilogue warp finishes each head segment but the CTA's last while the
//     consumers move on: it merges the four warp partials from a double-buffered
//     shared-memory slot, writes the output of a head the CTA covers alone, or
//     writes a partial record (m, l, O); the last CTA to arrive on a split head's
//     counter merges all records (log-sum-exp combine) and writes the output.
//     The CTA's last segment has nothing left to overlap with, so the four
//     consumer warps finish it themselves, each merging a quarter of the query
//     heads; when every other CTA of a split last head has already counted its
//     record (read while the last page is in flight), they merge those records
//     straight away instead of publishing their own.
// A CTA takes its pages in the order: its first head's part, its last head's part
// (the two it may share with neighbours), then the heads in between, so the
// cross-CTA combines happen early and the CTA ends on directly written heads.
// Arithmetic intensity is G flop per byte of K/V, far below the tensor-core ridge:
// the kernel is HBM-bound and the tensor cores only keep the issue slots free.
//
// Simple kernel (DMS_DECODE_SIMPLE): one CTA per (sequence, KV head), one warp per
// query head, scalar fp32 dot products with warp shuffles.  A cross-check path.
#include <math.h>

#include "dms_internal.cuh"
#include "dms_ptx.cuh"

namespace dms {
namespace {

constexpr int kConsumerWarps = 4;
constexpr int kProducerWarp = 4;
constexpr int kEpilogueWarp = 5;
constexpr int kThreads = 6 * 32;
constexpr int kQBytes = kMaxGroup * kRowBytes;                 // 4096
// Staged query rows are read by ldmatrix, eight rows at a time at the same column: at a
// 256-byte row stride those eight 16-byte reads fall on the same four banks.  Groups of
// up to 8 query heads are staged one row per bulk copy at a 272-byte stride instead, which
// puts the eight rows on distinct banks (16 rows at that stride would not fit the area).
constexpr int kQRowPadded = kRowBytes + 16;
static_assert(8 * kQRowPadded <= kQBytes, "padded rows of one n-tile fit the query area");
template <int NT>
__host__ __device__ constexpr int q_row_stride() { return NT == 1 ? kQRowPadded : kRowBytes; }
constexpr int kPatchBytes = 2 * kRowBytes;                     // new K and V row (fused append)
constexpr int kStageBytesPlain = 2 * kHalfPageBytes + kQBytes;  // 36864
constexpr int kStageBytesFused = kStageBytesPlain + kPatchBytes;  // 37376
// fp8 E4M3 pages: K rows (8 KiB), V^T (8 KiB), the queries, the page's scales (and, fused,
// the new token's bf16 K and V rows).
constexpr int kStageBytesFp8 = 2 * kHalfPageBytesFp8 + kQBytes + kScaleBytes;  // 20992
__host__ __device__ constexpr int stage_bytes(bool fused, bool fp8 = false) {
  return fp8 ? kStageBytesFp8 + (fused ? kPatchBytes : 0)
             : (fused ? kStageBytesFused : kStageBytesPlain);
}
// Bytes of one staged half (K rows, or V rows / V^T) of a page.
__host__ __device__ constexpr int kv_half_bytes(bool fp8) {
  return fp8 ? kHalfPageBytesFp8 : kHalfPageBytes;
}
// Largest batch * kv_heads the fused append + decode kernel takes (its per-head
// slot table must fit next to the stages); larger caches use the two kernels.
constexpr int kMaxHeadsFused = 4000;
// Merge rows (one per query head, 128 floats of head_dim) are padded to 132
// floats: the stores of an O^T accumulator fragment then hit 32 distinct banks.
constexpr int kMergeRow = kHeadDim + 4;
// Pipeline depth per CTA: 4 stages with one CTA per SM, 2 stages with two; fp8 pages
// are half the size, so 7 stages keep about as many bytes in flight.
constexpr int kStagesOneCta = 4;
constexpr int kStagesTwoCta = 2;
constexpr int kStagesFp8 = 7;
constexpr int kStagesFp8Fused = 6;  // room for the fused variant's per-head slot table

// Shared-memory plan that depends on the number of 8-head n-tiles (NT).
template <int NT>
struct Plan {
  static constexpr int kHeadsPad = 8 * NT;
  static constexpr int kSlots = NT == 1 ? 2 : 1;  // merge slots (double-buffered if they fit)
  static constexpr int kSlotOFloats = kConsumerWarps * kHeadsPad * kMergeRow;
  static constexpr int kSlotMLFloats = kConsumerWarps * kHeadsPad * 2;
};

struct DecodeParams {
  uint8_t* pool;
  int32_t* page_table;        // this layer
  const int32_t* counts;      // this layer, current buffer
  const __nv_bfloat16* q;
  __nv_bfloat16* out;
  float* pieces;
  int32_t* piece_counters;
  int32_t* ctrl;
  int32_t heads, kv_heads, group, max_pages, min_pages;
  float scale_log2;  // sm_scale * log2(e)
  // Fused single-token append (position j) in front of the decode.
  const uint16_t* k_new;      // [batch, 1, kv_heads, 128]
  const uint16_t* v_new;
  const uint16_t* logit_new;  // decision logit of head h at logit_new[h * logit_stride]
  int64_t logit_stride;
  int32_t* counts_next;       // this layer, buffer after the append
  uint32_t* ring;             // this layer: [heads][ring_len]
  int32_t* pos;
  int64_t j, window, pool_pages;
  int64_t decider;  // the eviction bit of token i is the decision of token i + decider
  int32_t ring_len;
  // Nonzero when the launch just before on the stream was a tiled decode of another layer
  // with one CTA per SM: the state is then read, and the first pages are staged, before
  // waiting for that kernel; only the inputs (q, the new K/V rows, the logits), the
  // outputs and the shared split-K scratch wait.  Why that is safe: this launch's CTAs
  // start only after the launch before has started all its CTAs (programmatic launch).
  // Those CTAs need more than half an SM's shared memory each, one per SM, and every one
  // of them -- also one without pages -- waits for ITS predecessor before it exits.  So
  // while the launch two back runs, the launch before fills every SM and no CTA of this
  // launch can be resident: whatever last wrote this layer (two or more launches back) has
  // completed.
  int32_t state_ready;
  // Cluster kernel: this layer's per-head completion flags, the number the launch that
  // last wrote the layer's state published (0: none; wait for the dependency first) and
  // the number this launch publishes (fused; 0: none).
  uint32_t* head_flags;
  uint32_t flag_expect, flag_publish;
  int64_t flag_wait_ns;  // limit of the wait for a head's flag; 0: kWaitLimitNs
  // Nonzero: attend with element 0 of every group's first query head taken as 0 (that
  // element carries the decision logit, App. B).
  int32_t zero_first;
};

// ---------------------------------------------------------------- decode-only helpers

// Barrier of the four consumer warps only (named barrier 1; barrier 0 is the
// CTA-wide __syncthreads).
__device__ __forceinline__ void consumer_bar_sync() {
  asm volatile("bar.sync 1, %0;" ::"n"(kConsumerWarps * 32) : "memory");
}

// ---------------------------------------------------------------- partition helpers

// Balanced split of N pages over P CTAs in 32-bit arithmetic (N < 2^31): with
// N = q P + r, CTA k owns pages [k q + min(k, r), (k + 1) q + min(k + 1, r)).
struct Split {
  int q, r;
  __device__ __forceinline__ int begin(int k) const { return k * q + min(k, r); }
  // CTA owning flat page x.
  __device__ __forceinline__ int cta_of(int x) const {
    const int big = r * (q + 1);  // pages of the CTAs that hold q + 1 pages
    return x < big ? x / (q + 1) : r + (x - big) / q;
  }
};

// Page partition over P CTAs.  Launched behind another kernel, the CTAs with the
// highest indices are placed last (on the SMs that kernel frees last) and start
// streaming a few microseconds late: the last kTaperCtas CTAs share their pages at
// kTaperPermille / 1000 of the others' weight.  Small launches split evenly.
constexpr int kTaperCtas = 16;
constexpr int kTaperPermille = 900;
struct Partition {
  Split a, b;
  int P1, N1;  // CTAs [0, P1) own pages [0, N1) (split a); the rest split b
  __device__ __forceinline__ void init(int N, int P) {
    P1 = P;
    N1 = N;
    if (kTaperCtas > 0 && P > 4 * kTaperCtas && N >= 8 * P) {
      P1 = P - kTaperCtas;
      N1 = (int)((int64_t)N * P1 * 1000 / ((int64_t)P1 * 1000 + (int64_t)kTaperCtas * kTaperPermille));
    }
    a = Split{N1 / P1, N1 % P1};
    const int T = P - P1, N2 = N - N1;
    b = Split{T > 0 ? N2 / T : 0, T > 0 ? N2 % T : 0};
  }
  __device__ __forceinline__ int begin(int k) const { return k <= P1 ? a.begin(k) : N1 + b.begin(k - P1); }
  __device__ __forceinline__ int cta_of(int x) const { return x < N1 ? a.cta_of(x) : P1 + b.cta_of(x - N1); }
};

// Last head h with pstart[h] <= x (x < pstart[heads]).
__device__ __forceinline__ int head_of_page(const int32_t* pstart, int heads, int x) {
  int lo = 0, hi = heads;
  while (lo < hi) {
    const int mid = (lo + hi) >> 1;
    if (pstart[mid] > x) hi = mid; else lo = mid + 1;
  }
  return lo - 1;
}

template <int NT, bool kFused, bool kFp8 = false>
size_t tiled_smem_bytes(int heads, int stages) {
  using PL = Plan<NT>;
  return (size_t)stages * stage_bytes(kFused, kFp8) +
         (size_t)PL::kSlots * (PL::kSlotOFloats + PL::kSlotMLFloats) * 4 +
         (size_t)(2 * stages + 2 * PL::kSlots) * sizeof(uint64_t) + 64 +
         (size_t)((kFused ? 3 : 2) * heads + 1) * sizeof(int32_t);
}

// Iteration order over a CTA's pages (parts A, C, B; see the file comment) and the
// per-iteration position (head h, page pg within the head).  Every warp role walks
// it identically from shared-memory tables only.
struct PageWalk {
  const int32_t* pstart;  // [heads + 1] page prefix
  int heads;
  int pbeg, a_end, c_beg;
  int nA, nC;
  int h, pg;

  __device__ __forceinline__ int flat(int it) const {
    return it < nA ? pbeg + it : (it < nA + nC ? c_beg + (it - nA) : a_end + (it - nA - nC));
  }
  // Position for iteration `it` (call with it = 0, 1, 2, ... in order).
  __device__ __forceinline__ void enter(int it) {
    if (it == 0 || it == nA || it == nA + nC) {
      const int x = flat(it);
      h = head_of_page(pstart, heads, x);
      pg = x - pstart[h];
    }
  }
  __device__ __forceinline__ int pages_of_head() const { return pstart[h + 1] - pstart[h]; }
  __device__ __forceinline__ bool seg_start(int it) const { return it == 0 || pg == 0; }
  __device__ __forceinline__ bool seg_end(int it, int niters) const {
    return it == nA - 1 || it == nA + nC - 1 || it == niters - 1 || pg == pages_of_head() - 1;
  }
  __device__ __forceinline__ void advance() {
    if (++pg == pages_of_head()) {
      pg = 0;
      do { ++h; } while (h < heads && pstart[h + 1] == pstart[h]);
      if (h >= heads) h = heads - 1;  // only past the end of a part
    }
  }
};

template <int kStages, int NT, bool kFused, bool kFp8 = false>
__global__ void __launch_bounds__(kThreads, kStages == kStagesTwoCta ? 2 : 1)
    decode_tiled_kernel(const DecodeParams p) {
  using PL = Plan<NT>;
  constexpr int HP = PL::kHeadsPad;
  constexpr int kStageBytes = stage_bytes(kFused, kFp8);
  constexpr int kKvHalf = kv_half_bytes(kFp8);     // offset of the V half in a stage
  constexpr int kOffScales = 2 * kKvHalf;           // fp8: key scales [64], value scales [64]
  constexpr int kOffQ = kOffScales + (kFp8 ? kScaleBytes : 0);  // the group's queries
  constexpr int kOffPatch = kFp8 ? kStageBytesFp8 : kStageBytesPlain;  // fused: new K, V rows
  extern __shared__ __align__(128) uint8_t smem[];
  uint8_t* stages = smem;
  float* merge_o = reinterpret_cast<float*>(smem + kStages * kStageBytes);  // [slots][4][HP][132]
  float* merge_ml = merge_o + PL::kSlots * PL::kSlotOFloats;                  // [slots][4][HP][2]
  uint64_t* full_bar = reinterpret_cast<uint64_t*>(merge_ml + PL::kSlots * PL::kSlotMLFloats);
  uint64_t* empty_bar = full_bar + kStages;
  uint64_t* mfull_bar = empty_bar + kStages;
  uint64_t* mempty_bar = mfull_bar + PL::kSlots;
  // s_misc: [0] abort, [2..7] warp sums, [8..8+kStages) page id staged in each stage
  int* s_misc = reinterpret_cast<int*>(mempty_bar + PL::kSlots);
  int32_t* s_cnt = s_misc + 16;                                   // [heads] n_h (after the append)
  int32_t* s_pstart = s_cnt + p.heads;                            // [heads + 1]
  // fused: new token's slot | fresh << 30 per head
  uint32_t* s_slot = reinterpret_cast<uint32_t*>(s_pstart + p.heads + 1);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int heads = p.heads, G = p.group, Hq = p.kv_heads * p.group;
  volatile int* abort_flag = s_misc;

  // ---- prologue: barriers (before the dependency), per-head counts, page prefix
  pdl_launch_dependents();
  if (tid == 0) {
    s_misc[0] = 0;
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], kConsumerWarps);
    }
    for (int s = 0; s < PL::kSlots; ++s) {
      mbar_init(&mfull_bar[s], kConsumerWarps);
      mbar_init(&mempty_bar[s], 1);
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  // While the previous kernel finishes, warm L2 with the small tables the prologue
  // reads next (this CTA's slice of the layer's page table; the counts, leaving ring
  // entries and decision logits).  L2 is coherent with the previous kernel's
  // writes, so a prefetch can never make a later load stale.
  {
    // The bulk prefetch wants a 16-byte aligned start and length: it covers the
    // 16-byte aligned span inside the layer's page table (whose base need not be
    // aligned), split into per-CTA slices of whole 16-byte units.
    const uintptr_t pt_lo = (reinterpret_cast<uintptr_t>(p.page_table) + 15) & ~(uintptr_t)15;
    const uintptr_t pt_hi = (reinterpret_cast<uintptr_t>(p.page_table) +
                             (size_t)heads * p.max_pages * sizeof(int32_t)) & ~(uintptr_t)15;
    const size_t span = pt_hi > pt_lo ? (size_t)(pt_hi - pt_lo) : 0;
    const size_t slice = ((span + gridDim.x - 1) / gridDim.x + 15) & ~(size_t)15;
    const size_t beg = slice * blockIdx.x;
    if (tid == 0 && beg < span) {
      const size_t len = beg + slice <= span ? slice : span - beg;  // a multiple of 16
      asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(pt_lo + beg),
                   "r"((uint32_t)len)
                   : "memory");
    }
    for (int h = blockIdx.x * kThreads + tid; h < heads; h += gridDim.x * kThreads) {
      asm volatile("prefetch.global.L2 [%0];" ::"l"(p.counts + h));
      if constexpr (kFused) {
        const int64_t R = p.window + 1;
        if (p.j >= R)
          asm volatile("prefetch.global.L2 [%0];" ::"l"(
              p.ring + (int64_t)h * p.ring_len + (p.j - R) % ring_period(p.window)));
        asm volatile("prefetch.global.L2 [%0];" ::"l"(p.logit_new + (int64_t)h * p.logit_stride));
      }
    }
  }
  if (!p.state_ready) pdl_wait_prerequisites();
  {
    // Per-head state, with every load of a batch issued before any is used.  In the
    // fused variant: delayed eviction for position j (Sec. 3.1-3.2) -- the token
    // j - window - 1 leaves the window; if it was flagged, the new token takes its
    // slot, otherwise the fresh slot n_h.  Every CTA derives this for every head
    // from the ring; only the CTA owning a head's last page stores the new count
    // and ring entry.
    constexpr int kPer = 8;
    const int64_t R = p.window + 1, RP = ring_period(p.window);
    for (int base = 0; base < heads; base += kThreads * kPer) {
      int32_t nn[kPer];
      uint32_t ee[kPer];
#pragma unroll
      for (int i = 0; i < kPer; ++i) {
        const int h = base + tid + i * kThreads;
        if (h < heads) {  // L2 reads (the state may come from a kernel that ran on this SM)
          nn[i] = __ldcg(p.counts + h);
          if constexpr (kFused)
            ee[i] = p.j >= R ? __ldcg(p.ring + (int64_t)h * p.ring_len + (p.j - R) % RP) : 0u;
        }
      }
#pragma unroll
      for (int i = 0; i < kPer; ++i) {
        const int h = base + tid + i * kThreads;
        if (h < heads) {
          if constexpr (kFused) {
            const bool reuse = (ee[i] & kAlphaBit) != 0u;
            const uint32_t slot = reuse ? (ee[i] & kSlotMask) : (uint32_t)nn[i];
            const uint32_t fresh = reuse ? 0u : 1u;
            s_cnt[h] = nn[i] + (int32_t)fresh;
            s_slot[h] = slot | (fresh << 30);
          } else {
            s_cnt[h] = nn[i];
          }
        }
      }
    }
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
  const int N = s_pstart[heads];

  if (N == 0) {  // nothing appended yet: every output is zero
    if (p.state_ready) pdl_wait_prerequisites();
    for (int h = blockIdx.x; h < heads; h += gridDim.x) {
      const int b = h / p.kv_heads, hk = h - b * p.kv_heads;
      __nv_bfloat16* o = p.out + ((int64_t)b * Hq + (int64_t)hk * G) * kHeadDim;
      for (int i = tid; i < G * kHeadDim; i += kThreads) o[i] = __float2bfloat16_rn(0.f);
    }
    return;
  }
  int P = N / (p.min_pages > 0 ? p.min_pages : 1);
  if (P < 1) P = 1;
  if (P > (int)gridDim.x) P = (int)gridDim.x;
  const int k = blockIdx.x;
  if (k >= P) {  // no pages: still wait for the previous kernel before leaving (see state_ready)
    if (p.state_ready) pdl_wait_prerequisites();
    return;
  }
  Partition split;
  split.init(N, P);
  const int pbeg = split.begin(k), pend = split.begin(k + 1);
  const int niters = pend - pbeg;
  PageWalk walk;
  walk.pstart = s_pstart;
  walk.heads = heads;
  walk.pbeg = pbeg;
  {
    const int h_first = head_of_page(s_pstart, heads, pbeg);
    const int h_last = head_of_page(s_pstart, heads, pend - 1);
    walk.a_end = (h_first == h_last) ? pend : s_pstart[h_first + 1];
    walk.c_beg = (h_first == h_last) ? pend : s_pstart[h_last];
    walk.nA = walk.a_end - pbeg;
    walk.nC = pend - walk.c_beg;
    walk.h = h_first;
    walk.pg = 0;
  }

  if (warp == kProducerWarp) {
    // ================================================================ producer warp
    int issued = 0;
    // With ready state, the first kStages pages are staged before the dependency
    // wait; their input copies (queries, new K/V rows) and the ring entries, which
    // read inputs, are issued once the previous kernel has completed.
    bool waited = !p.state_ready;
    int d_s[kStages], d_h[kStages], d_pg[kStages], d_flags[kStages];
    int nd = 0;
    auto issue_inputs = [&](int s, int h_i, int pg_i, bool seg_start, bool patch) {
      uint8_t* st = stages + s * kStageBytes;
      if (seg_start) {
        const int b = h_i / p.kv_heads, hk = h_i - b * p.kv_heads;
        const __nv_bfloat16* qsrc = p.q + ((int64_t)b * Hq + (int64_t)hk * G) * kHeadDim;
        if constexpr (NT == 1) {
          for (int i = 0; i < G; ++i)
            bulk_copy_g2s(st + kOffQ + i * kQRowPadded, qsrc + (int64_t)i * kHeadDim, kRowBytes,
                          &full_bar[s]);
        } else {
          bulk_copy_g2s(st + kOffQ, qsrc, (uint32_t)G * kRowBytes, &full_bar[s]);
        }
      }
      if constexpr (kFused) {
        if (patch) {  // the new token's K and V rows, as given (unpermuted)
          bulk_copy_g2s(st + kOffPatch, p.k_new + (int64_t)h_i * kHeadDim, kRowBytes,
                        &full_bar[s]);
          bulk_copy_g2s(st + kOffPatch + kRowBytes, p.v_new + (int64_t)h_i * kHeadDim,
                        kRowBytes, &full_bar[s]);
        }
        if (pg_i == s_pstart[h_i + 1] - s_pstart[h_i] - 1) {  // owner of the head's last page
          const uint32_t sl = s_slot[h_i] & 0x3fffffffu;
          const uint32_t alpha = decision_from_bf16(p.logit_new[(int64_t)h_i * p.logit_stride]);
          p.counts_next[h_i] = s_cnt[h_i];
          // the new token's decision: its own eviction bit (delayed), or that of token
          // j - decider (immediate-eviction ablation; still in the ring, and not the
          // leaving token's entry that every CTA reads)
          uint32_t* rh = p.ring + (int64_t)h_i * p.ring_len;
          const int64_t RP = ring_period(p.window);
          rh[p.j % RP] = sl | ((p.decider == 0 ? alpha : 0u) << 31);
          if (p.decider > 0 && p.j >= p.decider) rh[(p.j - p.decider) % RP] |= alpha << 31;
        }
      }
    };
    auto finish_wait = [&]() {
      if (waited) return;
      pdl_wait_prerequisites();
      waited = true;
      for (int d = 0; d < nd; ++d)
        issue_inputs(d_s[d], d_h[d], d_pg[d], (d_flags[d] & 1) != 0, (d_flags[d] & 2) != 0);
      nd = 0;
    };
    for (int it0 = 0; it0 < niters; it0 += 32) {
      const int it = it0 + lane;
      int hh = 0, pg = 0, nv = 0, page = 0;
      if (it < niters) {
        const int x = walk.flat(it);
        hh = head_of_page(s_pstart, heads, x);
        pg = x - s_pstart[hh];
        nv = min(kPageTokens, s_cnt[hh] - pg * kPageTokens);
        bool new_page = false;
        if constexpr (kFused) {
          const uint32_t sl = s_slot[hh];
          const int32_t slot = (int32_t)(sl & 0x3fffffffu);
          new_page = ((sl >> 30) & 1u) && (slot % kPageTokens == 0) && (pg == slot / kPageTokens);
        }
        if (new_page) {  // fused: the new token opens a page
          page = atomicAdd(p.ctrl + kCtrlPoolNext, 1);
          if ((int64_t)page >= p.pool_pages) {  // entered as -1: nothing is written there
            set_device_error(p.ctrl, DMS_ERR_CAPACITY);
            page = -1;
          }
          p.page_table[(int64_t)hh * p.max_pages + pg] = page;
        } else {
          page = __ldcg(p.page_table + (int64_t)hh * p.max_pages + pg);
        }
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
          if (use > 0) {
            finish_wait();
            mbar_wait(&empty_bar[s], (use - 1) & 1, abort_flag, p.ctrl);
          }
          const bool seg_start = (itg == 0) || (pg_i == 0);
          const uint32_t kv_bytes = (uint32_t)nv_i * (kFp8 ? 128u : (uint32_t)kRowBytes);
          const uint32_t q_bytes = seg_start ? (uint32_t)G * kRowBytes : 0u;
          uint8_t* st = stages + s * kStageBytes;
          bool patch = false;
          if constexpr (kFused) {
            patch = (int32_t)(s_slot[h_i] & 0x3fffffffu) / kPageTokens == pg_i;
            s_misc[8 + s] = page_i;
          }
          const int64_t page0 = page_i < 0 ? 0 : page_i;
          if constexpr (kFp8) {
            // the whole page (K codes, V^T codes, row scales) in one copy: K rows past n_valid
            // are masked like stale ones, and all of V^T is needed (its rows interleave the
            // slots)
            static_assert(kKvHalf == kHalfPageBytesFp8 && kOffScales == kPageCodesBytesFp8,
                          "a stage holds the page as laid out in the pool");
            mbar_arrive_expect_tx(&full_bar[s], (uint32_t)kPageBytesFp8 + q_bytes +
                                                    (patch ? (uint32_t)kPatchBytes : 0u));
            bulk_copy_g2s(st, p.pool + page0 * kPageBytesFp8, kPageBytesFp8, &full_bar[s]);
          } else {
            mbar_arrive_expect_tx(&full_bar[s],
                                  2 * kv_bytes + q_bytes + (patch ? (uint32_t)kPatchBytes : 0u));
            const uint8_t* src = p.pool + page0 * kPageBytes;
            bulk_copy_g2s(st, src, kv_bytes, &full_bar[s]);
            bulk_copy_g2s(st + kHalfPageBytes, src + kHalfPageBytes, kv_bytes, &full_bar[s]);
          }
          if (waited) {
            issue_inputs(s, h_i, pg_i, seg_start, patch);
          } else {
            d_s[nd] = s;
            d_h[nd] = h_i;
            d_pg[nd] = pg_i;
            d_flags[nd] = (seg_start ? 1 : 0) | (patch ? 2 : 0);
            ++nd;
          }
          ++issued;
        }
      }
    }
    if (lane == 0) finish_wait();  // fewer pages than stages
    // Drain: do not leave while a bulk copy may still be writing shared memory.
    if (lane == 0) {
      for (int s = 0; s < kStages && s < issued; ++s) {
        const int last_it = s + ((issued - 1 - s) / kStages) * kStages;
        mbar_wait(&full_bar[s], (last_it / kStages) & 1, abort_flag, p.ctrl);
      }
    }
    return;
  }

  if (warp == kEpilogueWarp) {
    // ================================================================ epilogue warp
    // Everything it writes (outputs, records, counters) may be read by the previous
    // kernel until that completes.
    if (p.state_ready) pdl_wait_prerequisites();
    for (int h = k; h < heads; h += P) {  // heads with no tokens yet produce zeros
      if (s_cnt[h] != 0) continue;
      const int b = h / p.kv_heads, hk = h - b * p.kv_heads;
      __nv_bfloat16* o = p.out + ((int64_t)b * Hq + (int64_t)hk * G) * kHeadDim;
      for (int i = lane; i < G * kHeadDim; i += 32) o[i] = __float2bfloat16_rn(0.f);
    }
    int q = 0;  // segment counter
    // The CTA's last segment is finished by the consumer warps themselves.
    for (int it = 0; it < niters - 1; ++it) {
      walk.enter(it);
      if (walk.seg_end(it, niters)) {
        const int h = walk.h;
        const int slot = q % PL::kSlots;
        mbar_wait(&mfull_bar[slot], (q / PL::kSlots) & 1, abort_flag, p.ctrl);
        const float* so = merge_o + slot * PL::kSlotOFloats;
        const float* sml = merge_ml + slot * PL::kSlotMLFloats;
        const int b = h / p.kv_heads, hk = h - b * p.kv_heads;
        const int k_lo = split.cta_of(s_pstart[h]), k_hi = split.cta_of(s_pstart[h + 1] - 1);
        const bool single = (k_lo == k_hi);
        __nv_bfloat16* out_h = p.out + ((int64_t)b * Hq + (int64_t)hk * G) * kHeadDim;
        float* rec = p.pieces + (int64_t)(k + h) * kPieceFloats;  // m[16] l[16] o[16][128]
        // Row statistics in parallel (lane r < G owns row r: the four warps' maxima,
        // their weights and the merged sum), then the outputs: lane owns head_dim
        // columns 4 lane .. 4 lane + 3, four rows' shared-memory loads in flight.
        const int d4 = 4 * lane;
        float rM = -INFINITY, rL = 0.f, rw[kConsumerWarps];
        if (lane < G) {
#pragma unroll
          for (int w = 0; w < kConsumerWarps; ++w) rM = fmaxf(rM, sml[(w * HP + lane) * 2]);
#pragma unroll
          for (int w = 0; w < kConsumerWarps; ++w) {
            rw[w] = exp2f(sml[(w * HP + lane) * 2] - rM);
            rL += rw[w] * sml[(w * HP + lane) * 2 + 1];
          }
          if (!single) {
            rec[lane] = rM;
            rec[kMaxGroup + lane] = rL;
          }
        } else {
#pragma unroll
          for (int w = 0; w < kConsumerWarps; ++w) rw[w] = 0.f;
        }
        for (int r0 = 0; r0 < G; r0 += 4) {
          float4 x[4][kConsumerWarps];
#pragma unroll
          for (int rr = 0; rr < 4; ++rr)
#pragma unroll
            for (int w = 0; w < kConsumerWarps; ++w)
              x[rr][w] = (r0 + rr < G) ? *reinterpret_cast<const float4*>(
                                             so + (w * HP + r0 + rr) * kMergeRow + d4)
                                       : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
          for (int rr = 0; rr < 4; ++rr) {
            const int r = r0 + rr;
            float wt[kConsumerWarps];
#pragma unroll
            for (int w = 0; w < kConsumerWarps; ++w) wt[w] = __shfl_sync(0xffffffffu, rw[w], r & 31);
            const float L = __shfl_sync(0xffffffffu, rL, r & 31);
            if (r < G) {
              float4 O = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
              for (int w = 0; w < kConsumerWarps; ++w) {
                O.x += wt[w] * x[rr][w].x;
                O.y += wt[w] * x[rr][w].y;
                O.z += wt[w] * x[rr][w].z;
                O.w += wt[w] * x[rr][w].w;
              }
              if (single) {
                const float inv = 1.f / L;
                store_bf16x4(out_h + r * kHeadDim + d4, O.x * inv, O.y * inv, O.z * inv, O.w * inv);
              } else {
                *reinterpret_cast<float4*>(rec + 2 * kMaxGroup + r * kHeadDim + d4) = O;
              }
            }
          }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&mempty_bar[slot]);  // the slot may be refilled
        if (!single) {
          // Publish this record and count the arrival in one acquire-release atomic
          // (the warp barrier orders every lane's record stores before it).
          __syncwarp();
          int is_last = 0;
          if (lane == 0) is_last = (atomic_add_acq_rel(p.piece_counters + h, 1) == k_hi - k_lo) ? 1 : 0;
          is_last = __shfl_sync(0xffffffffu, is_last, 0);
          __syncwarp();
          if (is_last) {
            // Last CTA of this head: online log-sum-exp merge of all records in CTA
            // order, eight rows at a time; the loads of the next record are in
            // flight while the current one is merged.
            for (int r0 = 0; r0 < G; r0 += 8) {
              float Mr[8], Lr[8];
              float4 Or[8];
#pragma unroll
              for (int r = 0; r < 8; ++r) {
                Mr[r] = -INFINITY;
                Lr[r] = 0.f;
                Or[r] = make_float4(0.f, 0.f, 0.f, 0.f);
              }
              float mA[8], lA[8], mB[8], lB[8];
              float4 oA[8], oB[8];
              auto load = [&](float (&m)[8], float (&l)[8], float4 (&o)[8], int kk) {
                const float* rk = p.pieces + (int64_t)(kk + h) * kPieceFloats;
#pragma unroll
                for (int r = 0; r < 8; ++r) {
                  if (r0 + r < G) {
                    m[r] = __ldcg(rk + r0 + r);
                    l[r] = __ldcg(rk + kMaxGroup + r0 + r);
                    o[r] = __ldcg(reinterpret_cast<const float4*>(rk + 2 * kMaxGroup +
                                                                  (r0 + r) * kHeadDim + d4));
                  }
                }
              };
              auto merge = [&](const float (&m)[8], const float (&l)[8], const float4 (&o)[8]) {
#pragma unroll
                for (int r = 0; r < 8; ++r) {
                  if (r0 + r < G) {
                    const float Mn = fmaxf(Mr[r], m[r]);
                    const float a = exp2f(Mr[r] - Mn), bw = exp2f(m[r] - Mn);
                    Lr[r] = Lr[r] * a + l[r] * bw;
                    Or[r].x = Or[r].x * a + o[r].x * bw;
                    Or[r].y = Or[r].y * a + o[r].y * bw;
                    Or[r].z = Or[r].z * a + o[r].z * bw;
                    Or[r].w = Or[r].w * a + o[r].w * bw;
                    Mr[r] = Mn;
                  }
                }
              };
              load(mA, lA, oA, k_lo);
              for (int kk = k_lo; kk <= k_hi; kk += 2) {
                if (kk + 1 <= k_hi) load(mB, lB, oB, kk + 1);
                merge(mA, lA, oA);
                if (kk + 1 <= k_hi) {
                  if (kk + 2 <= k_hi) load(mA, lA, oA, kk + 2);
                  merge(mB, lB, oB);
                }
              }
#pragma unroll
              for (int r = 0; r < 8; ++r) {
                if (r0 + r < G) {
                  const float inv = 1.f / Lr[r];
                  store_bf16x4(out_h + (r0 + r) * kHeadDim + d4, Or[r].x * inv, Or[r].y * inv,
                               Or[r].z * inv, Or[r].w * inv);
                }
              }
            }
            if (lane == 0) p.piece_counters[h] = 0;
          }
        }
        ++q;
      }
      walk.advance();
    }
    return;
  }

  // ================================================================ consumer warps
  const int g = lane >> 2, c4 = lane & 3;
  const int tb = warp * 16;  // this warp's first token within a page
  const int mi = lane >> 3;  // ldmatrix: which of the four 8x8 matrices this lane addresses
  uint32_t qb[8][NT][2];     // Q^T B-fragments: (d = 16 kk + 2c.., head 8 nt + g)
  float o[8][NT][4];         // O^T accumulators: (d = 16 mt + g (+8), heads 8 nt + 2c, +1)
  float me[NT], mo[NT], le[NT], lo[NT];  // running max / sum of heads 8 nt + 2c and + 1
  int q = 0;
  // Arrivals on the last segment's head, read while its last page is in flight: if
  // every other CTA of a split head has already arrived, this CTA merges their
  // records directly, without publishing its own.
  int arrivals_seen = -1;

  for (int it = 0; it < niters; ++it) {
    walk.enter(it);
    const int s = it % kStages;
    const int use = it / kStages;
    const int nvalid = min(kPageTokens, s_cnt[walk.h] - walk.pg * kPageTokens);
    const bool seg_start = walk.seg_start(it);
    const bool seg_end = walk.seg_end(it, niters);
    uint8_t* st = stages + s * kStageBytes;
    if (it == niters - 1 && tid == 0 &&
        split.cta_of(s_pstart[walk.h]) != split.cta_of(s_pstart[walk.h + 1] - 1))
      arrivals_seen = ld_relaxed_gpu(p.piece_counters + walk.h);
    mbar_wait(&full_bar[s], use & 1, abort_flag, p.ctrl);

    if constexpr (kFused) {
      const uint32_t sl = s_slot[walk.h];
      const int32_t slot = (int32_t)(sl & 0x3fffffffu);
      const uint32_t r = (uint32_t)(slot % kPageTokens);
      if (kFp8 && slot / kPageTokens == walk.pg && (int)(r >> 4) == warp) {
        // fp8 pages: the warp whose 16 rows hold the new token quantises its K and V rows
        // (scale = amax / 448, code = E4M3(x / scale), as the append kernels do) into the
        // staged page and the pool; lane l takes head_dim 4 l .. 4 l + 3 of both rows.
        const int page = s_misc[8 + s];
        const uint2 kw = *reinterpret_cast<const uint2*>(st + kOffPatch + lane * 8);
        const uint2 vw = *reinterpret_cast<const uint2*>(st + kOffPatch + kRowBytes + lane * 8);
        const uint32_t in[2][2] = {{kw.x, kw.y}, {vw.x, vw.y}};
#pragma unroll
        for (int kv = 0; kv < 2; ++kv) {
          float x[4];
#pragma unroll
          for (int i = 0; i < 2; ++i) {
            x[2 * i] = __uint_as_float(in[kv][i] << 16);
            x[2 * i + 1] = __uint_as_float(in[kv][i] & 0xffff0000u);
          }
          float a = fmaxf(fmaxf(fabsf(x[0]), fabsf(x[1])), fmaxf(fabsf(x[2]), fabsf(x[3])));
#pragma unroll
          for (int off = 1; off < 32; off <<= 1) a = fmaxf(a, __shfl_xor_sync(0xffffffffu, a, off));
          const float scale = a == 0.f ? 0.f : __fdiv_rn(a, 448.f);
#pragma unroll
          for (int e = 0; e < 2; ++e) {
            const float lo = scale == 0.f ? 0.f : __fdiv_rn(x[2 * e], scale);
            const float hi = scale == 0.f ? 0.f : __fdiv_rn(x[2 * e + 1], scale);
            uint16_t pair;
            asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(pair) : "f"(hi), "f"(lo));
            const uint32_t d = 4u * (uint32_t)lane + 2u * (uint32_t)e;
            if (kv == 0) {
              const uint32_t off = k8_offset(r, d);
              *reinterpret_cast<uint16_t*>(st + off) = pair;
              if (page >= 0) *reinterpret_cast<uint16_t*>(p.pool + (int64_t)page * kPageBytesFp8 + off) = pair;
            } else {
              const uint32_t o0 = vt8_offset(r, d), o1 = vt8_offset(r, d + 1);
              st[o0] = (uint8_t)(pair & 0xffu);
              st[o1] = (uint8_t)(pair >> 8);
              if (page >= 0) {
                p.pool[(int64_t)page * kPageBytesFp8 + o0] = (uint8_t)(pair & 0xffu);
                p.pool[(int64_t)page * kPageBytesFp8 + o1] = (uint8_t)(pair >> 8);
              }
            }
          }
          if (lane == 0) {
            reinterpret_cast<float*>(st + kOffScales)[kv * kPageTokens + r] = scale;
            if (page >= 0)
              page_scales_fp8(p.pool, page)[kv * kPageTokens + r] = scale;
          }
        }
        if (page >= 0 && lane == 0) p.pos[(int64_t)page * kPageTokens + r] = (int32_t)p.j;
        // These generic writes precede the next bulk copy into this stage.
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        __syncwarp();
      } else if (!kFp8 && slot / kPageTokens == walk.pg && (int)(r >> 4) == warp) {
        // The warp whose 16 rows hold the new token moves its K and V row from the
        // patch buffer into the staged page (permuted layout) and into the pool.
        const int half = lane >> 4, chunk = lane & 15;
        const uint4 val =
            *reinterpret_cast<const uint4*>(st + kOffPatch + half * kRowBytes + chunk * 16);
        const uint32_t off = (uint32_t)half * kHalfPageBytes + swizzled_offset(r, (uint32_t)chunk);
        *reinterpret_cast<uint4*>(st + off) = val;
        const int page = s_misc[8 + s];
        if (page >= 0) {
          *reinterpret_cast<uint4*>(p.pool + (int64_t)page * kPageBytes + off) = val;
          if (lane == 0) p.pos[(int64_t)page * kPageTokens + r] = (int32_t)p.j;
        }
        // These generic writes precede the next bulk copy into this stage.
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        __syncwarp();
      }
    }

    if (seg_start) {
      const uint32_t qbase = smem_addr(st + kOffQ);
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) {
        const int row = 8 * nt + (lane & 7);
#pragma unroll
        for (int k2 = 0; k2 < 4; ++k2) {
          const int kk = 2 * k2 + (mi >> 1);
          uint32_t r0, r1, r2, r3;
          ldsm_x4(qbase + row * q_row_stride<NT>() + (2 * kk + (mi & 1)) * 16, r0, r1, r2, r3);
          const bool live = 8 * nt + g < G;
          qb[2 * k2][nt][0] = live ? r0 : 0u;
          qb[2 * k2][nt][1] = live ? r1 : 0u;
          qb[2 * k2 + 1][nt][0] = live ? r2 : 0u;
          qb[2 * k2 + 1][nt][1] = live ? r3 : 0u;
        }
        me[nt] = mo[nt] = -INFINITY;
        le[nt] = lo[nt] = 0.f;
#pragma unroll
        for (int mt = 0; mt < 8; ++mt) o[mt][nt][0] = o[mt][nt][1] = o[mt][nt][2] = o[mt][nt][3] = 0.f;
      }
      if constexpr (kFp8) {  // the fp8 path multiplies in f16
#pragma unroll
        for (int kk = 0; kk < 8; ++kk)
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) {
            qb[kk][nt][0] = bf16x2_to_f16x2(qb[kk][nt][0]);
            qb[kk][nt][1] = bf16x2_to_f16x2(qb[kk][nt][1]);
          }
      }
      // Lane 0 holds (d = 0, 1) of the group's first query head in the low / high half.
      if (p.zero_first && lane == 0) qb[0][0][0] &= 0xffff0000u;
    }

    if (tb < nvalid) {
      // ---- S^T = K Q^T for tokens tb .. tb+15: four independent chains over k
      float sacc[4][NT][4];
#pragma unroll
      for (int c = 0; c < 4; ++c)
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
#pragma unroll
          for (int e = 0; e < 4; ++e) sacc[c][nt][e] = 0.f;
      if constexpr (kFp8) {
        // rows tb + g and tb + g + 8; the 16-byte chunk of k-steps 4 kg .. 4 kg + 3 holds
        // this thread's codes (d = 16 kk + {2c, 2c+1, 2c+8, 2c+9}) in word kk % 4
#pragma unroll
        for (int kg = 0; kg < 2; ++kg) {
          const uint4 w0 = *reinterpret_cast<const uint4*>(
              st + (tb + g) * 128 + (((4 * kg + c4) ^ k8_swizzle(g)) << 4));
          const uint4 w1 = *reinterpret_cast<const uint4*>(
              st + (tb + g + 8) * 128 + (((4 * kg + c4) ^ k8_swizzle(g)) << 4));
          const uint32_t x0[4] = {w0.x, w0.y, w0.z, w0.w}, x1[4] = {w1.x, w1.y, w1.z, w1.w};
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            const int kk = 4 * kg + i;
            uint32_t a[4];
            a[0] = e4m3x2_to_f16x2(x0[i]);
            a[1] = e4m3x2_to_f16x2(x1[i]);
            a[2] = e4m3x2_to_f16x2(x0[i] >> 16);
            a[3] = e4m3x2_to_f16x2(x1[i] >> 16);
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) mma_f16_16816(sacc[kk & 3][nt], a, qb[kk][nt][0], qb[kk][nt][1]);
          }
        }
      } else {
        const uint32_t kbase = smem_addr(st);
        const uint32_t row = (uint32_t)(tb + (mi & 1) * 8 + (lane & 7));
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
          uint32_t a[4];
          ldsm_x4(kbase + swizzled_offset(row, (uint32_t)(2 * kk + (mi >> 1))), a[0], a[1], a[2], a[3]);
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) mma_bf16_16816(sacc[kk & 3][nt], a, qb[kk][nt][0], qb[kk][nt][1]);
        }
      }
      // ---- mask tokens past n_valid, online softmax per head (column), P^T fragments
      const bool v0 = tb + g < nvalid, v1 = tb + g + 8 < nvalid;
      // score scale of tokens tb + g and tb + g + 8 (fp8: times the keys' row scales)
      float sl0 = p.scale_log2, sl1 = p.scale_log2;
      if constexpr (kFp8) {
        const float* ksc = reinterpret_cast<const float*>(st + kOffScales);
        sl0 *= ksc[tb + g];
        sl1 *= ksc[tb + g + 8];
      }
      bool rescale = false;
      float ce[NT], co[NT];
      uint32_t pb[NT][2];
      // fp8: each value's row scale is folded into P (O^T += V^T (s P^T)), per token instead
      // of per value; stale tokens take 0 (their P is 0 and their scale word is not theirs)
      float vs0 = 1.f, vs1 = 1.f;
      if constexpr (kFp8) {
        const float* vsc = reinterpret_cast<const float*>(st + kOffScales) + kPageTokens;
        vs0 = v0 ? vsc[tb + g] : 0.f;
        vs1 = v1 ? vsc[tb + g + 8] : 0.f;
      }
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) {
        float sc[4];
#pragma unroll
        for (int e = 0; e < 4; ++e)
          sc[e] = (sacc[0][nt][e] + sacc[1][nt][e]) + (sacc[2][nt][e] + sacc[3][nt][e]);
        const float s0 = v0 ? sc[0] * sl0 : -INFINITY;
        const float s1 = v0 ? sc[1] * sl0 : -INFINITY;
        const float s2 = v1 ? sc[2] * sl1 : -INFINITY;
        const float s3 = v1 ? sc[3] * sl1 : -INFINITY;
        float xe = fmaxf(s0, s2), xo = fmaxf(s1, s3);
#pragma unroll
        for (int off = 4; off < 32; off <<= 1) {
          xe = fmaxf(xe, __shfl_xor_sync(0xffffffffu, xe, off));
          xo = fmaxf(xo, __shfl_xor_sync(0xffffffffu, xo, off));
        }
        const float ne = fmaxf(me[nt], xe), no = fmaxf(mo[nt], xo);
        ce[nt] = ex2_approx(me[nt] - ne);  // 0 while the running max is -inf
        co[nt] = ex2_approx(mo[nt] - no);
        me[nt] = ne;
        mo[nt] = no;
        const float p0 = ex2_approx(s0 - ne), p1 = ex2_approx(s1 - no);
        const float p2 = ex2_approx(s2 - ne), p3 = ex2_approx(s3 - no);
        le[nt] = le[nt] * ce[nt] + (p0 + p2);
        lo[nt] = lo[nt] * co[nt] + (p1 + p3);
        rescale |= (ce[nt] != 1.f) || (co[nt] != 1.f);
        // (token g, heads 2c..) -> transpose -> (head g, tokens 2c..): the B operand
        if constexpr (kFp8) {
          pb[nt][0] = movmatrix_trans(pack_f16x2(p0 * vs0, p1 * vs0));
          pb[nt][1] = movmatrix_trans(pack_f16x2(p2 * vs1, p3 * vs1));
        } else {
          pb[nt][0] = movmatrix_trans(pack_bf16x2(p0, p1));
          pb[nt][1] = movmatrix_trans(pack_bf16x2(p2, p3));
        }
      }
      if (__any_sync(0xffffffffu, rescale)) {
#pragma unroll
        for (int mt = 0; mt < 8; ++mt)
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) {
            o[mt][nt][0] *= ce[nt];
            o[mt][nt][1] *= co[nt];
            o[mt][nt][2] *= ce[nt];
            o[mt][nt][3] *= co[nt];
          }
      }
      // ---- O^T += V^T P^T over head_dim (8 m-tiles of 16)
      uint32_t mk_lo = 0xffffffffu, mk_hi = 0xffffffffu;
      if (tb + 16 > nvalid) {  // stale rows past n_valid must not reach the tensor cores
        const int t = tb + 2 * c4;
        mk_lo = (t < nvalid ? 0x0000ffffu : 0u) | (t + 1 < nvalid ? 0xffff0000u : 0u);
        mk_hi = (t + 8 < nvalid ? 0x0000ffffu : 0u) | (t + 9 < nvalid ? 0xffff0000u : 0u);
      }
      if constexpr (kFp8) {
        // V^T rows d = 16 mt + g and + 8: one word holds the codes of tokens tb + {2c, 2c+1,
        // 2c+8, 2c+9} (the row scales are in P); stale tokens masked
        const int blk = tb >> 4;
#pragma unroll
        for (int mt = 0; mt < 8; ++mt) {
          const int d0 = 16 * mt + g, d1 = d0 + 8;
          const uint32_t w0 = *reinterpret_cast<const uint32_t*>(
              st + kKvHalf + d0 * 64 + ((blk ^ ((d0 >> 1) & 3)) << 4) + 4 * c4);
          const uint32_t w1 = *reinterpret_cast<const uint32_t*>(
              st + kKvHalf + d1 * 64 + ((blk ^ ((d1 >> 1) & 3)) << 4) + 4 * c4);
          uint32_t a[4];
          a[0] = e4m3x2_to_f16x2(w0) & mk_lo;
          a[1] = e4m3x2_to_f16x2(w1) & mk_lo;
          a[2] = e4m3x2_to_f16x2(w0 >> 16) & mk_hi;
          a[3] = e4m3x2_to_f16x2(w1 >> 16) & mk_hi;
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) mma_f16_16816(o[mt][nt], a, pb[nt][0], pb[nt][1]);
        }
      } else {
        const uint32_t vbase = smem_addr(st + kHalfPageBytes);
        const uint32_t row = (uint32_t)(tb + (mi >> 1) * 8 + (lane & 7));
#pragma unroll
        for (int mt = 0; mt < 8; ++mt) {
          uint32_t a[4];
          ldsm_x4_trans(vbase + swizzled_offset(row, (uint32_t)(2 * mt + (mi & 1))), a[0], a[1], a[2],
                        a[3]);
          a[0] &= mk_lo;
          a[1] &= mk_lo;
          a[2] &= mk_hi;
          a[3] &= mk_hi;
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) mma_bf16_16816(o[mt][nt], a, pb[nt][0], pb[nt][1]);
        }
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&empty_bar[s]);

    if (seg_end) {
      // ---- hand this warp's partial (m, l, O^T) of the segment to the epilogue warp
      const int slot = q % PL::kSlots;
      if (q >= PL::kSlots) mbar_wait(&mempty_bar[slot], ((q / PL::kSlots) - 1) & 1, abort_flag, p.ctrl);
      float* so = merge_o + slot * PL::kSlotOFloats + warp * HP * kMergeRow;
      float* sml = merge_ml + slot * PL::kSlotMLFloats + warp * HP * 2;
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) {
        float te = le[nt], to = lo[nt];
#pragma unroll
        for (int off = 4; off < 32; off <<= 1) {
          te += __shfl_xor_sync(0xffffffffu, te, off);
          to += __shfl_xor_sync(0xffffffffu, to, off);
        }
        const int he = 8 * nt + 2 * c4, ho = he + 1;
        if (g == 0) {
          sml[he * 2] = me[nt];
          sml[he * 2 + 1] = te;
          sml[ho * 2] = mo[nt];
          sml[ho * 2 + 1] = to;
        }
#pragma unroll
        for (int mt = 0; mt < 8; ++mt) {
          so[he * kMergeRow + 16 * mt + g] = o[mt][nt][0];
          so[ho * kMergeRow + 16 * mt + g] = o[mt][nt][1];
          so[he * kMergeRow + 16 * mt + g + 8] = o[mt][nt][2];
          so[ho * kMergeRow + 16 * mt + g + 8] = o[mt][nt][3];
        }
      }
      if (it != niters - 1) {
        __syncwarp();
        if (lane == 0) mbar_arrive(&mfull_bar[slot]);
        ++q;
      } else {
        // ---- the CTA's last segment: nothing is left to stream, so the four warps
        // finish it together: warp w merges query-head rows w, w + 4, ..., lane l
        // head_dim columns 4 l .. 4 l + 3.
        const int h = walk.h;
        const int b = h / p.kv_heads, hk = h - b * p.kv_heads;
        const int k_lo = split.cta_of(s_pstart[h]), k_hi = split.cta_of(s_pstart[h + 1] - 1);
        const bool single = (k_lo == k_hi);
        if (tid == 0) {
          int early = 0;
          if (!single && arrivals_seen == k_hi - k_lo) {
            asm volatile("fence.acq_rel.gpu;" ::: "memory");  // acquire the others' records
            early = 1;
          }
          s_misc[1] = early;
        }
        consumer_bar_sync();
        const bool early_last = s_misc[1] != 0;
        constexpr int RPW = HP / kConsumerWarps;  // rows per warp
        const int d4 = 4 * lane;
        __nv_bfloat16* out_h = p.out + ((int64_t)b * Hq + (int64_t)hk * G) * kHeadDim;
        const float* mo_all = merge_o + slot * PL::kSlotOFloats;
        const float* ml_all = merge_ml + slot * PL::kSlotMLFloats;
        float Mo[RPW], Lo[RPW];
        float4 Oo[RPW];
#pragma unroll
        for (int i = 0; i < RPW; ++i) {
          const int r = warp + kConsumerWarps * i;
          Mo[i] = -INFINITY;
          Lo[i] = 0.f;
          Oo[i] = make_float4(0.f, 0.f, 0.f, 0.f);
          if (r < G) {
            float mw[kConsumerWarps];
#pragma unroll
            for (int w = 0; w < kConsumerWarps; ++w) {
              mw[w] = ml_all[(w * HP + r) * 2];
              Mo[i] = fmaxf(Mo[i], mw[w]);
            }
#pragma unroll
            for (int w = 0; w < kConsumerWarps; ++w) {
              const float a = exp2f(mw[w] - Mo[i]);
              const float4 x = *reinterpret_cast<const float4*>(mo_all + (w * HP + r) * kMergeRow + d4);
              Lo[i] += a * ml_all[(w * HP + r) * 2 + 1];
              Oo[i].x += a * x.x;
              Oo[i].y += a * x.y;
              Oo[i].z += a * x.z;
              Oo[i].w += a * x.w;
            }
          }
        }
        if (single) {
#pragma unroll
          for (int i = 0; i < RPW; ++i) {
            const int r = warp + kConsumerWarps * i;
            if (r < G) {
              const float inv = 1.f / Lo[i];
              store_bf16x4(out_h + r * kHeadDim + d4, Oo[i].x * inv, Oo[i].y * inv, Oo[i].z * inv,
                           Oo[i].w * inv);
            }
          }
        } else {
          bool last = early_last;
          if (!last) {
            // Publish this CTA's record GPU-wide and count it.
            float* rec = p.pieces + (int64_t)(k + h) * kPieceFloats;  // m[16] l[16] o[16][128]
#pragma unroll
            for (int i = 0; i < RPW; ++i) {
              const int r = warp + kConsumerWarps * i;
              if (r < G) {
                *reinterpret_cast<float4*>(rec + 2 * kMaxGroup + r * kHeadDim + d4) = Oo[i];
                if (lane == 0) {
                  rec[r] = Mo[i];
                  rec[kMaxGroup + r] = Lo[i];
                }
              }
            }
            // The barrier orders every consumer thread's record stores before thread
            // 0's acquire-release atomic, whose release covers them.
            consumer_bar_sync();
            if (tid == 0)
              s_misc[1] = (atomic_add_acq_rel(p.piece_counters + h, 1) == k_hi - k_lo) ? 1 : 0;
            consumer_bar_sync();
            last = s_misc[1] != 0;
          }
          if (last) {
            // Log-sum-exp merge of every CTA's part in CTA order (this CTA's from
            // registers), four records' loads in flight at a time.
            float Mr[RPW], Lr[RPW];
            float4 Or[RPW];
#pragma unroll
            for (int i = 0; i < RPW; ++i) {
              Mr[i] = -INFINITY;
              Lr[i] = 0.f;
              Or[i] = make_float4(0.f, 0.f, 0.f, 0.f);
            }
            constexpr int kBatch = NT == 1 ? 4 : 2;
            for (int kk0 = k_lo; kk0 <= k_hi; kk0 += kBatch) {
              float mb[kBatch][RPW], lb[kBatch][RPW];
              float4 ob[kBatch][RPW];
#pragma unroll
              for (int u = 0; u < kBatch; ++u) {
                const int kk = kk0 + u;
                const float* rk = p.pieces + (int64_t)(kk + h) * kPieceFloats;
#pragma unroll
                for (int i = 0; i < RPW; ++i) {
                  const int r = warp + kConsumerWarps * i;
                  if (kk == k) {
                    mb[u][i] = Mo[i];
                    lb[u][i] = Lo[i];
                    ob[u][i] = Oo[i];
                  } else if (kk <= k_hi && r < G) {
                    mb[u][i] = __ldcg(rk + r);
                    lb[u][i] = __ldcg(rk + kMaxGroup + r);
                    ob[u][i] = __ldcg(reinterpret_cast<const float4*>(rk + 2 * kMaxGroup + r * kHeadDim + d4));
                  }
                }
              }
#pragma unroll
              for (int u = 0; u < kBatch; ++u) {
#pragma unroll
                for (int i = 0; i < RPW; ++i) {
                  if (kk0 + u <= k_hi && warp + kConsumerWarps * i < G) {
                    const float Mn = fmaxf(Mr[i], mb[u][i]);
                    const float a = exp2f(Mr[i] - Mn), bw = exp2f(mb[u][i] - Mn);
                    Lr[i] = Lr[i] * a + lb[u][i] * bw;
                    Or[i].x = Or[i].x * a + ob[u][i].x * bw;
                    Or[i].y = Or[i].y * a + ob[u][i].y * bw;
                    Or[i].z = Or[i].z * a + ob[u][i].z * bw;
                    Or[i].w = Or[i].w * a + ob[u][i].w * bw;
                    Mr[i] = Mn;
                  }
                }
              }
            }
#pragma unroll
            for (int i = 0; i < RPW; ++i) {
              const int r = warp + kConsumerWarps * i;
              if (r < G) {
                const float inv = 1.f / Lr[i];
                store_bf16x4(out_h + r * kHeadDim + d4, Or[i].x * inv, Or[i].y * inv, Or[i].z * inv,
                             Or[i].w * inv);
              }
            }
            if (tid == 0) p.piece_counters[h] = 0;
          }
        }
      }
    }
    walk.advance();
  }
}

// ---------------------------------------------------------------- cluster kernel
//
// Few heads (a batch of one or two sequences): one flat split of their pages over all
// SMs would split every head over many CTAs, and the merge of a head's records then
// costs global round trips (an arrival atomic, then the records).  Instead a
// thread-block cluster of C CTAs takes each head: CTA r of the cluster streams the
// head's pages r, r + C, r + 2C, ... exactly as a tiled CTA streams one segment and
// stores its partial (m, l, O) of each query-head row i into the shared memory of CTA
// i mod C of the cluster (asynchronous distributed-shared-memory stores counted on that
// CTA's mbarrier); once its rows' partials have landed, that CTA merges each row over the
// C partials in rank order (deterministic) and writes it.
//
// Early start.  The layer's state (count, ring, page table, pages) changes only in
// launches that append to this layer.  A fused cluster launch publishes, per head, a
// sequence number as soon as its writes of that head's state (count, ring entry, an
// opened page, the new row) are visible.  No launch can still be reading what these
// writes change: opening a page writes past every earlier launch's reads, and everything
// else is written after the launch's own dependency wait, when every earlier launch has
// completed.  The host knows the number the last such launch published (flag_expect; 0
// if the state was last written otherwise).  A launch with flag_expect != 0 waits only
// for its head's flag, then reads the state and stages its first pages before the
// dependency wait, which then guards only the inputs (q, the new K/V rows and logits)
// and the output.  A flag that does not arrive within the wait limit records
// DMS_ERR_TIMEOUT and the launch falls back to the dependency wait, which orders
// everything before it.
// Two groups of four consumer warps take alternate pages (a page's 64 rows are 16 per
// warp of its group), so that two pages are in the tensor cores at once: one warp per
// sub-partition leaves the MMA and shared-memory latencies of a page exposed.
constexpr int kClusterGroups = 2;
constexpr int kClusterConsumerWarps = 4 * kClusterGroups;
constexpr int kClusterThreads = (kClusterConsumerWarps + 1) * 32;  // + a producer warp
// Stages of the page ring: six 32 KiB bf16 pages, or twelve 16.5 KiB fp8 pages (K codes,
// V^T codes, the 128 row scales), in about the same 210 KB.
template <bool kFp8>
__host__ __device__ constexpr int cluster_stages() { return kFp8 ? 12 : 6; }
constexpr int kClusterMaxSize = 16;
constexpr int kClusterMinSize = 1;  // a cluster of one CTA: the head's pages, no merge
constexpr int kClusterShortSize = 6;
constexpr int kClusterLongSize = 10;
constexpr int64_t kClusterShortTokens = 8192;
constexpr int kClusterQBytes = 8 * kQRowPadded;  // up to 8 query heads, padded rows

__host__ __device__ constexpr int cluster_stage_bytes(bool fused, bool fp8) {
  return (fp8 ? 2 * kHalfPageBytesFp8 + kScaleBytes : 2 * kHalfPageBytes) + (fused ? kPatchBytes : 0);
}

// Partials received from every CTA of the cluster for the query-head rows this CTA owns
// (rows r with r % C == rank: at most ceil(8 / C) rows, ceil(8 / C) C <= 16 partials for
// every C in [1, 16]): O, then (m, l).
constexpr int kClusterRecvSlots = 16;
constexpr int kClusterRecvBytes = kClusterRecvSlots * (kHeadDim + 2) * 4;

template <bool kFused, bool kFp8>
size_t cluster_smem_bytes() {
  return (size_t)cluster_stages<kFp8>() * cluster_stage_bytes(kFused, kFp8) + kClusterQBytes +
         kClusterRecvBytes + (size_t)(2 * cluster_stages<kFp8>() + 2) * sizeof(uint64_t) +
         16 * sizeof(int);
}

// The per-warp partials overlay the stages once every page is consumed.
static_assert(kClusterConsumerWarps * 8 * (kMergeRow + 2) * 4 <=
                  cluster_stages<false>() * cluster_stage_bytes(false, false) &&
              kClusterConsumerWarps * 8 * (kMergeRow + 2) * 4 <=
                  cluster_stages<true>() * cluster_stage_bytes(false, true),
              "merge buffers must fit in the stages");
// The consumers wait on a stage's full barrier by phase parity, which only tells the last
// completed phase from the one before: a group must never wait for use u + 1 of a stage
// before use u has completed.  That holds when every use of a stage is read by the same
// group (in order), i.e. when the stage count is a multiple of the group count.
static_assert(cluster_stages<false>() % kClusterGroups == 0 &&
              cluster_stages<true>() % kClusterGroups == 0, "a stage is always read by the same group");

// E4M3 codes of head_dim 4 lane .. 4 lane + 3 of a bf16 row (two words per lane, the whole
// warp holding the row) and the row's scale, as the append kernels quantise: scale =
// amax(|row|) / 448 (fp32 division), code = E4M3(x / scale) rounded to nearest even and
// saturated; a row of zeros has scale 0 and codes 0.  pair[e] holds dims 4 lane + 2e (low
// byte) and 4 lane + 2e + 1.
__device__ __forceinline__ float quantize_row_e4m3(uint2 w, uint16_t (&pair)[2]) {
  float x[4];
  x[0] = __uint_as_float(w.x << 16);
  x[1] = __uint_as_float(w.x & 0xffff0000u);
  x[2] = __uint_as_float(w.y << 16);
  x[3] = __uint_as_float(w.y & 0xffff0000u);
  float a = fmaxf(fmaxf(fabsf(x[0]), fabsf(x[1])), fmaxf(fabsf(x[2]), fabsf(x[3])));
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) a = fmaxf(a, __shfl_xor_sync(0xffffffffu, a, off));
  const float scale = a == 0.f ? 0.f : __fdiv_rn(a, 448.f);
#pragma unroll
  for (int e = 0; e < 2; ++e) {
    const float lo = scale == 0.f ? 0.f : __fdiv_rn(x[2 * e], scale);
    const float hi = scale == 0.f ? 0.f : __fdiv_rn(x[2 * e + 1], scale);
    asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(pair[e]) : "f"(hi), "f"(lo));
  }
  return scale;
}

template <bool kFused, bool kFp8>
__global__ void __launch_bounds__(kClusterThreads, 1) decode_cluster_kernel(const DecodeParams p) {
  constexpr int HP = 8;
  constexpr int kClusterStages = cluster_stages<kFp8>();
  constexpr int kStageBytes = cluster_stage_bytes(kFused, kFp8);
  constexpr int kKvHalf = kFp8 ? kHalfPageBytesFp8 : kHalfPageBytes;  // the V half of a stage
  constexpr int kOffScales = 2 * kHalfPageBytesFp8;                   // fp8: K, V row scales
  constexpr int kOffPatch = kFp8 ? kOffScales + kScaleBytes : 2 * kHalfPageBytes;
  extern __shared__ __align__(128) uint8_t smem[];
  uint8_t* stages = smem;
  uint8_t* q_buf = smem + kClusterStages * kStageBytes;
  float* recv_o = reinterpret_cast<float*>(q_buf + kClusterQBytes);  // [C][128]
  float* recv_ml = recv_o + kClusterRecvSlots * kHeadDim;             // [C][2]
  uint64_t* full_bar = reinterpret_cast<uint64_t*>(recv_ml + 2 * kClusterRecvSlots);
  uint64_t* empty_bar = full_bar + kClusterStages;
  uint64_t* q_bar = empty_bar + kClusterStages;
  // [0] abort, [1] count after the append, [2] new slot | fresh << 30
  uint64_t* recv_bar = q_bar + 1;  // the partials of this CTA's rows have landed
  int* s_misc = reinterpret_cast<int*>(recv_bar + 1);
  float* merge_o = reinterpret_cast<float*>(smem);                    // [8][HP][132]
  float* merge_ml = merge_o + kClusterConsumerWarps * HP * kMergeRow;  // [8][HP][2]

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int G = p.group, Hq = p.kv_heads * p.group;
  volatile int* abort_flag = s_misc;
  const int C = (int)(gridDim.x / (unsigned)p.heads);  // cluster size (one cluster per head)
  const int rank = (int)cluster_ctarank();
  const int h = (int)blockIdx.x / C;
  const int b = h / p.kv_heads, hk = h - b * p.kv_heads;
  const int32_t* pt = p.page_table + (int64_t)h * p.max_pages;
  // Parameters used after the dependency wait, read before it (see pin_u32).
  const float scale_log2 = pin_f32(p.scale_log2);
  const uint32_t zero_first = pin_u32((uint32_t)p.zero_first);
  __nv_bfloat16* const out = pin_ptr(p.out);
  const __nv_bfloat16* const q_src = pin_ptr(p.q);
  const uint16_t* const k_new = pin_ptr(p.k_new);
  const uint16_t* const v_new = pin_ptr(p.v_new);
  const uint16_t* const logit_new = pin_ptr(p.logit_new);
  const int64_t logit_stride = pin_i64(p.logit_stride);
  int32_t* const counts_next = pin_ptr(p.counts_next);
  int32_t* const pos_out = pin_ptr(p.pos);
  const uint32_t flag_publish = pin_u32(p.flag_publish);

  pdl_launch_dependents();
  if (tid == 0) {
    s_misc[0] = 0;
    for (int s = 0; s < kClusterStages; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], kClusterConsumerWarps / kClusterGroups);
    }
    mbar_init(q_bar, 1);
    mbar_init(recv_bar, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    // Query-head rows r = rank, rank + C, ... (< G) are this CTA's: C partials of 520 bytes
    // each arrive for every one of them.
    const int own = G > rank ? (G - 1 - rank) / C + 1 : 0;
    if (own > 0 && C > 1) mbar_arrive_expect_tx(recv_bar, (uint32_t)(own * C * (kHeadDim + 2) * 4));
  }
  // Waited for before the first store into another CTA: that CTA runs, and its receive
  // barrier is initialised and expects its bytes (release / acquire).
  cluster_arrive_release();
  bool waited = false;  // producer warp: the dependency wait is behind it
  int32_t spec_page = -1, spec_page2 = -1;  // producer: page ids of its pages lane, lane + 32
  if (warp == kClusterConsumerWarps) {
    bool early = p.flag_expect != 0u;
    if (early) {
      int ok = 1;
      if (lane == 0 && ld_acquire_gpu_u32(p.head_flags + h) != p.flag_expect) {
        // Not yet published (the timer is read only here: it costs a round trip).
        const unsigned long long t0 = global_timer_ns();
        const unsigned long long limit =
            p.flag_wait_ns > 0 ? (unsigned long long)p.flag_wait_ns : kWaitLimitNs;
        for (uint32_t spin = 1;; ++spin) {
          __nanosleep(32);
          if (ld_acquire_gpu_u32(p.head_flags + h) == p.flag_expect) break;
          if ((spin & 31u) == 0u && global_timer_ns() - t0 > limit) {
            ok = 0;
            break;
          }
        }
        if (!ok) set_device_error(p.ctrl, DMS_ERR_TIMEOUT);
      }
      if (lane == 0) fence_proxy_async_global();  // the pages were written through the generic proxy
      early = __shfl_sync(0xffffffffu, ok, 0) != 0;
      // Lane 0's acquire, then a warp barrier (which orders memory among its threads): every
      // lane's state reads below come after the flag.
      __syncwarp();
    }
    if (!early) {
      pdl_wait_prerequisites();
      waited = true;
    }
    // The head's count, (fused) the ring entry of the token leaving the window, and the
    // page-table entries of this CTA's first 64 pages (two per lane), all in flight at once.
    // Fused: delayed eviction for position j (Sec. 3.1-3.2): the token j - window - 1
    // leaves the window; if it was flagged, the new token takes its slot, otherwise the
    // fresh slot n_h.
    const int32_t n = __ldcg(p.counts + h);
    uint32_t e = 0u;
    if (kFused && lane == 0 && p.j >= p.window + 1)
      e = __ldcg(p.ring + (int64_t)h * p.ring_len + (p.j - p.window - 1) % ring_period(p.window));
    const int spec_pg = rank + C * lane;
    if (spec_pg < p.max_pages) spec_page = __ldcg(pt + spec_pg);
    if (spec_pg + 32 * C < p.max_pages) spec_page2 = __ldcg(pt + spec_pg + 32 * C);
    if (lane == 0) {
      int32_t cnt = n;
      uint32_t slot_info = 0u;
      if constexpr (kFused) {
        const bool reuse = (e & kAlphaBit) != 0u;
        const uint32_t slot = reuse ? (e & kSlotMask) : (uint32_t)n;
        cnt = n + (reuse ? 0 : 1);
        slot_info = slot | ((reuse ? 0u : 1u) << 30);
      }
      s_misc[1] = cnt;
      s_misc[2] = (int)slot_info;
    }
  }
  __syncthreads();
  const int cnt = s_misc[1];
  const uint32_t slot_info = (uint32_t)s_misc[2];
  const int32_t new_slot = (int32_t)(slot_info & 0x3fffffffu);
  const bool fresh = ((slot_info >> 30) & 1u) != 0u;
  const int pg_new = kFused ? new_slot / kPageTokens : -1;  // the page the new token lands in
  const bool opens = kFused && fresh && new_slot % kPageTokens == 0;
  const bool patch_cta = kFused && rank == pg_new % C;  // the CTA of the new row's page
  const int pages = (cnt + kPageTokens - 1) / kPageTokens;
  const int niters = rank < pages ? (pages - 1 - rank) / C + 1 : 0;

  if (warp == kClusterConsumerWarps) {
    // ================================================================ producer warp
    int patch_stage = -1;  // a stage staged before the wait whose patch is still to come
    // Fused, the CTA whose pages include the new row's page (pg_new): that page's id,
    // opened here if the new token starts it.
    int patch_page = -1;
    if (patch_cta) {
      // An existing page among this CTA's first 64 has its id in a lane already.
      const int li = (pg_new - rank) / C;  // pg_new's place among this CTA's pages
      const int known = __shfl_sync(0xffffffffu, li < 32 ? spec_page : spec_page2, li & 31);
      if (lane == 0) {
        if (opens) {
          patch_page = atomicAdd(p.ctrl + kCtrlPoolNext, 1);
          if ((int64_t)patch_page >= p.pool_pages) {  // entered as -1: nothing is written there
            set_device_error(p.ctrl, DMS_ERR_CAPACITY);
            patch_page = -1;
          }
          p.page_table[(int64_t)h * p.max_pages + pg_new] = patch_page;
        } else {
          patch_page = li < 64 ? known : __ldcg(pt + pg_new);
        }
      }
      patch_page = __shfl_sync(0xffffffffu, patch_page, 0);
    }
    // After the dependency wait: the query rows and a pending patch.  Then (fused, the CTA
    // of the new row's page, write_new_row) the new K and V rows into the pool (from the
    // inputs), the position, the head's new count and ring entry: the layer's state of this
    // head is then complete and this launch's flag for the head is published.  (A later
    // launch writes this state only after its dependency wait, when this grid has
    // completed, so the flag need not wait for this launch's page reads; and this launch's
    // consumer warps take the new row from their own copy of it, whatever the bulk copy of
    // the page read.)
    auto after_wait = [&]() {
      if (lane == 0) {
        if (niters > 0) {
          mbar_arrive_expect_tx(q_bar, (uint32_t)G * kRowBytes);
          const __nv_bfloat16* qs = q_src + ((int64_t)b * Hq + (int64_t)hk * G) * kHeadDim;
          for (int i = 0; i < G; ++i)
            bulk_copy_g2s(q_buf + i * kQRowPadded, qs + (int64_t)i * kHeadDim, kRowBytes, q_bar);
        }
        if (kFused && patch_stage >= 0) {
          uint8_t* st = stages + patch_stage * kStageBytes;
          bulk_copy_g2s(st + kOffPatch, k_new + (int64_t)h * kHeadDim, kRowBytes, &full_bar[patch_stage]);
          bulk_copy_g2s(st + kOffPatch + kRowBytes, v_new + (int64_t)h * kHeadDim, kRowBytes,
                        &full_bar[patch_stage]);
        }
      }
      __syncwarp();
    };
    // Fused, the CTA of the new row's page, once the dependency wait is behind it and its
    // first pages are in flight: the new row and the head's state, then the flag.
    bool row_done = !(kFused && patch_cta);
    auto write_new_row = [&]() {
      if (kFused && patch_cta) {
        const uint32_t r = (uint32_t)(new_slot % kPageTokens);
        if constexpr (kFp8) {  // quantise both rows (lane: head_dim 4 lane .. 4 lane + 3)
          uint8_t* pg8 = p.pool + (int64_t)(patch_page < 0 ? 0 : patch_page) * kPageBytesFp8;
#pragma unroll
          for (int kv = 0; kv < 2; ++kv) {
            const uint2 w = __ldg(reinterpret_cast<const uint2*>((kv ? v_new : k_new) +
                                                                 (int64_t)h * kHeadDim) + lane);
            uint16_t pair[2];
            const float scale = quantize_row_e4m3(w, pair);
            if (patch_page >= 0) {
#pragma unroll
              for (int e = 0; e < 2; ++e) {
                const uint32_t d = 4u * (uint32_t)lane + 2u * (uint32_t)e;
                if (kv == 0) {
                  *reinterpret_cast<uint16_t*>(pg8 + k8_offset(r, d)) = pair[e];
                } else {
                  pg8[vt8_offset(r, d)] = (uint8_t)(pair[e] & 0xffu);
                  pg8[vt8_offset(r, d + 1)] = (uint8_t)(pair[e] >> 8);
                }
              }
              if (lane == 0)
                page_scales_fp8(p.pool, patch_page)[kv * kPageTokens + r] = scale;
            }
          }
          if (patch_page >= 0 && lane == 0)
            pos_out[(int64_t)patch_page * kPageTokens + r] = (int32_t)p.j;
        } else {
          const int half = lane >> 4, chunk = lane & 15;
          const uint4 val = __ldg(reinterpret_cast<const uint4*>((half ? v_new : k_new) +
                                                                 (int64_t)h * kHeadDim) + chunk);
          if (patch_page >= 0) {
            const uint32_t off = (uint32_t)half * kHalfPageBytes + swizzled_offset(r, (uint32_t)chunk);
            *reinterpret_cast<uint4*>(p.pool + (int64_t)patch_page * kPageBytes + off) = val;
            if (lane == 0) pos_out[(int64_t)patch_page * kPageTokens + r] = (int32_t)p.j;
          }
        }
        if (lane == 0) {
          const uint32_t alpha = decision_from_bf16(logit_new[(int64_t)h * logit_stride]);
          counts_next[h] = cnt;
          uint32_t* rh = p.ring + (int64_t)h * p.ring_len;
          const int64_t RP = ring_period(p.window);
          rh[p.j % RP] = (uint32_t)new_slot | ((p.decider == 0 ? alpha : 0u) << 31);
          if (p.decider > 0 && p.j >= p.decider) rh[(p.j - p.decider) % RP] |= alpha << 31;
        }
        fence_proxy_async_global();  // a later launch reads the row with a bulk copy
        __threadfence();
        __syncwarp();
        if (lane == 0 && flag_publish != 0u) st_release_gpu_u32(p.head_flags + h, flag_publish);
      }
      row_done = true;
    };
    if (waited) after_wait();
    const int first = niters < kClusterStages ? niters : kClusterStages;  // staged before the wait
    for (int it0 = 0; it0 < niters; it0 += 32) {
      const int it = it0 + lane;
      int nv = 0, page = 0;
      if (it < niters) {
        const int pg = rank + C * it;
        nv = min(kPageTokens, cnt - pg * kPageTokens);
        if (kFused && pg == pg_new) {
          page = patch_page;
        } else {
          page = it0 == 0 ? spec_page : it0 == 32 ? spec_page2 : __ldcg(pt + pg);
        }
      }
      const int nb = min(32, niters - it0);
      for (int i = 0; i < nb; ++i) {
        const int nv_i = __shfl_sync(0xffffffffu, nv, i);
        const int page_i = __shfl_sync(0xffffffffu, page, i);
        const int itg = it0 + i;
        if (lane == 0) {
          const int s = itg % kClusterStages;
          const int use = itg / kClusterStages;
          if (use > 0) mbar_wait(&empty_bar[s], (use - 1) & 1, abort_flag, p.ctrl);
          const bool patch = kFused && rank + C * itg == pg_new;
          uint8_t* st = stages + s * kStageBytes;
          const int64_t page0 = page_i < 0 ? 0 : page_i;
          if constexpr (kFp8) {
            // the whole page (K codes, V^T codes, row scales) in one copy, as each bulk copy
            // has a fixed issue cost: K rows past n_valid are masked like stale ones, and all
            // of V^T is needed (its rows interleave the slots)
            static_assert(kKvHalf == kHalfPageBytesFp8 && kOffScales == kPageCodesBytesFp8,
                          "a stage holds the page as laid out in the pool");
            mbar_arrive_expect_tx(&full_bar[s], (uint32_t)kPageBytesFp8 +
                                                    (patch ? (uint32_t)kPatchBytes : 0u));
            bulk_copy_g2s(st, p.pool + page0 * kPageBytesFp8, kPageBytesFp8, &full_bar[s]);
          } else {
            const uint32_t kv_bytes = (uint32_t)nv_i * (uint32_t)kRowBytes;
            mbar_arrive_expect_tx(&full_bar[s], 2 * kv_bytes + (patch ? (uint32_t)kPatchBytes : 0u));
            const uint8_t* src = p.pool + page0 * kPageBytes;
            if (nv_i == kPageTokens) {  // a full page: K and V halves in one copy
              bulk_copy_g2s(st, src, 2 * kHalfPageBytes, &full_bar[s]);
            } else {  // the valid rows of each half
              bulk_copy_g2s(st, src, kv_bytes, &full_bar[s]);
              bulk_copy_g2s(st + kHalfPageBytes, src + kHalfPageBytes, kv_bytes, &full_bar[s]);
            }
          }
          if (patch) {  // the new token's K and V rows, as given (unpermuted)
            if (waited) {
              bulk_copy_g2s(st + kOffPatch, k_new + (int64_t)h * kHeadDim, kRowBytes, &full_bar[s]);
              bulk_copy_g2s(st + kOffPatch + kRowBytes, v_new + (int64_t)h * kHeadDim, kRowBytes,
                            &full_bar[s]);
            } else {
              patch_stage = s;
            }
          }
        }
        if (!waited && itg + 1 == first) {  // the first stages are in flight: now the inputs
          pdl_wait_prerequisites();
          waited = true;
          patch_stage = __shfl_sync(0xffffffffu, patch_stage, 0);
          after_wait();
        }
        if (!row_done && itg + 1 >= first) write_new_row();
      }
    }
    if (!waited) {  // a CTA without pages
      pdl_wait_prerequisites();
      waited = true;
      after_wait();
    }
    if (!row_done) write_new_row();
    // Drain: do not leave while a bulk copy may still be writing shared memory.
    if (lane == 0) {
      for (int s = 0; s < kClusterStages && s < niters; ++s) {
        const int last_it = s + ((niters - 1 - s) / kClusterStages) * kClusterStages;
        mbar_wait(&full_bar[s], (last_it / kClusterStages) & 1, abort_flag, p.ctrl);
      }
      if (niters > 0) mbar_wait(q_bar, 0, abort_flag, p.ctrl);
    }
    __syncwarp();
    cluster_wait();
  } else {
    // ================================================================ consumer warps
    const int g = lane >> 2, c4 = lane & 3;
    const int grp = warp >> 2, sub = warp & 3;  // pages grp, grp + 2, ...; rows 16 sub ..
    const int tb = sub * 16;                     // this warp's first token within a page
    const int mi = lane >> 3;
    uint32_t qb[8][2];
    float o[8][4];
    float me = -INFINITY, mo = -INFINITY, le = 0.f, lo = 0.f;
#pragma unroll
    for (int mt = 0; mt < 8; ++mt) o[mt][0] = o[mt][1] = o[mt][2] = o[mt][3] = 0.f;
    if (niters > 0) {
      mbar_wait(q_bar, 0, abort_flag, p.ctrl);
      const uint32_t qbase = smem_addr(q_buf);
      const int row = lane & 7;
#pragma unroll
      for (int k2 = 0; k2 < 4; ++k2) {
        const int kk = 2 * k2 + (mi >> 1);
        uint32_t r0, r1, r2, r3;
        ldsm_x4(qbase + row * kQRowPadded + (2 * kk + (mi & 1)) * 16, r0, r1, r2, r3);
        const bool live = g < G;
        qb[2 * k2][0] = live ? r0 : 0u;
        qb[2 * k2][1] = live ? r1 : 0u;
        qb[2 * k2 + 1][0] = live ? r2 : 0u;
        qb[2 * k2 + 1][1] = live ? r3 : 0u;
      }
      if constexpr (kFp8) {  // the fp8 path multiplies in f16
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
          qb[kk][0] = bf16x2_to_f16x2(qb[kk][0]);
          qb[kk][1] = bf16x2_to_f16x2(qb[kk][1]);
        }
      }
      if (zero_first && lane == 0) qb[0][0] &= 0xffff0000u;
    }
    for (int it = grp; it < niters; it += kClusterGroups) {
      const int s = it % kClusterStages;
      const int use = it / kClusterStages;
      const int pg = rank + C * it;
      const int nvalid = min(kPageTokens, cnt - pg * kPageTokens);
      uint8_t* st = stages + s * kStageBytes;
      mbar_wait(&full_bar[s], use & 1, abort_flag, p.ctrl);
      if constexpr (kFused) {
        const uint32_t r = (uint32_t)(new_slot % kPageTokens);
        if (pg == pg_new && (int)(r >> 4) == sub) {
          // The warp whose 16 rows hold the new token moves its K and V row from the
          // patch buffer into the staged page (permuted layout; fp8: quantised, with the
          // row scales, exactly as the producer warp writes them to the pool); the producer
          // warp writes the row to the pool and the head's state.
          if constexpr (kFp8) {
#pragma unroll
            for (int kv = 0; kv < 2; ++kv) {
              const uint2 w = *reinterpret_cast<const uint2*>(st + kOffPatch + kv * kRowBytes + lane * 8);
              uint16_t pair[2];
              const float scale = quantize_row_e4m3(w, pair);
#pragma unroll
              for (int e = 0; e < 2; ++e) {
                const uint32_t d = 4u * (uint32_t)lane + 2u * (uint32_t)e;
                if (kv == 0) {
                  *reinterpret_cast<uint16_t*>(st + k8_offset(r, d)) = pair[e];
                } else {
                  st[vt8_offset(r, d)] = (uint8_t)(pair[e] & 0xffu);
                  st[vt8_offset(r, d + 1)] = (uint8_t)(pair[e] >> 8);
                }
              }
              if (lane == 0) reinterpret_cast<float*>(st + kOffScales)[kv * kPageTokens + r] = scale;
            }
          } else {
            const int half = lane >> 4, chunk = lane & 15;
            const uint4 val =
                *reinterpret_cast<const uint4*>(st + kOffPatch + half * kRowBytes + chunk * 16);
            const uint32_t off = (uint32_t)half * kHalfPageBytes + swizzled_offset(r, (uint32_t)chunk);
            *reinterpret_cast<uint4*>(st + off) = val;
          }
          fence_proxy_async_shared();
          __syncwarp();
        }
      }
      if (tb < nvalid) {
        float sacc[4][4];
#pragma unroll
        for (int c = 0; c < 4; ++c)
#pragma unroll
          for (int e = 0; e < 4; ++e) sacc[c][e] = 0.f;
        if constexpr (kFp8) {
          // rows tb + g and tb + g + 8; the 16-byte chunk of k-steps 4 kg .. 4 kg + 3 holds
          // this thread's codes (d = 16 kk + {2c, 2c+1, 2c+8, 2c+9}) in word kk % 4
#pragma unroll
          for (int kg = 0; kg < 2; ++kg) {
            const uint4 w0 = *reinterpret_cast<const uint4*>(st + (tb + g) * 128 + (((4 * kg + c4) ^ k8_swizzle(g)) << 4));
            const uint4 w1 =
                *reinterpret_cast<const uint4*>(st + (tb + g + 8) * 128 + (((4 * kg + c4) ^ k8_swizzle(g)) << 4));
            const uint32_t x0[4] = {w0.x, w0.y, w0.z, w0.w}, x1[4] = {w1.x, w1.y, w1.z, w1.w};
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              const int kk = 4 * kg + i;
              uint32_t a[4];
              a[0] = e4m3x2_to_f16x2(x0[i]);
              a[1] = e4m3x2_to_f16x2(x1[i]);
              a[2] = e4m3x2_to_f16x2(x0[i] >> 16);
              a[3] = e4m3x2_to_f16x2(x1[i] >> 16);
              mma_f16_16816(sacc[kk & 3], a, qb[kk][0], qb[kk][1]);
            }
          }
        } else {
          const uint32_t kbase = smem_addr(st);
          const uint32_t krow = (uint32_t)(tb + (mi & 1) * 8 + (lane & 7));
#pragma unroll
          for (int kk = 0; kk < 8; ++kk) {
            uint32_t a[4];
            ldsm_x4(kbase + swizzled_offset(krow, (uint32_t)(2 * kk + (mi >> 1))), a[0], a[1], a[2], a[3]);
            mma_bf16_16816(sacc[kk & 3], a, qb[kk][0], qb[kk][1]);
          }
        }
        const bool v0 = tb + g < nvalid, v1 = tb + g + 8 < nvalid;
        // score scale of tokens tb + g and tb + g + 8 (fp8: times the keys' row scales); fp8
        // also folds each value's row scale into P, per token (stale tokens take 0)
        float sl0 = scale_log2, sl1 = scale_log2, vs0 = 1.f, vs1 = 1.f;
        if constexpr (kFp8) {
          const float* ksc = reinterpret_cast<const float*>(st + kOffScales);
          sl0 *= ksc[tb + g];
          sl1 *= ksc[tb + g + 8];
          vs0 = v0 ? ksc[kPageTokens + tb + g] : 0.f;
          vs1 = v1 ? ksc[kPageTokens + tb + g + 8] : 0.f;
        }
        float sc[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) sc[e] = (sacc[0][e] + sacc[1][e]) + (sacc[2][e] + sacc[3][e]);
        const float s0 = v0 ? sc[0] * sl0 : -INFINITY, s1 = v0 ? sc[1] * sl0 : -INFINITY;
        const float s2 = v1 ? sc[2] * sl1 : -INFINITY, s3 = v1 ? sc[3] * sl1 : -INFINITY;
        float xe = fmaxf(s0, s2), xo = fmaxf(s1, s3);
#pragma unroll
        for (int off = 4; off < 32; off <<= 1) {
          xe = fmaxf(xe, __shfl_xor_sync(0xffffffffu, xe, off));
          xo = fmaxf(xo, __shfl_xor_sync(0xffffffffu, xo, off));
        }
        const float ne = fmaxf(me, xe), no = fmaxf(mo, xo);
        const float ce = ex2_approx(me - ne), co = ex2_approx(mo - no);
        me = ne;
        mo = no;
        const float p0 = ex2_approx(s0 - ne), p1 = ex2_approx(s1 - no);
        const float p2 = ex2_approx(s2 - ne), p3 = ex2_approx(s3 - no);
        le = le * ce + (p0 + p2);
        lo = lo * co + (p1 + p3);
        const uint32_t pb0 = kFp8 ? movmatrix_trans(pack_f16x2(p0 * vs0, p1 * vs0))
                                  : movmatrix_trans(pack_bf16x2(p0, p1));
        const uint32_t pb1 = kFp8 ? movmatrix_trans(pack_f16x2(p2 * vs1, p3 * vs1))
                                  : movmatrix_trans(pack_bf16x2(p2, p3));
        if (__any_sync(0xffffffffu, (ce != 1.f) || (co != 1.f))) {
#pragma unroll
          for (int mt = 0; mt < 8; ++mt) {
            o[mt][0] *= ce;
            o[mt][1] *= co;
            o[mt][2] *= ce;
            o[mt][3] *= co;
          }
        }
        uint32_t mk_lo = 0xffffffffu, mk_hi = 0xffffffffu;
        if (tb + 16 > nvalid) {  // stale rows past n_valid must not reach the tensor cores
          const int t = tb + 2 * c4;
          mk_lo = (t < nvalid ? 0x0000ffffu : 0u) | (t + 1 < nvalid ? 0xffff0000u : 0u);
          mk_hi = (t + 8 < nvalid ? 0x0000ffffu : 0u) | (t + 9 < nvalid ? 0xffff0000u : 0u);
        }
        if constexpr (kFp8) {
          // V^T rows d = 16 mt + g and + 8: one word holds the codes of tokens tb + {2c, 2c+1,
          // 2c+8, 2c+9} (the row scales are in P); stale tokens masked
          const int blk = tb >> 4;
#pragma unroll
          for (int mt = 0; mt < 8; ++mt) {
            const int d0 = 16 * mt + g, d1 = d0 + 8;
            const uint32_t w0 = *reinterpret_cast<const uint32_t*>(
                st + kKvHalf + d0 * 64 + ((blk ^ ((d0 >> 1) & 3)) << 4) + 4 * c4);
            const uint32_t w1 = *reinterpret_cast<const uint32_t*>(
                st + kKvHalf + d1 * 64 + ((blk ^ ((d1 >> 1) & 3)) << 4) + 4 * c4);
            uint32_t a[4];
            a[0] = e4m3x2_to_f16x2(w0) & mk_lo;
            a[1] = e4m3x2_to_f16x2(w1) & mk_lo;
            a[2] = e4m3x2_to_f16x2(w0 >> 16) & mk_hi;
            a[3] = e4m3x2_to_f16x2(w1 >> 16) & mk_hi;
            mma_f16_16816(o[mt], a, pb0, pb1);
          }
        } else {
          const uint32_t vbase = smem_addr(st + kHalfPageBytes);
          const uint32_t vrow = (uint32_t)(tb + (mi >> 1) * 8 + (lane & 7));
#pragma unroll
          for (int mt = 0; mt < 8; ++mt) {
            uint32_t a[4];
            ldsm_x4_trans(vbase + swizzled_offset(vrow, (uint32_t)(2 * mt + (mi & 1))), a[0], a[1], a[2], a[3]);
            a[0] &= mk_lo;
            a[1] &= mk_lo;
            a[2] &= mk_hi;
            a[3] &= mk_hi;
            mma_bf16_16816(o[mt], a, pb0, pb1);
          }
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty_bar[s]);
    }
    // ---- every consumer warp is done with the stages (and every copy into them has
    // landed): the partials overlay them.  This warp's partial, then the CTA's (warp w
    // merges query-head row w).
    named_bar_sync<1>(kClusterConsumerWarps * 32);
    {
      float te = le, to = lo;
#pragma unroll
      for (int off = 4; off < 32; off <<= 1) {
        te += __shfl_xor_sync(0xffffffffu, te, off);
        to += __shfl_xor_sync(0xffffffffu, to, off);
      }
      float* so = merge_o + warp * HP * kMergeRow;
      float* sml = merge_ml + warp * HP * 2;
      const int he = 2 * c4, ho = he + 1;
      if (g == 0) {
        sml[he * 2] = me;
        sml[he * 2 + 1] = te;
        sml[ho * 2] = mo;
        sml[ho * 2 + 1] = to;
      }
#pragma unroll
      for (int mt = 0; mt < 8; ++mt) {
        so[he * kMergeRow + 16 * mt + g] = o[mt][0];
        so[ho * kMergeRow + 16 * mt + g] = o[mt][1];
        so[he * kMergeRow + 16 * mt + g + 8] = o[mt][2];
        so[ho * kMergeRow + 16 * mt + g + 8] = o[mt][3];
      }
    }
    named_bar_sync<1>(kClusterConsumerWarps * 32);
    // The CTA's partial of query-head row r goes straight into the shared memory of its
    // owner, CTA r % C of the cluster, slot (r / C) C + rank (rows past G are not formed).
    const int d4 = 4 * lane;
    static_assert(kClusterConsumerWarps == 8, "one query-head row per consumer warp");
    cluster_wait();  // every CTA of the cluster runs
    {
      const int r = warp;
      if (r < G) {
        float M = -INFINITY, L = 0.f;
        float4 O = make_float4(0.f, 0.f, 0.f, 0.f);
        float mw[kClusterConsumerWarps];
#pragma unroll
        for (int w = 0; w < kClusterConsumerWarps; ++w) {
          mw[w] = merge_ml[(w * HP + r) * 2];
          M = fmaxf(M, mw[w]);
        }
#pragma unroll
        for (int w = 0; w < kClusterConsumerWarps; ++w) {
          const float a = mw[w] == -INFINITY ? 0.f : exp2f(mw[w] - M);
          const float4 x = *reinterpret_cast<const float4*>(merge_o + (w * HP + r) * kMergeRow + d4);
          L += a * merge_ml[(w * HP + r) * 2 + 1];
          O.x += a * x.x;
          O.y += a * x.y;
          O.z += a * x.z;
          O.w += a * x.w;
        }
        if (C == 1) {  // the CTA holds the whole head: its partial is the result
          const float inv = L > 0.f ? 1.f / L : 0.f;  // an empty head gives zeros
          store_bf16x4(out + ((int64_t)b * Hq + (int64_t)hk * G + r) * kHeadDim + d4, O.x * inv,
                       O.y * inv, O.z * inv, O.w * inv);
        } else {
          const int slot = (r / C) * C + rank;
          const uint32_t owner = (uint32_t)(r % C);
          const uint32_t rbar = mapa_shared(smem_addr(recv_bar), owner);
          st_async_cluster_v4(mapa_shared(smem_addr(recv_o + slot * kHeadDim + d4), owner), O, rbar);
          if (lane == 0)
            st_async_cluster_v2(mapa_shared(smem_addr(recv_ml + slot * 2), owner), M, L, rbar);
        }
      }
    }
  }
  // ---- CTA `rank` merges its rows r = li C + rank (warp li) over the cluster, in rank
  // order, once every CTA's partials of them have landed (no barrier across the cluster: a
  // CTA without rows leaves, and no CTA's shared memory is written after its rows are in)
  if (C > 1 && warp * C + rank < G) {
    mbar_wait(recv_bar, 0, abort_flag, p.ctrl);
    const int li = warp, r = li * C + rank, d4 = 4 * lane;
    const float* rml = recv_ml + li * C * 2;
    const float* ro = recv_o + li * C * kHeadDim;
    float M = -INFINITY, L = 0.f;
    float4 O = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int j = 0; j < C; ++j) {
      const float mj = rml[j * 2], lj = rml[j * 2 + 1];
      if (mj == -INFINITY) continue;  // a CTA without pages (or tokens) adds nothing
      const float4 oj = *reinterpret_cast<const float4*>(ro + j * kHeadDim + d4);
      const float Mn = fmaxf(M, mj);
      const float a = exp2f(M - Mn), w = exp2f(mj - Mn);
      L = L * a + lj * w;
      O.x = O.x * a + oj.x * w;
      O.y = O.y * a + oj.y * w;
      O.z = O.z * a + oj.z * w;
      O.w = O.w * a + oj.w * w;
      M = Mn;
    }
    const float inv = L > 0.f ? 1.f / L : 0.f;  // an empty head gives zeros
    store_bf16x4(out + ((int64_t)b * Hq + (int64_t)hk * G + r) * kHeadDim + d4, O.x * inv,
                 O.y * inv, O.z * inv, O.w * inv);
  }
}

// ---------------------------------------------------------------- simple kernel

__global__ void __launch_bounds__(128) decode_simple_kernel(const uint8_t* pool,
                                                            const int32_t* page_table,
                                                            const int32_t* counts,
                                                            const __nv_bfloat16* q,
                                                            __nv_bfloat16* out, int32_t kv_heads,
                                                            int32_t group, int32_t max_pages,
                                                            float scale, int32_t zero_first) {
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
    if (zero_first && gq == 0 && lane == 0) qv[0] = 0.f;  // the decision element (App. B)
    float m = -INFINITY, l = 0.f, acc[4] = {0.f, 0.f, 0.f, 0.f};
    for (int s = 0; s < n; ++s) {
      const int32_t page = pt[s / kPageTokens];
      if (page < 0) continue;  // the page pool ran out when this slot's page was to open
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

// Self-test of the bounded wait used by every kernel: thread 0 waits on an
// mbarrier of count 1; thread 32 arrives on it only when `arrive` is set.
__global__ void bounded_wait_probe_kernel(int arrive, unsigned long long limit_ns, int32_t* status) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    abort_flag = 0;
    mbar_init(&bar, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();
  if (threadIdx.x == 32 && arrive) mbar_arrive(&bar);
  if (threadIdx.x == 0) {
    const bool ok = mbar_try_wait(&bar, 0) ||
                    mbar_wait_slow(&bar, 0, &abort_flag, status, limit_ns);
    if (ok) status[kCtrlError + 1] = 1;  // completion seen
  }
}

}  // namespace

cudaError_t launch_bounded_wait_probe(int arrive, int64_t limit_ns, int32_t* dev_status,
                                      cudaStream_t stream) {
  bounded_wait_probe_kernel<<<1, 64, 0, stream>>>(arrive, (unsigned long long)limit_ns, dev_status);
  return cudaGetLastError();
}

cudaError_t prepare_decode(const Cache& c) {
  (void)c;
  // Sized for the largest head count any cache may have, so that caches of
  // different sizes never lower the limit under one another.
  cudaError_t e = cudaSuccess;
  auto set = [&](auto kernel, size_t bytes) {
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
  };
  set(decode_tiled_kernel<kStagesOneCta, 1, false>,
      tiled_smem_bytes<1, false>(kMaxHeads, kStagesOneCta));
  set(decode_tiled_kernel<kStagesOneCta, 2, false>,
      tiled_smem_bytes<2, false>(kMaxHeads, kStagesOneCta));
  set(decode_tiled_kernel<kStagesTwoCta, 1, false>,
      tiled_smem_bytes<1, false>(kMaxHeads, kStagesTwoCta));
  set(decode_tiled_kernel<kStagesTwoCta, 2, false>,
      tiled_smem_bytes<2, false>(kMaxHeads, kStagesTwoCta));
  set(decode_tiled_kernel<kStagesOneCta, 1, true>,
      tiled_smem_bytes<1, true>(kMaxHeadsFused, kStagesOneCta));
  set(decode_tiled_kernel<kStagesOneCta, 2, true>,
      tiled_smem_bytes<2, true>(kMaxHeadsFused, kStagesOneCta));
  set(decode_tiled_kernel<kStagesFp8, 1, false, true>,
      tiled_smem_bytes<1, false, true>(kMaxHeads, kStagesFp8));
  set(decode_tiled_kernel<kStagesFp8, 2, false, true>,
      tiled_smem_bytes<2, false, true>(kMaxHeads, kStagesFp8));
  set(decode_tiled_kernel<kStagesFp8Fused, 1, true, true>,
      tiled_smem_bytes<1, true, true>(kMaxHeadsFused, kStagesFp8Fused));
  set(decode_tiled_kernel<kStagesFp8Fused, 2, true, true>,
      tiled_smem_bytes<2, true, true>(kMaxHeadsFused, kStagesFp8Fused));
  auto set_cluster = [&](auto kernel, size_t bytes) {
    set(kernel, bytes);
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  };
  set_cluster(decode_cluster_kernel<false, false>, cluster_smem_bytes<false, false>());
  set_cluster(decode_cluster_kernel<true, false>, cluster_smem_bytes<true, false>());
  set_cluster(decode_cluster_kernel<false, true>, cluster_smem_bytes<false, true>());
  set_cluster(decode_cluster_kernel<true, true>, cluster_smem_bytes<true, true>());
  return e;
}

// Clusters of C CTAs of the cluster kernel that fit on the device at once (0 if none):
// one head per cluster, so a launch takes the cluster kernel only when every head's
// cluster is resident at the same time.
template <bool kFused, bool kFp8>
int max_active_clusters(int cluster_size) {
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)cluster_size;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.gridDim = dim3((unsigned)cluster_size * 16u);
  cfg.blockDim = dim3(kClusterThreads);
  cfg.dynamicSmemBytes = cluster_smem_bytes<kFused, kFp8>();
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  const cudaError_t e =
      cudaOccupancyMaxActiveClusters(&n, decode_cluster_kernel<kFused, kFp8>, &cfg);
  if (e != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  return n;
}

cudaError_t prepare_cluster_decode(Cache& c) {
  for (int cs = kClusterMinSize; cs <= kClusterMaxSize; ++cs) {
    const int n[4] = {max_active_clusters<false, false>(cs), max_active_clusters<true, false>(cs),
                      max_active_clusters<false, true>(cs), max_active_clusters<true, true>(cs)};
    int m = n[0];
    for (int i = 1; i < 4; ++i) m = n[i] < m ? n[i] : m;
    c.max_clusters[cs] = m;
  }
  return cudaSuccess;
}

// Cluster size for a decode of `group` query heads per KV head over a layer of `tokens`
// tokens on cache `c`, or 0 for the flat split: up to 8 query heads, the default split
// options, and a resident cluster for every head at once.  The default
// kernel takes clusters only when those of the largest size that fits cover at least half
// of the SMs: with fewer, a head of many pages streams faster through the flat split over
// every SM.  The size: a layer of at most kClusterShortTokens tokens (at most 22 pages per
// CTA at size 6 even if nothing was evicted) takes kClusterShortSize, small enough that
// the clusters of consecutive launches fit on the device side by side, so that each
// launch stages its pages while the one before runs; a longer layer takes
// kClusterLongSize, which spreads its pages over more SMs; either is capped by the largest
// size that fits.  The constants were measured on GB300 (152 SMs) on batch-1, 8-head
// layers from 4K to 64K tokens at 1x to 8x compression.
int decode_cluster_size(const Cache& c, int group, int64_t tokens) {
  if (group > 8 || c.ctas_per_sm >= 2 || c.min_pages_per_cta != 2 ||
      (c.decode_kernel != DMS_DECODE_TILED && c.decode_kernel != DMS_DECODE_CLUSTER))
    return 0;
  int largest = 0;
  for (int cs = kClusterMaxSize; cs >= kClusterMinSize && largest == 0; --cs)
    if (c.heads <= c.max_clusters[cs]) largest = cs;
  if (largest == 0) return 0;
  if (c.decode_kernel == DMS_DECODE_TILED && 2 * c.heads * largest < c.num_sms) return 0;
  const int want = tokens <= kClusterShortTokens ? kClusterShortSize : kClusterLongSize;
  return largest < want ? largest : want;
}

namespace {

// Launch with programmatic stream serialisation (the kernel waits for its
// prerequisites itself); the variant is picked by CTAs per SM, group size and
// whether the single-token append is fused in.
cudaError_t launch_tiled(const DecodeParams& p, int num_sms, int ctas_per_sm, cudaStream_t stream,
                         bool programmatic, bool fused, bool fp8 = false) {
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.blockDim = dim3(kThreads);
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = programmatic ? 1 : 0;
  if (fp8 && fused) {  // one CTA per SM
    cfg.gridDim = dim3(num_sms);
    if (p.group <= 8) {
      cfg.dynamicSmemBytes = tiled_smem_bytes<1, true, true>(p.heads, kStagesFp8Fused);
      return cudaLaunchKernelEx(&cfg, decode_tiled_kernel<kStagesFp8Fused, 1, true, true>, p);
    }
    cfg.dynamicSmemBytes = tiled_smem_bytes<2, true, true>(p.heads, kStagesFp8Fused);
    return cudaLaunchKernelEx(&cfg, decode_tiled_kernel<kStagesFp8Fused, 2, true, true>, p);
  }
  if (fp8) {  // one CTA per SM
    cfg.gridDim = dim3(num_sms);
    if (p.group <= 8) {
      cfg.dynamicSmemBytes = tiled_smem_bytes<1, false, true>(p.heads, kStagesFp8);
      return cudaLaunchKernelEx(&cfg, decode_tiled_kernel<kStagesFp8, 1, false, true>, p);
    }
    cfg.dynamicSmemBytes = tiled_smem_bytes<2, false, true>(p.heads, kStagesFp8);
    return cudaLaunchKernelEx(&cfg, decode_tiled_kernel<kStagesFp8, 2, false, true>, p);
  }
  const bool two = !fused && ctas_per_sm >= 2;
  const int stages = two ? kStagesTwoCta : kStagesOneCta;
  cfg.gridDim = dim3(num_sms * (two ? ctas_per_sm : 1));
  if (fused) {
    if (p.group <= 8) {
      cfg.dynamicSmemBytes = tiled_smem_bytes<1, true>(p.heads, stages);
      return cudaLaunchKernelEx(&cfg, decode_tiled_kernel<kStagesOneCta, 1, true>, p);
    }
    cfg.dynamicSmemBytes = tiled_smem_bytes<2, true>(p.heads, stages);
    return cudaLaunchKernelEx(&cfg, decode_tiled_kernel<kStagesOneCta, 2, true>, p);
  }
  if (p.group <= 8) {
    cfg.dynamicSmemBytes = tiled_smem_bytes<1, false>(p.heads, stages);
    return two ? cudaLaunchKernelEx(&cfg, decode_tiled_kernel<kStagesTwoCta, 1, false>, p)
               : cudaLaunchKernelEx(&cfg, decode_tiled_kernel<kStagesOneCta, 1, false>, p);
  }
  cfg.dynamicSmemBytes = tiled_smem_bytes<2, false>(p.heads, stages);
  return two ? cudaLaunchKernelEx(&cfg, decode_tiled_kernel<kStagesTwoCta, 2, false>, p)
             : cudaLaunchKernelEx(&cfg, decode_tiled_kernel<kStagesOneCta, 2, false>, p);
}

cudaError_t launch_cluster(const DecodeParams& p, int cluster_size, cudaStream_t stream, bool fused,
                           bool fp8) {
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)cluster_size;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.gridDim = dim3((unsigned)(p.heads * cluster_size));
  cfg.blockDim = dim3(kClusterThreads);
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  if (fp8) {
    if (fused) {
      cfg.dynamicSmemBytes = cluster_smem_bytes<true, true>();
      return cudaLaunchKernelEx(&cfg, decode_cluster_kernel<true, true>, p);
    }
    cfg.dynamicSmemBytes = cluster_smem_bytes<false, true>();
    return cudaLaunchKernelEx(&cfg, decode_cluster_kernel<false, true>, p);
  }
  if (fused) {
    cfg.dynamicSmemBytes = cluster_smem_bytes<true, false>();
    return cudaLaunchKernelEx(&cfg, decode_cluster_kernel<true, false>, p);
  }
  cfg.dynamicSmemBytes = cluster_smem_bytes<false, false>();
  return cudaLaunchKernelEx(&cfg, decode_cluster_kernel<false, false>, p);
}

DecodeParams cache_params(const Cache& c, int32_t layer, const void* q, void* out, int32_t group,
                          float scale_log2) {
  DecodeParams p = {};
  p.state_ready = (c.last_full_tiled && c.last_layer != layer) ? 1 : 0;
  p.pool = c.pool;
  p.page_table = c.page_table + (int64_t)layer * c.heads * c.max_pages;
  p.counts = c.counts_at(layer, c.lengths[layer]);
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
  return p;
}

}  // namespace

cudaError_t launch_decode_tiled(const Cache& c, int32_t layer, const void* q, void* out,
                                int32_t group, float scale_log2, bool zero_first,
                                cudaStream_t stream) {
  DecodeParams p = cache_params(c, layer, q, out, group, scale_log2);
  p.zero_first = zero_first ? 1 : 0;
  const int cs = decode_cluster_size(c, group, c.lengths[layer]);
  if (cs > 0) {
    p.state_ready = 0;
    p.head_flags = c.head_flags + (int64_t)layer * c.heads;
    p.flag_expect = c.flag_valid[layer] ? c.flag_seq[layer] : 0u;
    p.flag_wait_ns = c.flag_test_layer == layer ? c.flag_test_wait_ns : 0;
    return launch_cluster(p, cs, stream, false, c.fp8());
  }
  return launch_tiled(p, c.num_sms, c.ctas_per_sm, stream, true, false, c.fp8());
}

bool append_decode_fusable(const Cache& c) {
  return c.decode_kernel != DMS_DECODE_SIMPLE && c.heads <= kMaxHeadsFused && c.ctas_per_sm < 2;
}

bool tiled_one_cta_per_sm(const Cache& c) { return c.ctas_per_sm < 2; }

// Single-token append of position lengths[layer] fused with the decode (requires
// append_decode_fusable).
cudaError_t launch_append_decode(const Cache& c, int32_t layer, const void* k, const void* v,
                                 const void* logit, int64_t logit_stride, const void* q, void* out,
                                 int32_t group, float scale_log2, bool zero_first,
                                 cudaStream_t stream) {
  const int64_t t0 = c.lengths[layer];
  DecodeParams p = cache_params(c, layer, q, out, group, scale_log2);
  p.zero_first = zero_first ? 1 : 0;
  p.k_new = static_cast<const uint16_t*>(k);
  p.v_new = static_cast<const uint16_t*>(v);
  p.logit_new = static_cast<const uint16_t*>(logit);
  p.logit_stride = logit_stride;
  p.counts_next = c.counts_at(layer, t0 + 1);
  p.ring = c.rings + (int64_t)layer * c.heads * c.ring_len;
  p.pos = c.pos;
  p.j = t0;
  p.window = c.window;
  p.decider = c.decider();
  p.pool_pages = c.pool_pages;
  p.ring_len = c.ring_len;
  const int cs = decode_cluster_size(c, group, t0 + 1);
  if (cs > 0) {
    p.state_ready = 0;
    p.head_flags = c.head_flags + (int64_t)layer * c.heads;
    p.flag_expect = c.flag_valid[layer] ? c.flag_seq[layer] : 0u;
    p.flag_publish = next_flag_seq(c.flag_seq[layer]);
    p.flag_wait_ns = c.flag_test_layer == layer ? c.flag_test_wait_ns : 0;
    return launch_cluster(p, cs, stream, true, c.fp8());
  }
  return launch_tiled(p, c.num_sms, 1, stream, true, true, c.fp8());
}

cudaError_t launch_decode_simple(const Cache& c, int32_t layer, const void* q, void* out,
                                 int32_t group, float scale, bool zero_first, cudaStream_t stream) {
  decode_simple_kernel<<<c.heads, 128, 0, stream>>>(
      c.pool, c.page_table + (int64_t)layer * c.heads * c.max_pages,
      c.counts_at(layer, c.lengths[layer]), static_cast<const __nv_bfloat16*>(q),
      static_cast<__nv_bfloat16*>(out), c.kv_heads, group, c.max_pages, scale, zero_first ? 1 : 0);
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

namespace {

// One-time set-up per device, with that device current: the device address of the
// scratch array (the host-side name is only a stand-in), the kernel's shared-memory
// limit and the SM count.  Returns false on a CUDA error.
bool static_device_state(StaticDeviceState* out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) {
    cudaGetLastError();
    return false;
  }
  std::lock_guard<std::mutex> lock(g_static_mu);
  StaticDeviceState& s = g_static_state[dev];
  if (!s.ready) {
    void* ptr = nullptr;
    if (cudaGetSymbolAddress(&ptr, g_decode_scratch) != cudaSuccess) {
      cudaGetLastError();
      return false;
    }
    int sms = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
        dms::prepare_decode(dms::Cache()) != cudaSuccess) {
      cudaGetLastError();
      return false;
    }
    s.scratch = static_cast<float*>(ptr);
    s.num_sms = sms;
    s.ready = true;
  }
  *out = s;
  return true;
}

int32_t* static_counters(const StaticDeviceState& st) {
  return reinterpret_cast<int32_t*>(st.scratch + (size_t)kStaticRecords * dms::kPieceFloats);
}
int32_t* static_ctrl(const StaticDeviceState& st) { return static_counters(st) + kStaticCounters; }

}  // namespace

extern "C" dms_status dms_decode_attention_paged_noalloc(
    const void* pool, const int32_t* page_table, const int32_t* counts, int32_t batch,
    int32_t kv_heads, int32_t max_pages, const void* q, void* out, int32_t gqa_group,
    float sm_scale, void* stream) {
  using namespace dms;
  auto misaligned = [](const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) != 0; };
  if (pool == nullptr || page_table == nullptr || counts == nullptr || q == nullptr ||
      out == nullptr || misaligned(pool, 16) || misaligned(q, 16) || misaligned(out, 16) ||
      misaligned(page_table, 4) || misaligned(counts, 4) || batch < 1 || kv_heads < 1 ||
      max_pages < 1 || gqa_group < 1 || gqa_group > kMaxGroup || !(sm_scale == sm_scale))
    return DMS_ERR_INVALID_ARGUMENT;
  const int64_t heads = (int64_t)batch * kv_heads;
  if (heads > kMaxHeads) return DMS_ERR_INVALID_ARGUMENT;

  StaticDeviceState st;
  if (!static_device_state(&st)) return DMS_ERR_CUDA;
  const int grid = st.num_sms;
  if (grid + heads > kStaticRecords) return DMS_ERR_CAPACITY;  // scratch too small for this batch

  int32_t* counters = static_counters(st);
  int32_t* ctrl = static_ctrl(st);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // The array keeps whatever the previous call left: the arrival counters and the
  // error word must start at zero.
  if (cudaMemsetAsync(counters, 0, sizeof(int32_t) * (size_t)(kStaticCounters + kStaticCtrl), s) !=
      cudaSuccess)
    return DMS_ERR_CUDA;

  DecodeParams p = {};
  p.pool = static_cast<uint8_t*>(const_cast<void*>(pool));
  p.page_table = const_cast<int32_t*>(page_table);
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
  return launch_tiled(p, grid, 1, s, false, false) == cudaSuccess ? DMS_OK : DMS_ERR_CUDA;
}

extern "C" dms_status dms_decode_noalloc_device_error(void* stream, dms_status* out) {
  if (out == nullptr) return DMS_ERR_INVALID_ARGUMENT;
  StaticDeviceState st;
  if (!static_device_state(&st)) return DMS_ERR_CUDA;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int32_t word = 0;  // the error word, read into host (stack) memory: nothing is allocated
  if (cudaMemcpyAsync(&word, static_ctrl(st) + dms::kCtrlError, sizeof(word),
                      cudaMemcpyDeviceToHost, s) != cudaSuccess ||
      cudaStreamSynchronize(s) != cudaSuccess) {
    cudaGetLastError();
    return DMS_ERR_CUDA;
  }
  *out = static_cast<dms_status>(word);
  return DMS_OK;
}

extern "C" dms_status dms_selftest_noalloc_timeout(int64_t limit_ns, void* stream) {
  if (limit_ns < 1000 || limit_ns > 10000000000LL) return DMS_ERR_INVALID_ARGUMENT;
  StaticDeviceState st;
  if (!static_device_state(&st)) return DMS_ERR_CUDA;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int32_t* ctrl = static_ctrl(st);
  // A barrier that nothing completes: the bounded wait gives up after limit_ns and
  // records DMS_ERR_TIMEOUT in the error word the allocation-free decode uses.
  if (cudaMemsetAsync(ctrl, 0, sizeof(int32_t) * (size_t)kStaticCtrl, s) != cudaSuccess ||
      dms::launch_bounded_wait_probe(0, limit_ns, ctrl, s) != cudaSuccess ||
      cudaStreamSynchronize(s) != cudaSuccess) {
    cudaGetLastError();
    return DMS_ERR_CUDA;
  }
  return DMS_OK;
}
