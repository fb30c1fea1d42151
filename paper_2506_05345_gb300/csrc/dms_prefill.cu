// Sparse DMS prefill attention (arXiv 2506.05345, Sec. 3.1 / Fig. 1b for the mask, Sec. 3.2:
// the eviction sparsity is also used in prefill).  For a prompt of P tokens, query j of
// every query head attends, with plain softmax, to the keys i <= j of its KV head with
// alpha_i = 0 or j - i <= w (alpha_i = [bf16 decision logit of token i > 0]).
//
// The visible keys of a tile of 128 consecutive queries [j0, j0 + 128) split into two
// disjoint sets, each a contiguous run of rows once the prompt is laid out per KV head:
//   * retained keys: alpha_i = 0 and i < j - w.  In the per-head list of the alpha = 0
//     tokens in position order (the compacted list), they are a prefix: the first
//     before[jmax - w] entries, where before[x] counts the alpha = 0 tokens at positions
//     below x and jmax is the tile's last query.  Row j masks the entries at positions
//     >= j - w;
//   * window keys: j - w <= i <= j, a band of dense rows [j0 - w, jmax] (start rounded
//     down to a multiple of 8), masked per row.
// A pre-pass (two small kernels) lays every KV head out contiguously: dense K and V rows,
// the compacted K and V rows, the compacted rows' positions and the prefix counts, with
// each 256-byte row's 16-byte chunks permuted (chunk ^ (row & 7)) so that 1-D bulk copies
// land in shared memory conflict-free for ldmatrix.
//
// Attention kernel: one CTA per (query head, 128-query tile), heaviest tiles (latest
// queries) first.  A producer warp streams 64-key tiles (K, V and, for retained tiles,
// the keys' positions) into a 3-stage shared-memory ring with bulk copies on mbarriers;
// eight consumer warps own 16 queries each: S = Q K^T and O += P V with mma.sync
// m16n8k16 (bf16 in, fp32 accumulate), fp32 online softmax in the exp2 domain, P reused
// from the S accumulators as the A operand.  Each warp stages its queries in shared memory
// once and reloads their fragments with ldmatrix per tile (nine warps leave ~168
// registers per thread; holding Q in registers would spill).
#include <cuda.h>  // tensor-map types only; the encoder is reached through the runtime
#include <math.h>

#include <atomic>
#include <mutex>

#include "dms_internal.cuh"
#include "dms_ptx.cuh"

namespace dms {
namespace {

constexpr int kPfRows = 128;                                  // queries per CTA
constexpr int kPfWarps = kPfRows / 16;                        // consumer warps
constexpr int kPfKeys = 64;                                   // keys per tile
constexpr int kPfStages = 3;
constexpr int kPfThreads = (kPfWarps + 1) * 32;               // + producer warp
constexpr int kPfTileBytes = kPfKeys * kRowBytes;             // 16 KiB
constexpr int kPfStageBytes = 2 * kPfTileBytes + kPfKeys * 4;  // K, V, key positions
constexpr int kPfQBytes = kPfRows * kRowBytes;                // the CTA's queries, 32 KiB
constexpr int kPfSmemBytes = kPfStages * kPfStageBytes + kPfQBytes + 2 * kPfStages * 8 + 16;
constexpr int kPfChunk = 1024;                                // tokens per pre-pass block
constexpr int kPfPackThreads = 256;
constexpr int kPfPosPad = kPfKeys;  // compacted positions padded so whole tiles copy

// Row stride (int32 entries) of a head's compacted positions: whole 64-entry tiles copy
// from any tile start, and every row starts on a 16-byte boundary (bulk-copy sources).
__host__ __device__ __forceinline__ int64_t pc_stride(int64_t P) { return (P + kPfPosPad + 3) & ~(int64_t)3; }

// Workspace regions (byte offsets, each 256-byte aligned).  H = batch * kv_heads.
struct PfLayout {
  size_t err, kd, vd, kc, vc, pc, before, cc, total;
};

size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

PfLayout pf_layout(int64_t H, int64_t P) {
  PfLayout L;
  const int64_t nch = (P + kPfChunk - 1) / kPfChunk;
  size_t o = 0;
  L.err = o; o = align256(o + 64);
  L.kd = o; o = align256(o + (size_t)H * P * kRowBytes);
  L.vd = o; o = align256(o + (size_t)H * P * kRowBytes);
  L.kc = o; o = align256(o + (size_t)H * P * kRowBytes);
  L.vc = o; o = align256(o + (size_t)H * P * kRowBytes);
  L.pc = o; o = align256(o + (size_t)H * pc_stride(P) * 4);
  L.before = o; o = align256(o + (size_t)H * (P + 1) * 4);
  L.cc = o; o = align256(o + (size_t)H * nch * 4);
  L.total = o;
  return L;
}

struct PackParams {
  const uint16_t* k;         // [B, P, Hkv, 128]
  const uint16_t* v;
  const uint16_t* logit;     // decision logit of (b, i, h) at logit[((b P + i) Hkv + h) stride]
  int64_t logit_stride;
  int64_t decider;           // token i is evicted by the decision of token i + decider
  uint8_t* kd;               // [H][2 d-halves][P][128 B] permuted half-rows
  uint8_t* vd;
  uint8_t* kc;               // [H][2][P][128 B]: the alpha = 0 tokens, position order
  uint8_t* vc;
  int32_t* pc;               // [H][pc_stride(P)] positions of the compacted rows
  int32_t* before;           // [H][P + 1] alpha = 0 tokens at positions below i
  int32_t* cc;               // [H][nch] alpha = 0 tokens per chunk
  int32_t P, kv_heads, nch;
};

// Byte offset of logical 16-byte chunk `chunk` (0..7) inside the 128-byte half-row `row`
// (the row's own offset is added by the caller in 64-bit arithmetic).
__device__ __forceinline__ uint32_t chunk_in_row(int64_t row, int chunk) {
  return (uint32_t)((chunk ^ (int)(row & 7)) << 4);
}

// Byte offset of logical chunk c (0..15, head_dim 8c .. 8c + 7) of row r inside a staged
// 64-row tile stored as two 8 KiB d-halves [half][row][128 B].
__device__ __forceinline__ uint32_t tile_off(uint32_t r, uint32_t c) {
  return (c >> 3) * (kPfKeys * 128u) + r * 128u + (((c & 7u) ^ (r & 7u)) << 4);
}

// Token i stays visible outside the window iff the decision that evicts it is 0: its
// own (delayed eviction) or that of token i + decider (immediate-eviction ablation).  A
// token whose deciding token lies past the prompt is inside the window of every query
// of the prompt, so it is never needed in the compacted list.
__device__ __forceinline__ bool keep_token(const PackParams& p, int b, int hk, int i) {
  const int64_t d = i + p.decider;
  return d < p.P &&
         decision_from_bf16(p.logit[(((int64_t)b * p.P + d) * p.kv_heads + hk) * p.logit_stride]) == 0u;
}

// Alpha = 0 tokens of each (head, chunk).
__global__ void __launch_bounds__(kPfPackThreads) prefill_count_kernel(const PackParams p) {
  const int ch = blockIdx.x, head = blockIdx.y;
  const int b = head / p.kv_heads, hk = head - b * p.kv_heads;
  const int i_end = min(p.P, (ch + 1) * kPfChunk);
  int cnt = 0;
  for (int i = ch * kPfChunk + threadIdx.x; i < i_end; i += kPfPackThreads)
    cnt += keep_token(p, b, hk, i) ? 1 : 0;
  __shared__ int s_sum[kPfPackThreads / 32];
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) cnt += __shfl_xor_sync(0xffffffffu, cnt, off);
  if ((threadIdx.x & 31) == 0) s_sum[threadIdx.x >> 5] = cnt;
  __syncthreads();
  if (threadIdx.x == 0) {
    int t = 0;
    for (int w = 0; w < kPfPackThreads / 32; ++w) t += s_sum[w];
    p.cc[(int64_t)head * p.nch + ch] = t;
  }
}

// Lays out one (head, chunk): dense rows, compacted rows and their positions, and the
// prefix counts.  Thread t owns tokens 4t .. 4t + 3 of the chunk for the scan; the
// warps then move the rows, one 512-byte K + V row pair per warp step.
__global__ void __launch_bounds__(kPfPackThreads) prefill_pack_kernel(const PackParams p) {
  const int ch = blockIdx.x, head = blockIdx.y;
  const int b = head / p.kv_heads, hk = head - b * p.kv_heads;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int i0 = ch * kPfChunk, n = min(kPfChunk, p.P - i0);
  __shared__ int s_idx[kPfChunk];  // compacted index of each token, or -1 when evicted
  __shared__ int s_warp[kPfPackThreads / 32];
  __shared__ int s_base;
  // alpha = 0 tokens of the earlier chunks of this head
  int base = 0;
  for (int c = tid; c < ch; c += kPfPackThreads) base += p.cc[(int64_t)head * p.nch + c];
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) base += __shfl_xor_sync(0xffffffffu, base, off);
  if (lane == 0) s_warp[warp] = base;
  __syncthreads();
  if (tid == 0) {
    int t = 0;
    for (int w = 0; w < kPfPackThreads / 32; ++w) t += s_warp[w];
    s_base = t;
  }
  __syncthreads();
  base = s_base;
  // exclusive scan of the keep flags over the chunk
  int f[4], local = 0;
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    const int i = 4 * tid + e;
    f[e] = (i < n && keep_token(p, b, hk, i0 + i)) ? 1 : 0;
    local += f[e];
  }
  int x = local;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, off);
    if (lane >= off) x += y;
  }
  __syncthreads();  // s_warp reuse
  if (lane == 31) s_warp[warp] = x;
  __syncthreads();
  int run = base + x - local;
  for (int w = 0; w < warp; ++w) run += s_warp[w];
  int32_t* before = p.before + (int64_t)head * (p.P + 1);
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    const int i = 4 * tid + e;
    if (i < n) {
      before[i0 + i] = run;
      s_idx[i] = f[e] ? run : -1;
      if (i0 + i == p.P - 1) before[p.P] = run + f[e];
    }
    run += f[e];
  }
  __syncthreads();
  // rows: lanes 0-15 move K's sixteen 16-byte chunks, lanes 16-31 V's; chunk c goes to
  // d-half c / 8 of the row
  const int kv = lane >> 4, chunk = lane & 15, dh = chunk >> 3, c8 = chunk & 7;
  const uint16_t* src_base = kv ? p.v : p.k;
  uint8_t* dense = kv ? p.vd : p.kd;
  uint8_t* comp = kv ? p.vc : p.kc;
  const int64_t hrow = ((int64_t)head * 2 + dh) * p.P;  // this d-half of this head
  for (int i = warp; i < n; i += kPfPackThreads / 32) {
    const int pos = i0 + i;
    const uint4 val = *reinterpret_cast<const uint4*>(
        src_base + (((int64_t)b * p.P + pos) * p.kv_heads + hk) * kHeadDim + chunk * 8);
    *reinterpret_cast<uint4*>(dense + (hrow + pos) * 128 + chunk_in_row(pos, c8)) = val;
    const int c = s_idx[i];
    if (c >= 0) {
      *reinterpret_cast<uint4*>(comp + (hrow + c) * 128 + chunk_in_row(c, c8)) = val;
      if (lane == 0) p.pc[(int64_t)head * pc_stride(p.P) + c] = pos;
    }
  }
}

// Rows [r0, r0 + rows) of one head's K and V (two d-halves each) into a stage laid out as
// K [2][64][128 B] then V [2][64][128 B].
__device__ __forceinline__ void stage_tile(uint8_t* st, const uint8_t* k, const uint8_t* v,
                                           int64_t head, int P, int r0, int rows, uint64_t* bar) {
  const uint32_t bytes = (uint32_t)rows * 128u;
#pragma unroll
  for (int dh = 0; dh < 2; ++dh) {
    const int64_t row = (head * 2 + dh) * P + r0;
    bulk_copy_g2s(st + dh * (kPfKeys * 128), k + row * 128, bytes, bar);
    bulk_copy_g2s(st + kPfTileBytes + dh * (kPfKeys * 128), v + row * 128, bytes, bar);
  }
}

struct PrefillParams {
  const __nv_bfloat16* q;    // [B, P, Hq, 128]
  __nv_bfloat16* out;        // [B, P, Hq, 128]
  const uint8_t* kd;
  const uint8_t* vd;
  const uint8_t* kc;
  const uint8_t* vc;
  const int32_t* pc;
  const int32_t* before;
  int32_t* err;              // sticky error word (bounded waits)
  int32_t P, kv_heads, group, window, zero_first, n_qtiles, n_qheads, batch;
  float scale_log2;
};

__global__ void __launch_bounds__(kPfThreads, 1) prefill_attn_kernel(const PrefillParams p) {
  extern __shared__ __align__(128) uint8_t smem[];
  uint8_t* sq = smem + kPfStages * kPfStageBytes;  // [128 rows][256 B], permuted chunks
  uint64_t* full_bar = reinterpret_cast<uint64_t*>(sq + kPfQBytes);
  uint64_t* empty_bar = full_bar + kPfStages;
  volatile int* abort_flag = reinterpret_cast<volatile int*>(empty_bar + kPfStages);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int Hq = p.kv_heads * p.group;
  const int tile_rank = blockIdx.x / p.n_qheads;
  const int qt = p.n_qtiles - 1 - tile_rank;  // latest (heaviest) query tiles first
  const int qh = blockIdx.x - tile_rank * p.n_qheads;
  const int b = qh / Hq, hq = qh - b * Hq, hk = hq / p.group;
  const int64_t head = (int64_t)b * p.kv_heads + hk;
  const int P = p.P, w = p.window;
  const int j0 = qt * kPfRows;
  const int jmax = min(j0 + kPfRows, P) - 1;
  // retained keys: the first nc compacted rows; window keys: dense rows [bs, jmax]
  const int nc = (jmax - w > 0) ? p.before[head * (P + 1) + (jmax - w)] : 0;
  const int bs = max(0, j0 - w) & ~7;
  const int n_ct = (nc + kPfKeys - 1) / kPfKeys;
  const int n_tiles = n_ct + (jmax + 1 - bs + kPfKeys - 1) / kPfKeys;

  if (tid == 0) {
    *abort_flag = 0;
    for (int s = 0; s < kPfStages; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], kPfWarps);
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();

  if (warp == kPfWarps) {
    // ================================================================ producer warp
    if (lane == 0) {
      for (int t = 0; t < n_tiles; ++t) {
        const int s = t % kPfStages, use = t / kPfStages;
        if (use > 0) mbar_wait(&empty_bar[s], (use - 1) & 1, abort_flag, p.err);
        uint8_t* st = smem + s * kPfStageBytes;
        if (t < n_ct) {
          const int r0 = t * kPfKeys, rows = min(kPfKeys, nc - r0);
          mbar_arrive_expect_tx(&full_bar[s], 2 * (uint32_t)rows * kRowBytes + kPfKeys * 4);
          stage_tile(st, p.kc, p.vc, head, P, r0, rows, &full_bar[s]);
          bulk_copy_g2s(st + 2 * kPfTileBytes, p.pc + head * pc_stride(P) + r0, kPfKeys * 4,
                        &full_bar[s]);
        } else {
          const int r0 = bs + (t - n_ct) * kPfKeys, rows = min(kPfKeys, jmax + 1 - r0);
          mbar_arrive_expect_tx(&full_bar[s], 2 * (uint32_t)rows * kRowBytes);
          stage_tile(st, p.kd, p.vd, head, P, r0, rows, &full_bar[s]);
        }
      }
      // Drain: do not leave while a bulk copy may still be writing shared memory.
      for (int s = 0; s < kPfStages && s < n_tiles; ++s) {
        const int last_t = s + ((n_tiles - 1 - s) / kPfStages) * kPfStages;
        mbar_wait(&full_bar[s], (last_t / kPfStages) & 1, abort_flag, p.err);
      }
    }
    return;
  }

  // ================================================================ consumer warps
  const int g = lane >> 2, c4 = lane & 3, mi = lane >> 3;
  const int r_lo = j0 + 16 * warp + g, r_hi = r_lo + 8;  // this lane's two query rows
  // This warp's 16 queries into shared memory (permuted chunks, read back with ldmatrix);
  // App. B: element 0 of a group's first query head carries the decision, not attention.
  {
    const bool zero = p.zero_first && hq % p.group == 0;
#pragma unroll
    for (int it = 0; it < 8; ++it) {
      const int idx = it * 32 + lane, row = idx >> 4, chunk = idx & 15;
      const int j = j0 + 16 * warp + row;
      uint4 val = make_uint4(0u, 0u, 0u, 0u);
      if (j < P)
        val = *reinterpret_cast<const uint4*>(p.q + (((int64_t)b * P + j) * Hq + hq) * kHeadDim +
                                              chunk * 8);
      if (zero && chunk == 0) val.x &= 0xffff0000u;
      *reinterpret_cast<uint4*>(sq + (16 * warp + row) * kRowBytes + chunk_in_row(row, chunk)) = val;
    }
    __syncwarp();
  }
  const uint32_t qbase = smem_addr(sq + 16 * warp * kRowBytes);
  float o[16][4];
#pragma unroll
  for (int nt = 0; nt < 16; ++nt) o[nt][0] = o[nt][1] = o[nt][2] = o[nt][3] = 0.f;
  float m_lo = -INFINITY, m_hi = -INFINITY, l_lo = 0.f, l_hi = 0.f;

  for (int t = 0; t < n_tiles; ++t) {
    const int s = t % kPfStages, use = t / kPfStages;
    const bool retained = t < n_ct;
    const int r0 = retained ? t * kPfKeys : bs + (t - n_ct) * kPfKeys;
    const int rows = retained ? min(kPfKeys, nc - r0) : min(kPfKeys, jmax + 1 - r0);
    const uint8_t* st = smem + s * kPfStageBytes;
    mbar_wait(&full_bar[s], use & 1, abort_flag, p.err);

    // ---- S = Q K^T (16 x 64): 8 n-tiles of 8 keys, 8 k-steps of 16 head_dim
    float sc[8][4];
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) sc[nt][0] = sc[nt][1] = sc[nt][2] = sc[nt][3] = 0.f;
    {
      const uint32_t kbase = smem_addr(st);
      const uint32_t qrow = (uint32_t)((mi & 1) * 8 + (lane & 7));
#pragma unroll
      for (int kk = 0; kk < 8; ++kk) {
        uint32_t qa[4];  // A-fragment: rows 0-7 / 8-15 of the warp, d 16 kk .. 16 kk + 15
        ldsm_x4(qbase + swizzled_offset(qrow, (uint32_t)(2 * kk + (mi >> 1))), qa[0], qa[1], qa[2],
                qa[3]);
#pragma unroll
        for (int np = 0; np < 4; ++np) {
          const uint32_t row = (uint32_t)(16 * np + (mi >> 1) * 8 + (lane & 7));
          uint32_t b0, b1, b2, b3;
          ldsm_x4(kbase + tile_off(row, (uint32_t)(2 * kk + (mi & 1))), b0, b1, b2, b3);
          mma_bf16_16816(sc[2 * np], qa, b0, b1);
          mma_bf16_16816(sc[2 * np + 1], qa, b2, b3);
        }
      }
    }
    // ---- mask (retained: position < j - w; window: j - w <= position <= j), online softmax
    const int32_t* spos = reinterpret_cast<const int32_t*>(st + 2 * kPfTileBytes);
    float mx_lo = -INFINITY, mx_hi = -INFINITY;
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int kidx = 8 * nt + 2 * c4 + e;
        const bool valid = kidx < rows;
        const int pos = retained ? (valid ? spos[kidx] : 0) : r0 + kidx;
        const bool vis_lo = valid && (retained ? pos < r_lo - w : (pos >= r_lo - w && pos <= r_lo));
        const bool vis_hi = valid && (retained ? pos < r_hi - w : (pos >= r_hi - w && pos <= r_hi));
        sc[nt][e] = vis_lo ? sc[nt][e] * p.scale_log2 : -INFINITY;
        sc[nt][2 + e] = vis_hi ? sc[nt][2 + e] * p.scale_log2 : -INFINITY;
        mx_lo = fmaxf(mx_lo, sc[nt][e]);
        mx_hi = fmaxf(mx_hi, sc[nt][2 + e]);
      }
    }
#pragma unroll
    for (int off = 1; off < 4; off <<= 1) {
      mx_lo = fmaxf(mx_lo, __shfl_xor_sync(0xffffffffu, mx_lo, off));
      mx_hi = fmaxf(mx_hi, __shfl_xor_sync(0xffffffffu, mx_hi, off));
    }
    const float mn_lo = fmaxf(m_lo, mx_lo), mn_hi = fmaxf(m_hi, mx_hi);
    // a row that has seen no visible key yet keeps a zero base (no -inf - -inf)
    const float base_lo = mn_lo == -INFINITY ? 0.f : mn_lo;
    const float base_hi = mn_hi == -INFINITY ? 0.f : mn_hi;
    const float corr_lo = exp2f(m_lo - base_lo), corr_hi = exp2f(m_hi - base_hi);
    m_lo = mn_lo;
    m_hi = mn_hi;
    float sum_lo = 0.f, sum_hi = 0.f;
    uint32_t pa[4][4];  // P A-fragments of the four 16-key k-steps
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
      const float p0 = exp2f(sc[nt][0] - base_lo), p1 = exp2f(sc[nt][1] - base_lo);
      const float p2 = exp2f(sc[nt][2] - base_hi), p3 = exp2f(sc[nt][3] - base_hi);
      sum_lo += p0 + p1;
      sum_hi += p2 + p3;
      pa[nt >> 1][(nt & 1) * 2 + 0] = pack_bf16x2(p0, p1);
      pa[nt >> 1][(nt & 1) * 2 + 1] = pack_bf16x2(p2, p3);
    }
    l_lo = l_lo * corr_lo + sum_lo;
    l_hi = l_hi * corr_hi + sum_hi;
#pragma unroll
    for (int nt = 0; nt < 16; ++nt) {
      o[nt][0] *= corr_lo;
      o[nt][1] *= corr_lo;
      o[nt][2] *= corr_hi;
      o[nt][3] *= corr_hi;
    }
    // ---- O += P V (16 x 128): 4 k-steps of 16 keys, 16 n-tiles of 8 head_dim
    {
      const uint32_t vbase = smem_addr(st + kPfTileBytes);
#pragma unroll
      for (int kt = 0; kt < 4; ++kt) {
        // stale rows past the tile's valid keys must not reach the tensor cores (0 * NaN)
        const int tk = 16 * kt + 2 * c4;
        const uint32_t mk0 = (tk < rows ? 0x0000ffffu : 0u) | (tk + 1 < rows ? 0xffff0000u : 0u);
        const uint32_t mk1 = (tk + 8 < rows ? 0x0000ffffu : 0u) | (tk + 9 < rows ? 0xffff0000u : 0u);
        const uint32_t row = (uint32_t)(16 * kt + (mi & 1) * 8 + (lane & 7));
#pragma unroll
        for (int dp = 0; dp < 8; ++dp) {
          uint32_t b0, b1, b2, b3;
          ldsm_x4_trans(vbase + tile_off(row, (uint32_t)(2 * dp + (mi >> 1))), b0, b1, b2, b3);
          b0 &= mk0;
          b1 &= mk1;
          b2 &= mk0;
          b3 &= mk1;
          mma_bf16_16816(o[2 * dp], pa[kt], b0, b1);
          mma_bf16_16816(o[2 * dp + 1], pa[kt], b2, b3);
        }
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&empty_bar[s]);
  }

  // ---- normalise and store (rows past the prompt are not written)
#pragma unroll
  for (int off = 1; off < 4; off <<= 1) {
    l_lo += __shfl_xor_sync(0xffffffffu, l_lo, off);
    l_hi += __shfl_xor_sync(0xffffffffu, l_hi, off);
  }
  const float inv_lo = l_lo > 0.f ? 1.f / l_lo : 0.f, inv_hi = l_hi > 0.f ? 1.f / l_hi : 0.f;
  __nv_bfloat16* o_lo = p.out + (((int64_t)b * P + r_lo) * Hq + hq) * kHeadDim;
  __nv_bfloat16* o_hi = p.out + (((int64_t)b * P + r_hi) * Hq + hq) * kHeadDim;
#pragma unroll
  for (int nt = 0; nt < 16; ++nt) {
    const int d = 8 * nt + 2 * c4;
    if (r_lo < P)
      *reinterpret_cast<uint32_t*>(o_lo + d) = pack_bf16x2(o[nt][0] * inv_lo, o[nt][1] * inv_lo);
    if (r_hi < P)
      *reinterpret_cast<uint32_t*>(o_hi + d) = pack_bf16x2(o[nt][2] * inv_hi, o[nt][3] * inv_hi);
  }
}

// ============================================================================ tcgen05 kernel
// The same attention on the 5th-generation tensor cores: a persistent kernel, one CTA per SM,
// each walking work units (one query head x one 128-query tile; heaviest tiles first, and
// consecutive units are the query heads of one KV head, so their K / V tiles are read from L2
// close together in time) with a static stride.  Key tiles hold 128 keys, so every MMA is
// M 128 x N 128 x K 16 (on this tensor core an N 64 MMA costs 3/4 of the time of an N 128 one
// for half its work).
// 384 threads: warp 0 stages the K tiles (3-slot ring) and V tiles (2-slot ring) of the units
// with bulk copies, K two tiles ahead of V; warp 2 moves Q in and O out (tensor-map copies, 128-byte swizzle: a Q tile
// lands in the MMA operand layout; two Q buffers, each also staging its unit's O); warps 4-11
// run the softmax as two sets of four warps, one thread per query row in each (a warp reaches
// only TMEM lanes 32 (warp % 4) ..).  Set s takes the key tiles of one parity: tile tau of the
// CTA goes to set tau % 2, so two tiles are in the softmax at once while a row's max and sum
// stay in a thread.  Warps 1 and 3 issue the MMAs of sets 0 and 1: the two streams share no
// tensor memory, so the tensor cores interleave them and one set's waits do not stall the
// other's products (warp 1 also owns the tensor memory).
// Tensor memory (512 columns): per set an O accumulator (128 fp32 columns, at 128 s) and an S
// buffer (at 256 + 128 s); the scores of a tile are computed while the other set works on the
// previous one.  A set overwrites its S in place with P = 2^(S scale - m) as packed bf16 pairs
// (keys 2c, 2c + 1 in column c), the A operand of O_s += P V straight from tensor memory;
// S(tau + 2) reuses the buffer after O += P(tau) V(tau), in issue order.  The reference max m
// of a row in a set moves only when its tile max exceeds m by more than 2^8; the thread then
// rescales its row of O_s before its P-ready arrival (the previous product into O_s completed
// before S(tau), which was issued after it).
// A unit ends with both sets: each publishes its row's (m, l), combines the two accumulators
// for one d-half, O = (O_0 2^(m_0 - M) + O_1 2^(m_1 - M)) / (l_0 2^(m_0 - M) + l_1 2^(m_1 - M)),
// M = max(m_0, m_1), and stages it as bf16 in the unit's Q buffer (every score of the unit is
// done); warp 2 stores the tile (rows past the prompt fall outside the tensor map) and then
// loads the Q two units on into the buffer.  The set that did not take the unit's last tile
// first writes the P of its next tile, so the tensor cores wait only for the accumulators to
// be read out before the next unit's products.
// Visibility: the retained keys query j sees are the first before[j - w] compacted rows, so
// one count masks a retained tile; window keys are a contiguous run of the band.  Stale rows
// of a partial V tile are zeroed before its copy (P is 0 there, but 0 * NaN is not).  Each
// role loads the counts of its next unit one unit ahead.
// Shared-memory operands use the 128-byte-swizzled layout: rows of two 128-byte d-halves,
// 16-byte chunks permuted by (row & 7), 1 KiB-aligned bases; Q and K are K-major, V is
// MN-major (head_dim contiguous).
constexpr int kTcSets = 2;                               // softmax sets (tile parities)
constexpr int kTcSoftmaxWarps = 4 * kTcSets;             // one thread per query row per set
constexpr int kTcThreads = (4 + kTcSoftmaxWarps) * 32;   // 384
constexpr int kTcQWarp = 2;
constexpr int kTcMmaWarp1 = 3;                           // MMAs of set 1 (set 0: warp 1)
constexpr int kTcSoftmax0 = 4;                           // first softmax warp
// Kernel of the plain entry points (the faster of the two as measured).
constexpr int32_t kPrefillDefaultKernel = DMS_PREFILL_TCGEN05;
constexpr int kTcKeys = 128;                             // keys per tile
constexpr int kTcKSlots = 3;                             // K ring
constexpr int kTcVSlots = 2;                             // V ring
constexpr int kTcHalfBytes = kTcKeys * 128;              // one d-half of a tile, 16 KiB
constexpr int kTcTileBytes = 2 * kTcHalfBytes;           // [2 d-halves][128 rows][128 B]
constexpr int kTcQBytes = kPfRows * kRowBytes;           // Q (then O), same layout
constexpr int kTcOffV = kTcKSlots * kTcTileBytes;
constexpr int kTcOffQ = kTcOffV + kTcVSlots * kTcTileBytes;        // two Q buffers
constexpr int kTcOffBar = kTcOffQ + 2 * kTcQBytes;                 // barrier block
constexpr int kTcOffX = kTcOffBar + 256;                           // (m, l) exchange
constexpr int kTcSmemBytes = kTcOffX + kTcSets * kPfRows * 8;      // [set][row] float2
// The dynamic shared memory base is 1 KiB aligned (no static shared memory precedes it);
// the kernel checks this and reports DMS_ERR_CUDA otherwise.
static_assert(kTcSmemBytes <= 227 * 1024, "tcgen05 prefill shared memory");
constexpr uint32_t kTcCols = 512;
constexpr uint32_t kTcColS = 256;  // S buffers at 256, 384; O accumulators at 0, 128
constexpr float kTcRescale = 8.f;  // log2 of the largest growth of P before O is rescaled

// Barriers.  Tiles are counted globally over the CTA's units (tau), units by their ordinal
// (un).  s_full[i], p_full[i] and o_full[i] serve set i (the tiles with tau % 2 = i);
// q_full[i], q_ready[i] and o_staged[i] the units with un % 2 = i (Q buffer i); o_full[i] and
// o_free complete once per unit.  Every waiter is at most one phase behind the barrier it waits on (parity waits need
// that); the waits say why.
struct TcBars {
  uint64_t k_full[kTcKSlots], k_empty[kTcKSlots];
  uint64_t v_full[kTcVSlots], v_empty[kTcVSlots];
  uint64_t q_full[2];    // Q landed
  uint64_t q_ready[2];   // Q patched (borrowed decisions only)
  uint64_t o_staged[2];  // one arrival per softmax warp: the unit's O staged in its Q buffer
  uint64_t s_full[2];    // MMA commit: scores ready
  uint64_t p_full[2];    // one arrival per warp of the set: P written (and O rescaled)
  uint64_t o_full[2];    // MMA commit: every product of the unit into O_i done
  uint64_t o_free;       // one arrival per softmax warp: both accumulators read out
  uint64_t mma_done[2];  // MMA commit at exit
  uint32_t tmem;
  int abort;
};
static_assert(sizeof(TcBars) <= 256, "tcgen05 prefill barrier block");

// Tensor maps of q and out, both [B][P][Hq * 128] bf16 (innermost first: Hq * 128, P, B),
// box 64 x 128 x 1 (one d-half of 128 query rows of one head), 128-byte swizzle.
struct TcMaps {
  CUtensorMap q, out;
};

// Key tile t of a unit: the first n_ct tiles cover the nc retained rows, the rest the band
// [bs, jmax] of dense rows.
struct TcTile {
  bool retained;
  int r0, rows;
};
__device__ __forceinline__ TcTile tc_tile(int t, int n_ct, int nc, int bs, int jmax) {
  TcTile x;
  x.retained = t < n_ct;
  x.r0 = x.retained ? t * kTcKeys : bs + (t - n_ct) * kTcKeys;
  x.rows = min(kTcKeys, (x.retained ? nc : jmax + 1) - x.r0);
  return x;
}

// Work unit u = ((rank B + b) H + hk) G + g: query head hq = hk G + g of sequence b on query
// tile n_qtiles - 1 - rank (latest, heaviest tiles first).  A CTA visits u, u + stride, ...;
// its roles step these digits by the stride's digits with carries (no divisions per unit).
struct TcIter {
  int g, hk, b, rank;
};
__device__ __forceinline__ TcIter tc_iter(const PrefillParams& p, int u) {
  TcIter it;
  const int B = p.batch;
  it.g = u % p.group;
  u /= p.group;
  it.hk = u % p.kv_heads;
  u /= p.kv_heads;
  it.b = u % B;
  it.rank = u / B;
  return it;
}
__device__ __forceinline__ void tc_advance(const PrefillParams& p, TcIter& it, const TcIter& st) {
  const int B = p.batch;
  it.g += st.g;
  int c = it.g >= p.group;
  if (c) it.g -= p.group;
  it.hk += st.hk + c;
  c = it.hk >= p.kv_heads;
  if (c) it.hk -= p.kv_heads;
  it.b += st.b + c;
  c = it.b >= B;
  if (c) it.b -= B;
  it.rank += st.rank + c;
}
__device__ __forceinline__ bool tc_valid(const PrefillParams& p, const TcIter& it) {
  return it.rank < p.n_qtiles;
}
// The unit's fields; the retained count nc (a load) is fetched separately, one unit ahead,
// by tc_unit_nc.
struct TcUnit {
  int b, hq, j0, jmax, nc, bs, n_ct, n_tiles;
  int64_t head;  // b * kv_heads + hk: the packed K / V rows
};
__device__ __forceinline__ TcUnit tc_unit(const PrefillParams& p, const TcIter& it, int nc) {
  TcUnit x;
  x.b = it.b;
  x.hq = it.hk * p.group + it.g;
  x.head = (int64_t)it.b * p.kv_heads + it.hk;
  x.j0 = (p.n_qtiles - 1 - it.rank) * kPfRows;
  x.jmax = min(x.j0 + kPfRows, p.P) - 1;
  x.nc = nc;
  x.bs = max(0, x.j0 - p.window) & ~7;
  x.n_ct = (nc + kTcKeys - 1) / kTcKeys;
  x.n_tiles = x.n_ct + (x.jmax + 1 - x.bs + kTcKeys - 1) / kTcKeys;
  return x;
}
// Retained keys visible to the unit's last query (0 past the last unit).
__device__ __forceinline__ int tc_unit_nc(const PrefillParams& p, const TcIter& it) {
  if (!tc_valid(p, it)) return 0;
  const int64_t head = (int64_t)it.b * p.kv_heads + it.hk;
  const int jmax = min((p.n_qtiles - it.rank) * kPfRows, p.P) - 1;
  return jmax - p.window > 0 ? p.before[head * (p.P + 1) + (jmax - p.window)] : 0;
}

// Rows [r0, r0 + rows) of one head's packed K or V (two d-halves) into a 128-row tile.
__device__ __forceinline__ void tc_stage_rows(uint8_t* dst, const uint8_t* src, int64_t head,
                                              int P, int r0, int rows, uint64_t* bar) {
  const uint32_t bytes = (uint32_t)rows * 128u;
#pragma unroll
  for (int dh = 0; dh < 2; ++dh)
    bulk_copy_g2s(dst + dh * kTcHalfBytes, src + ((head * 2 + dh) * P + r0) * 128, bytes, bar);
}


__global__ void __launch_bounds__(kTcThreads, 1)
    prefill_tc_kernel(const __grid_constant__ PrefillParams p, const __grid_constant__ TcMaps maps) {
  extern __shared__ __align__(1024) uint8_t smem_tc[];
  uint8_t* smem = smem_tc;
  if (smem_addr(smem) & 1023u) {  // uniform over the CTA: nothing has started yet
    if (threadIdx.x == 0) set_device_error(p.err, DMS_ERR_CUDA);
    return;
  }
  TcBars& bars = *reinterpret_cast<TcBars*>(smem + kTcOffBar);
  volatile int* abort_flag = &bars.abort;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int P = p.P, w = p.window, G = p.group;
  const TcIter first = tc_iter(p, blockIdx.x), step = tc_iter(p, gridDim.x);

  if (tid == 0) {
    *abort_flag = 0;
    for (int s = 0; s < kTcKSlots; ++s) {
      mbar_init(&bars.k_full[s], 1);
      mbar_init(&bars.k_empty[s], 1);
    }
    for (int s = 0; s < kTcVSlots; ++s) {
      mbar_init(&bars.v_full[s], 1);
      mbar_init(&bars.v_empty[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&bars.q_full[i], 1);
      mbar_init(&bars.q_ready[i], 1);
      mbar_init(&bars.o_staged[i], kTcSoftmaxWarps);
      mbar_init(&bars.s_full[i], 1);
      mbar_init(&bars.p_full[i], 4);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&bars.o_full[i], 1);
      mbar_init(&bars.mma_done[i], 1);
    }
    mbar_init(&bars.o_free, kTcSoftmaxWarps);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    tmem_alloc(&bars.tmem, kTcCols);
    tc_fence_before();
  }
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bars.tmem;

  if (warp == 0) {
    // ================================================================ K / V producer
    // The whole warp waits and zeroes stale V rows; lane 0 issues the copies.  A slot is
    // refilled only after the MMAs that read its previous tile are done.  K runs two tiles
    // ahead of V in this warp's order (K(g + 2) before V(g)): a V slot is freed by the
    // product two tiles back, which must not hold up the keys the next scores need.
    struct PCur {  // a tile of the CTA: unit, next unit, its fields, tile in unit
      TcIter it, nx;
      TcUnit x;
      int nc_next, t;
      bool valid;
    };
    auto pstart = [&](PCur& c) {
      c.it = c.nx = first;
      tc_advance(p, c.nx, step);
      c.valid = tc_valid(p, c.it);
      c.x = tc_unit(p, c.it, tc_unit_nc(p, c.it));
      c.nc_next = tc_unit_nc(p, c.nx);  // used one unit later
      c.t = 0;
    };
    auto pnext = [&](PCur& c) {
      if (++c.t == c.x.n_tiles) {
        c.t = 0;
        c.it = c.nx;
        tc_advance(p, c.nx, step);
        c.valid = tc_valid(p, c.it);
        c.x = tc_unit(p, c.it, c.nc_next);
        c.nc_next = tc_unit_nc(p, c.nx);
      }
    };
    PCur kc, vc;
    pstart(kc);
    pstart(vc);
    int gk = 0, gv = 0;  // K and V tiles staged so far
    auto load_k = [&]() {
      const TcTile tl = tc_tile(kc.t, kc.x.n_ct, kc.x.nc, kc.x.bs, kc.x.jmax);
      const int ks = gk % kTcKSlots;
      if (gk >= kTcKSlots)
        mbar_wait(&bars.k_empty[ks], (gk / kTcKSlots - 1) & 1, abort_flag, p.err);
      if (lane == 0) {
        mbar_arrive_expect_tx(&bars.k_full[ks], 2u * (uint32_t)tl.rows * 128u);
        tc_stage_rows(smem + ks * kTcTileBytes, tl.retained ? p.kc : p.kd, kc.x.head, P, tl.r0,
                      tl.rows, &bars.k_full[ks]);
      }
      ++gk;
      pnext(kc);
    };
    auto load_v = [&]() {
      const TcTile tl = tc_tile(vc.t, vc.x.n_ct, vc.x.nc, vc.x.bs, vc.x.jmax);
      const int vs = gv % kTcVSlots;
      if (gv >= kTcVSlots)
        mbar_wait(&bars.v_empty[vs], (gv / kTcVSlots - 1) & 1, abort_flag, p.err);
      uint8_t* vt = smem + kTcOffV + vs * kTcTileBytes;
      if (tl.rows < kTcKeys) {
        const int n16 = (kTcKeys - tl.rows) * 8;  // 16-byte words past the rows, per d-half
        for (int e = lane; e < 2 * n16; e += 32) {
          const int dh = e >= n16 ? 1 : 0;
          *reinterpret_cast<uint4*>(vt + dh * kTcHalfBytes + tl.rows * 128 + (e - dh * n16) * 16) =
              make_uint4(0u, 0u, 0u, 0u);
        }
        fence_proxy_async_smem();  // visible to the tensor cores via the full barrier
        __syncwarp();
      }
      if (lane == 0) {
        mbar_arrive_expect_tx(&bars.v_full[vs], 2u * (uint32_t)tl.rows * 128u);
        tc_stage_rows(vt, tl.retained ? p.vc : p.vd, vc.x.head, P, tl.r0, tl.rows, &bars.v_full[vs]);
      }
      ++gv;
      pnext(vc);
    };
    // K(g + 2) needs only the scores of tile g - 1, whose V was staged before: no cycle
    for (int i = 0; i < 2 && kc.valid; ++i) load_k();
    while (vc.valid) {
      if (kc.valid) load_k();
      load_v();
    }
    // no copy may still be in flight when the CTA exits (matters only after a timeout)
    if (lane == 0) {
      for (int s = 0; s < kTcKSlots && s < gk; ++s) {
        const int last = s + ((gk - 1 - s) / kTcKSlots) * kTcKSlots;
        mbar_drain(&bars.k_full[s], (last / kTcKSlots) & 1);
      }
      for (int s = 0; s < kTcVSlots && s < gv; ++s) {
        const int last = s + ((gv - 1 - s) / kTcVSlots) * kTcVSlots;
        mbar_drain(&bars.v_full[s], (last / kTcVSlots) & 1);
      }
    }
  } else if (warp == kTcQWarp) {
    // ================================================================ Q in, O out
    // Before the Q of unit un goes into buffer un % 2, the O of unit un - 2 staged there is
    // stored and read out (its scores are done by then).
    int un = 0;
    TcUnit x1, x2;  // the units one and two before
    auto store_o = [&](int v, const TcUnit& y) {
      // o_staged[v % 2] is one phase ahead at most: unit v + 2 needs the Q loaded after this
      mbar_wait(&bars.o_staged[v & 1], (v >> 1) & 1, abort_flag, p.err);
      if (lane == 0) {
        const uint8_t* so = smem + kTcOffQ + (v & 1) * kTcQBytes;
        tma_store_3d(&maps.out, y.hq * kHeadDim, y.j0, y.b, so);
        tma_store_3d(&maps.out, y.hq * kHeadDim + 64, y.j0, y.b, so + kPfRows * 128);
        bulk_commit_group();
        bulk_wait_group_read0();
      }
      __syncwarp();
    };
    for (TcIter it = first; tc_valid(p, it); tc_advance(p, it, step), ++un) {
      const TcUnit x = tc_unit(p, it, 0);  // position fields only
      const int qi = un & 1;
      uint8_t* sq = smem + kTcOffQ + qi * kTcQBytes;  // [d-half][row][128 B], swizzled
      if (un >= 2) store_o(un - 2, x2);
      if (lane == 0) {
        mbar_arrive_expect_tx(&bars.q_full[qi], (uint32_t)kTcQBytes);
        for (int dh = 0; dh < 2; ++dh)
          tma_load_3d(sq + dh * (kPfRows * 128), &maps.q, x.hq * kHeadDim + 64 * dh, x.j0, x.b,
                      &bars.q_full[qi]);
      }
      if (p.zero_first) {
        // App. B: the decision element (head_dim 0 of the group's first head) is not a query
        // feature; zero it in the landed tile before any score reads it (q_full[qi] is one
        // phase ahead at most: the next Q for this buffer is loaded by this warp)
        mbar_wait(&bars.q_full[qi], (un >> 1) & 1, abort_flag, p.err);
        if (x.hq % G == 0)
          for (int r = lane; r < kPfRows; r += 32)
            *reinterpret_cast<uint16_t*>(sq + r * 128 + chunk_in_row(r, 0)) = 0;
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(&bars.q_ready[qi]);
      }
      x2 = x1;
      x1 = x;
    }
    if (un >= 2) store_o(un - 2, x2);
    if (un >= 1) store_o(un - 1, x1);
    if (lane == 0)  // no copy may still be in flight when the CTA exits
      for (int i = 0; i < 2 && i < un; ++i) {
        const int last = i + ((un - 1 - i) / 2) * 2;
        mbar_drain(&bars.q_full[i], (last >> 1) & 1);
      }
  } else if (warp == 1 || warp == kTcMmaWarp1) {
    // ================================================================ MMA issuers
    // Warp 1 issues set 0's products, warp 3 set 1's: per set, S of its first tile, then per
    // tile tau of the set O_s += P(tau) V(tau), S of the set's next tile (into the same buffer,
    // after the product that reads it, in issue order).  The warp runs the loop (its values
    // stay warp-uniform) and one elected lane, the same throughout, issues each group of MMAs
    // with its commits: issued from a divergent single thread the MMAs of a tile took up to
    // 1.5x the tensor cores' time.  Each unit of the CTA passes both warps: at its start
    // after both accumulators of the unit before are read out (o_free), at its end with an
    // o_full commit, also for a unit without a tile of the set.
    const int ms = warp == 1 ? 0 : 1;
    {
      constexpr uint32_t idesc_s = f16_idesc(kPfRows, kTcKeys, 0);    // Q K^T: both K-major
      constexpr uint32_t idesc_o = f16_idesc(kPfRows, kHeadDim, 1);   // P V: V MN-major
      // Descriptors are built once and their start address (16-byte units) stepped: +2 per
      // 16 head_dim elements of Q / K inside a d-half, + the d-half size at k-step 4; +128
      // (2 KiB) per 16 keys of V, whose two d-halves are the leading-offset atoms.
      const uint64_t dq0 = sw128_desc(smem_addr(smem + kTcOffQ), 16u, 1024u);
      const uint64_t dk0 = sw128_desc(smem_addr(smem), 16u, 1024u);
      const uint64_t dv0 = sw128_desc(smem_addr(smem + kTcOffV), (uint32_t)kTcHalfBytes, 1024u);
      constexpr uint64_t kQBuf = kTcQBytes >> 4, kQHalf = (kPfRows * 128) >> 4;
      constexpr uint64_t kKHalf = kTcHalfBytes >> 4, kSlot = kTcTileBytes >> 4;
      const uint32_t d_s = tmem + kTcColS + (uint32_t)(128 * ms);  // this set's S buffer
      const uint32_t d_o = tmem + (uint32_t)(128 * ms);            // and accumulator
      // Cursor over the set's tiles for the scores: unit and next unit, unit ordinal, tile in
      // unit, tiles of unit, global tile index, next unit's retained count (one unit ahead).
      struct Cur {
        TcIter it, nx;
        int un, t, n, tau, nc_next;
      };
      Cur sc;
      sc.it = sc.nx = first;
      tc_advance(p, sc.nx, step);
      sc.un = sc.t = sc.tau = 0;
      sc.n = tc_valid(p, sc.it) ? tc_unit(p, sc.it, tc_unit_nc(p, sc.it)).n_tiles : 0;
      sc.nc_next = tc_unit_nc(p, sc.nx);
      auto step_tile = [&]() {
        ++sc.tau;
        if (++sc.t == sc.n) {
          sc.t = 0;
          sc.it = sc.nx;
          tc_advance(p, sc.nx, step);
          ++sc.un;
          sc.n = tc_valid(p, sc.it) ? tc_unit(p, sc.it, sc.nc_next).n_tiles : 0;
          sc.nc_next = tc_unit_nc(p, sc.nx);
        }
      };
      auto seek = [&]() {  // to the set's next tile (n = 0: none left)
        while (sc.n > 0 && (sc.tau & 1) != ms) step_tile();
      };
      auto issue_scores = [&]() {
        const int tau = sc.tau, qi = sc.un & 1;
        // the set's first tile of a unit: the unit's Q has landed (and, borrowed decisions,
        // is patched); q_full is one phase ahead at most, since Q two units on needs this
        // unit's O staged
        if (sc.t < kTcSets)
          mbar_wait(p.zero_first ? &bars.q_ready[qi] : &bars.q_full[qi], (sc.un >> 1) & 1,
                    abort_flag, p.err);
        mbar_wait(&bars.k_full[tau % kTcKSlots], (tau / kTcKSlots) & 1, abort_flag, p.err);
        tc_fence_after();
        const uint64_t dq = dq0 + (uint64_t)qi * kQBuf;
        const uint64_t dk = dk0 + (uint64_t)(tau % kTcKSlots) * kSlot;
        if (elect_one()) {
          tc_mma_ss_k<false>(d_s, dq, dk, idesc_s);
          tc_mma_ss_k<true>(d_s, dq + 2, dk + 2, idesc_s);
          tc_mma_ss_k<true>(d_s, dq + 4, dk + 4, idesc_s);
          tc_mma_ss_k<true>(d_s, dq + 6, dk + 6, idesc_s);
          tc_mma_ss_k<true>(d_s, dq + kQHalf, dk + kKHalf, idesc_s);
          tc_mma_ss_k<true>(d_s, dq + kQHalf + 2, dk + kKHalf + 2, idesc_s);
          tc_mma_ss_k<true>(d_s, dq + kQHalf + 4, dk + kKHalf + 4, idesc_s);
          tc_mma_ss_k<true>(d_s, dq + kQHalf + 6, dk + kKHalf + 6, idesc_s);
          tc_commit(&bars.s_full[ms]);
          tc_commit(&bars.k_empty[tau % kTcKSlots]);  // the K slot is free once these are done
        }
        __syncwarp();
        step_tile();
        seek();
      };
      seek();
      if (sc.n > 0) issue_scores();
      // products, unit by unit
      TcIter it = first, nx = first;
      tc_advance(p, nx, step);
      int nc = tc_unit_nc(p, it), tau0 = 0, un = 0;
      for (; tc_valid(p, it); it = nx, tc_advance(p, nx, step), ++un) {
        const int nc_next = tc_unit_nc(p, nx);  // used one unit later
        const int n = tc_unit(p, it, nc).n_tiles;
        // a unit's products overwrite the accumulators: the previous unit's are read out
        // (o_free completes once per unit, after both o_full of that unit, which need this
        // warp's commit below)
        if (un > 0) mbar_wait(&bars.o_free, (un - 1) & 1, abort_flag, p.err);
        int t = (tau0 & 1) == ms ? 0 : 1;
        if (t >= n && elect_one()) tc_commit(&bars.o_full[ms]);  // no tile of this set
        __syncwarp();
        for (; t < n; t += kTcSets) {
          const int tau = tau0 + t;
          // S(tau) was issued after the set's previous product: p_full[ms] is one phase
          // ahead at most
          mbar_wait(&bars.p_full[ms], (tau >> 1) & 1, abort_flag, p.err);
          mbar_wait(&bars.v_full[tau % kTcVSlots], (tau / kTcVSlots) & 1, abort_flag, p.err);
          tc_fence_after();
          // keys 16 kk .. 16 kk + 15: P columns 8 kk .. of the buffer; V rows 16 kk ..
          // (2 KiB per 16 rows).  The set's first tile of the unit starts its accumulator.
          const uint64_t dv = dv0 + (uint64_t)(tau % kTcVSlots) * kSlot;
          const bool first_of_set = t < kTcSets, last_of_set = t + kTcSets >= n;
          if (elect_one()) {
            if (first_of_set)
              tc_mma_ts_k<false>(d_o, d_s, dv, idesc_o);
            else
              tc_mma_ts_k<true>(d_o, d_s, dv, idesc_o);
#pragma unroll
            for (int kk = 1; kk < kTcKeys / 16; ++kk)
              tc_mma_ts_k<true>(d_o, d_s + 8 * kk, dv + 128 * kk, idesc_o);
            tc_commit(&bars.v_empty[tau % kTcVSlots]);
            if (last_of_set) tc_commit(&bars.o_full[ms]);  // the set's part of the unit's O
          }
          __syncwarp();
          if (sc.n > 0) issue_scores();
        }
        tau0 += n;
        nc = nc_next;
      }
      // the tensor memory is released only after every product has landed
      if (elect_one()) tc_commit(&bars.mma_done[ms]);
      __syncwarp();
      mbar_drain(&bars.mma_done[ms], 0);
    }
  } else {
    // ================================================================ softmax
    const int set = (warp - kTcSoftmax0) >> 2;  // takes the tiles with tau % 2 = set
    const int quarter = warp & 3;
    const int row = 32 * quarter + lane;        // query row of the tile = TMEM lane
    const uint32_t lane_addr = tmem + ((uint32_t)(32 * quarter) << 16);
    const uint32_t o_own = lane_addr + (uint32_t)(128 * set);
    const uint32_t o_other = lane_addr + (uint32_t)(128 * (set ^ 1));
    const uint32_t s_own = lane_addr + kTcColS + (uint32_t)(128 * set);
    float2* xml = reinterpret_cast<float2*>(smem + kTcOffX);  // [set][row]: (m, l)
    const float scale = p.scale_log2;
    const float2 scale2 = make_float2(scale, scale);
    // the row's count of visible retained keys, before[j - w] (0 for j <= w), one unit ahead
    auto row_before = [&](const TcIter& it) {
      if (!tc_valid(p, it)) return 0;
      const TcUnit y = tc_unit(p, it, 0);
      const int j = y.j0 + row;
      return j - w > 0 ? p.before[y.head * (P + 1) + min(j - w, P)] : 0;
    };
    // End of unit v (both sets): publish this set's (m, l) of the row, combine the two
    // accumulators for d-half `set` and stage it as bf16 in the unit's Q buffer.  o_full is
    // one phase ahead at most: the next unit's products need this call's o_free arrival.
    auto finish_unit = [&](int v, float mv, float lv) {
      mbar_wait(&bars.o_full[0], v & 1, abort_flag, p.err);
      mbar_wait(&bars.o_full[1], v & 1, abort_flag, p.err);
      tc_fence_after();
      xml[set * kPfRows + row] = make_float2(mv, lv);
      named_barrier_sync_id(1 + quarter, 64);  // the two sets' warps of this quarter
      const float2 ot = xml[(set ^ 1) * kPfRows + row];
      named_barrier_sync_id(1 + quarter, 64);  // read before either writes the next unit's
      // weights 2^(m_s - M); a set without visible keys (m = -inf) contributes nothing
      const float M = fmaxf(mv, ot.x);
      const bool own = mv != -INFINITY, oth = ot.x != -INFINITY;
      const float a0 = own ? ex2_approx(mv - M) : 0.f, a1 = oth ? ex2_approx(ot.x - M) : 0.f;
      const float lt = (own ? lv * a0 : 0.f) + (oth ? ot.y * a1 : 0.f);
      const float inv = lt > 0.f ? 1.f / lt : 0.f;
      const float c0 = a0 * inv, c1 = a1 * inv;
      uint8_t* half_row = smem + kTcOffQ + (v & 1) * kTcQBytes + set * (kPfRows * 128) + row * 128;
#pragma unroll 1
      for (int hh = 0; hh < 2; ++hh) {  // head_dim 64 set + 32 hh .. + 31
        float r0[32], r1[32];
#pragma unroll
        for (int c = 0; c < 32; c += 16) {
          tmem_ld16_at(o_own + (uint32_t)(64 * set + 32 * hh + c), r0 + c);
          tmem_ld16_at(o_other + (uint32_t)(64 * set + 32 * hh + c), r1 + c);
        }
        tmem_wait_ld();
#pragma unroll
        for (int c = 0; c < 4; ++c) {  // logical chunk 4 hh + c of the d-half
          float o[8];
#pragma unroll
          for (int e = 0; e < 8; ++e)
            o[e] = (own ? r0[8 * c + e] * c0 : 0.f) + (oth ? r1[8 * c + e] * c1 : 0.f);
          uint4 q4;
          q4.x = pack_bf16x2(o[0], o[1]);
          q4.y = pack_bf16x2(o[2], o[3]);
          q4.z = pack_bf16x2(o[4], o[5]);
          q4.w = pack_bf16x2(o[6], o[7]);
          *reinterpret_cast<uint4*>(half_row + chunk_in_row(row, 4 * hh + c)) = q4;
        }
      }
      tc_fence_before();  // the reads precede the next unit's products (via o_free)
      __syncwarp();
      if (lane == 0) mbar_arrive(&bars.o_free);
      fence_proxy_async_smem();  // visible to the tensor-map store
      __syncwarp();
      if (lane == 0) mbar_arrive(&bars.o_staged[v & 1]);
    };
    int tau = 0, un = 0;
    TcIter it = first, nx = first;
    tc_advance(p, nx, step);
    int nc = tc_unit_nc(p, it), bj_next = row_before(it);
    // an unfinished unit: its ordinal (or -1) and this set's (m, l) of the row
    int pend = -1;
    float m_pend = -INFINITY, l_pend = 0.f;
    for (; tc_valid(p, it); it = nx, tc_advance(p, nx, step), ++un) {
      const TcUnit x = tc_unit(p, it, nc);
      const int bj = bj_next;  // the first bj compacted rows are this row's retained keys
      nc = tc_unit_nc(p, nx);  // both used one unit later
      bj_next = row_before(nx);
      const int j = x.j0 + row;
      float m = -INFINITY;  // reference max of the row in this set (log2 domain)
      float l = 0.f;        // running sum of the row in this set
      bool started = false; // this set has taken a tile of the unit
      for (int t = 0; t < x.n_tiles; ++t, ++tau) {
        if ((tau & 1) != set) continue;
        const TcTile tl = tc_tile(t, x.n_ct, x.nc, x.bs, x.jmax);
        int lo, nvis;  // visible keys of the tile: lo .. lo + nvis - 1
        if (tl.retained) {
          lo = 0;
          nvis = min(max(bj - tl.r0, 0), tl.rows);
        } else {
          lo = max(j - w - tl.r0, 0);
          nvis = max(min(j - tl.r0, tl.rows - 1) - lo + 1, 0);
        }
        // S(tau + 2) into this buffer follows this tile's P-ready arrival: one phase at most
        mbar_wait(&bars.s_full[set], (tau >> 1) & 1, abort_flag, p.err);
        tc_fence_after();
        float sc[kTcKeys];
#pragma unroll
        for (int c = 0; c < kTcKeys; c += 16) tmem_ld16_at(s_own + c, sc + c);
        tmem_wait_ld();
        if (!__all_sync(0xffffffffu, lo == 0 && nvis == kTcKeys)) {
#pragma unroll
          for (int k = 0; k < kTcKeys; ++k)
            if ((unsigned)(k - lo) >= (unsigned)nvis) sc[k] = -INFINITY;
        }
        float mx8[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) mx8[e] = fmaxf(sc[e], sc[8 + e]);
#pragma unroll
        for (int k = 16; k < kTcKeys; k += 16)
#pragma unroll
          for (int e = 0; e < 8; ++e) mx8[e] = max3f(mx8[e], sc[k + e], sc[k + 8 + e]);
        const float mt = max3f(max3f(mx8[0], mx8[1], mx8[2]), max3f(mx8[3], mx8[4], mx8[5]),
                               fmaxf(mx8[6], mx8[7])) * scale;
        float corr = 1.f;
        if (mt > m + kTcRescale) {
          corr = ex2_approx(m - mt);  // 0 when m = -inf
          m = mt;
        }
        const float nb = m == -INFINITY ? 0.f : -m;
        const float2 nb2 = make_float2(nb, nb);
        float2 s2[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
#pragma unroll
        for (int g = 0; g < kTcKeys / 16; ++g) {  // 16 keys -> 8 packed columns, stored at once
          uint32_t pk[8];
#pragma unroll
          for (int c = 0; c < 8; ++c) {
            const int k = 16 * g + 2 * c;
            const float2 y = fma_f32x2(make_float2(sc[k], sc[k + 1]), scale2, nb2);
            const float2 pp = make_float2(ex2_approx(y.x), ex2_approx(y.y));
            s2[c & 1] = add_f32x2(s2[c & 1], pp);
            pk[c] = pack_bf16x2(pp.x, pp.y);
          }
          tmem_st8_u32(s_own + (uint32_t)(8 * g), pk);
        }
        const float2 ss = add_f32x2(s2[0], s2[1]);
        l = l * corr + (ss.x + ss.y);
        if (started && __any_sync(0xffffffffu, corr != 1.f)) {
          // (rare) the row of O_s: the product of this set's previous tile completed before
          // S(tau) (issued after it); O += P(tau) V waits for the arrival below
#pragma unroll 1
          for (int c = 0; c < kHeadDim; c += 16) {
            float r[16];
            tmem_ld16(o_own + (uint32_t)c, r);
            tmem_wait_ld();
#pragma unroll
            for (int e = 0; e < 16; ++e) r[e] *= corr;
            tmem_st16(o_own + (uint32_t)c, r);
          }
        }
        started = true;
        tmem_wait_st();
        tc_fence_before();
        // the previous unit, when this set did not take its last tile: its accumulators are
        // read out before this tile's product may start the next one
        if (pend >= 0) {
          finish_unit(pend, m_pend, l_pend);
          pend = -1;
        }
        __syncwarp();  // the warp's stores are ordered before its one arrival
        if (lane == 0) mbar_arrive(&bars.p_full[set]);
        if (t == x.n_tiles - 1) finish_unit(un, m, l);  // this set took the unit's last tile
      }
      if (((tau - 1) & 1) != set) {  // the other set took the last tile: finish with the next
        pend = un;
        m_pend = m;
        l_pend = l;
      }
    }
    if (pend >= 0) finish_unit(pend, m_pend, l_pend);
  }
  // ---- teardown: every tensor-memory access is done before the columns are released
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTcCols);
  }
}

}  // namespace

// cuTensorMapEncodeTiled through the runtime's driver entry point (no link to the driver).
using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                   const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                   const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeTiledFn encode_tiled_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q = cudaDriverEntryPointSymbolNotFound;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(f);
  });
  return fn;
}

// [B][P][Hq * 128] bf16 tensor map with a box of one d-half of 128 rows of one head.
bool encode_qo_map(CUtensorMap* map, const void* base, int64_t batch, int64_t P, int64_t hq) {
  const EncodeTiledFn fn = encode_tiled_fn();
  if (fn == nullptr) return false;
  const cuuint64_t dims[3] = {(cuuint64_t)(hq * kHeadDim), (cuuint64_t)P, (cuuint64_t)batch};
  const cuuint64_t strides[2] = {(cuuint64_t)(hq * kRowBytes), (cuuint64_t)(P * hq * kRowBytes)};
  const cuuint32_t box[3] = {64u, (cuuint32_t)kPfRows, 1u};
  const cuuint32_t estr[3] = {1u, 1u, 1u};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3u, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

size_t prefill_workspace_bytes(int64_t heads, int64_t n_tokens) {
  return pf_layout(heads, n_tokens).total;
}

cudaError_t launch_prefill(const void* q, const void* k, const void* v, const void* logit,
                           int64_t logit_stride, int32_t batch, int32_t n_tokens, int32_t kv_heads,
                           int32_t group, int32_t window, bool immediate, float scale_log2,
                           bool zero_first, int32_t kernel, void* workspace, void* out,
                           cudaStream_t stream) {
  // The kernels' shared-memory limits, raised once per device.
  static std::atomic<uint64_t> attr_set{0};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const uint64_t bit = dev < 64 ? (1ull << dev) : 0ull;
  if (bit == 0 || (attr_set.load() & bit) == 0) {
    e = cudaFuncSetAttribute(prefill_attn_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             kPfSmemBytes);
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(prefill_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               kTcSmemBytes);
    if (e != cudaSuccess) return e;
    attr_set.fetch_or(bit);
  }
  const int64_t H = (int64_t)batch * kv_heads;
  const PfLayout L = pf_layout(H, n_tokens);
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  e = cudaMemsetAsync(ws + L.err, 0, 64, stream);
  if (e != cudaSuccess) return e;
  PackParams pk;
  pk.k = static_cast<const uint16_t*>(k);
  pk.v = static_cast<const uint16_t*>(v);
  pk.logit = static_cast<const uint16_t*>(logit);
  pk.logit_stride = logit_stride;
  pk.decider = immediate ? window : 0;
  pk.kd = ws + L.kd;
  pk.vd = ws + L.vd;
  pk.kc = ws + L.kc;
  pk.vc = ws + L.vc;
  pk.pc = reinterpret_cast<int32_t*>(ws + L.pc);
  pk.before = reinterpret_cast<int32_t*>(ws + L.before);
  pk.cc = reinterpret_cast<int32_t*>(ws + L.cc);
  pk.P = n_tokens;
  pk.kv_heads = kv_heads;
  pk.nch = (n_tokens + kPfChunk - 1) / kPfChunk;
  const dim3 pgrid((unsigned)pk.nch, (unsigned)H);
  prefill_count_kernel<<<pgrid, kPfPackThreads, 0, stream>>>(pk);
  prefill_pack_kernel<<<pgrid, kPfPackThreads, 0, stream>>>(pk);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  PrefillParams pp;
  pp.q = static_cast<const __nv_bfloat16*>(q);
  pp.out = static_cast<__nv_bfloat16*>(out);
  pp.kd = pk.kd;
  pp.vd = pk.vd;
  pp.kc = pk.kc;
  pp.vc = pk.vc;
  pp.pc = pk.pc;
  pp.before = pk.before;
  pp.err = reinterpret_cast<int32_t*>(ws + L.err);
  pp.P = n_tokens;
  pp.kv_heads = kv_heads;
  pp.group = group;
  pp.window = window;
  pp.zero_first = zero_first ? 1 : 0;
  pp.n_qtiles = (n_tokens + kPfRows - 1) / kPfRows;
  pp.n_qheads = (int32_t)(H * group);
  pp.batch = batch;
  pp.scale_log2 = scale_log2;
  const int64_t grid = (int64_t)pp.n_qtiles * pp.n_qheads;
  if (kernel == DMS_PREFILL_MMA_SYNC) {
    prefill_attn_kernel<<<(unsigned)grid, kPfThreads, kPfSmemBytes, stream>>>(pp);
  } else {
    TcMaps maps;
    if (!encode_qo_map(&maps.q, q, batch, n_tokens, pp.n_qheads / batch) ||
        !encode_qo_map(&maps.out, out, batch, n_tokens, pp.n_qheads / batch))
      return cudaErrorInvalidValue;
    // persistent: one CTA per SM (fewer when there are fewer work units)
    int sms = 0;
    e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    const int64_t units = (int64_t)pp.n_qtiles * pp.n_qheads;
    const unsigned ctas = (unsigned)(units < sms ? units : sms);
    prefill_tc_kernel<<<ctas, kTcThreads, kTcSmemBytes, stream>>>(pp, maps);
  }
  return cudaGetLastError();
}

}  // namespace dms

// ============================================================================ C ABI
namespace {

bool pf_aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

dms_status prefill_impl(const void* q, const void* k, const void* v, const void* logit,
                        int64_t logit_stride, int32_t batch, int32_t n_tokens, int32_t kv_heads,
                        int32_t gqa_group, int32_t window, int32_t policy, int32_t kernel,
                        float sm_scale, void* workspace, size_t workspace_bytes, void* out,
                        bool zero_first, void* stream) {
  if (q == nullptr || k == nullptr || v == nullptr || logit == nullptr || out == nullptr ||
      workspace == nullptr || !pf_aligned16(q) || !pf_aligned16(k) || !pf_aligned16(v) ||
      !pf_aligned16(out) || !pf_aligned16(workspace) ||
      (reinterpret_cast<uintptr_t>(logit) & 1u) != 0 || batch < 1 || n_tokens < 1 ||
      kv_heads < 1 || gqa_group < 1 || gqa_group > dms::kMaxGroup || window < 0 ||
      !(sm_scale == sm_scale) || policy < DMS_EVICT_DELAYED || policy > DMS_EVICT_IMMEDIATE ||
      kernel < DMS_PREFILL_TCGEN05 || kernel > DMS_PREFILL_MMA_SYNC)
    return DMS_ERR_INVALID_ARGUMENT;
  const int64_t H = (int64_t)batch * kv_heads;
  const int64_t qtiles = ((int64_t)n_tokens + 127) / 128;
  if (H > 65535 || qtiles * H * gqa_group > 0x7fffffffll || n_tokens > (1 << 30))
    return DMS_ERR_INVALID_ARGUMENT;
  if (workspace_bytes < dms::prefill_workspace_bytes(H, n_tokens)) return DMS_ERR_CAPACITY;
  const float scale = sm_scale > 0.f ? sm_scale : 1.0f / sqrtf((float)dms::kHeadDim);
  const cudaError_t e = dms::launch_prefill(
      q, k, v, logit, logit_stride, batch, n_tokens, kv_heads, gqa_group, window,
      policy == DMS_EVICT_IMMEDIATE, scale * 1.4426950408889634f, zero_first, kernel, workspace,
      out, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? DMS_OK : DMS_ERR_CUDA;
}

}  // namespace

extern "C" {

dms_status dms_prefill_workspace_bytes(int32_t batch, int32_t n_tokens, int32_t kv_heads,
                                       size_t* out_bytes) {
  if (out_bytes == nullptr || batch < 1 || n_tokens < 1 || kv_heads < 1)
    return DMS_ERR_INVALID_ARGUMENT;
  *out_bytes = dms::prefill_workspace_bytes((int64_t)batch * kv_heads, n_tokens);
  return DMS_OK;
}

dms_status dms_prefill_attention(const void* q, const void* k, const void* v,
                                 const void* decision_logit, int32_t batch, int32_t n_tokens,
                                 int32_t kv_heads, int32_t gqa_group, int32_t window,
                                 float sm_scale, void* workspace, size_t workspace_bytes,
                                 void* out, void* stream) {
  return prefill_impl(q, k, v, decision_logit, 1, batch, n_tokens, kv_heads, gqa_group, window,
                      DMS_EVICT_DELAYED, dms::kPrefillDefaultKernel, sm_scale, workspace,
                      workspace_bytes, out, false, stream);
}

dms_status dms_prefill_attention_borrowed(const void* q, const void* k, const void* v,
                                          int32_t batch, int32_t n_tokens, int32_t kv_heads,
                                          int32_t gqa_group, int32_t window, float sm_scale,
                                          void* workspace, size_t workspace_bytes, void* out,
                                          void* stream) {
  if (gqa_group < 1 || gqa_group > dms::kMaxGroup) return DMS_ERR_INVALID_ARGUMENT;
  return prefill_impl(q, k, v, q, (int64_t)gqa_group * dms::kHeadDim, batch, n_tokens, kv_heads,
                      gqa_group, window, DMS_EVICT_DELAYED, dms::kPrefillDefaultKernel, sm_scale,
                      workspace, workspace_bytes, out, true, stream);
}

dms_status dms_prefill_attention_ex(const void* q, const void* k, const void* v,
                                    const void* decision_logit, int32_t batch, int32_t n_tokens,
                                    int32_t kv_heads, int32_t gqa_group, int32_t window,
                                    int32_t eviction_policy, int32_t kernel, float sm_scale,
                                    void* workspace, size_t workspace_bytes, void* out,
                                    void* stream) {
  if (gqa_group < 1 || gqa_group > dms::kMaxGroup) return DMS_ERR_INVALID_ARGUMENT;
  const bool borrowed = decision_logit == nullptr;
  return prefill_impl(q, k, v, borrowed ? q : decision_logit,
                      borrowed ? (int64_t)gqa_group * dms::kHeadDim : 1, batch, n_tokens,
                      kv_heads, gqa_group, window, eviction_policy, kernel, sm_scale, workspace,
                      workspace_bytes, out, borrowed, stream);
}

dms_status dms_prefill_device_error(const void* workspace, void* stream, dms_status* out) {
  if (workspace == nullptr || out == nullptr) return DMS_ERR_INVALID_ARGUMENT;
  int32_t word = 0;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (cudaMemcpyAsync(&word, static_cast<const int32_t*>(workspace) + dms::kCtrlError,
                      sizeof(word), cudaMemcpyDeviceToHost, st) != cudaSuccess ||
      cudaStreamSynchronize(st) != cudaSuccess)
    return DMS_ERR_CUDA;
  *out = static_cast<dms_status>(word);
  return DMS_OK;
}

}  // extern "C"
