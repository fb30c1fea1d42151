// Internal declarations of libdms (not part of the C ABI).
//
// HBM layout of one cache (all device memory owned by the cache):
//   pool        [pool_pages][2][64][128] bf16   page = 64 K rows then 64 V rows (32 KiB).
//               Each 256-byte row is stored with its sixteen 16-byte chunks permuted:
//               logical chunk c of row r sits at physical chunk c ^ (r & 7).  A 1-D bulk
//               copy of whole rows therefore lands in shared memory already in a
//               bank-conflict-free order for ldmatrix (8 consecutive rows hit 8 distinct
//               16-byte bank groups).
//   (fp8 E4M3 format, DMS_KV_FP8_E4M3: pages of 16.5 KiB)
//   pool        [pool_pages][16896] bytes: 64 K rows of 128 codes, then V transposed,
//               128 rows (one per head_dim index d) of 64 codes (one per slot), then
//               the 64 key and 64 value row scales (fp32, page_scales_fp8), so that one
//               bulk copy fetches a page.  Both code halves
//               are laid out for the tiled decode kernel's m16n8k16 A fragments: in a
//               K row, the 16-code block of k-step kk sits in the 16-byte chunk group
//               kk / 4 and the four codes one thread needs (d = 16 kk + {2c, 2c+1,
//               2c+8, 2c+9}) are 4 consecutive bytes; in a V^T row the four codes of
//               tokens {2c, 2c+1, 2c+8, 2c+9} of a 16-slot block likewise.  16-byte
//               chunks are XOR-permuted by the row (K: k8_swizzle(row); V^T: (d >> 1) & 3) so
//               a warp's loads hit distinct banks.  k8_offset / vt8_offset below.
//   pos         [pool_pages][64] int32          position held by each slot (inspection only;
//                                               decode never reads it).
//   page_table  [layers][heads][max_pages] int32 page of slot s is page_table[.][s / 64].
//   counts      [layers][2][heads] int32         n_h: slots [0, n_h) hold the retained set.
//               Double-buffered: a layer of length T keeps its counts in buffer T & 1,
//               and an append of n tokens reads buffer T & 1 and writes (T + n) & 1, so
//               a kernel whose CTAs all read every head's count never sees a count
//               that another CTA of the same launch has already advanced.
//   rings       [layers][heads][ring_len] u32    decisions of recent tokens: the entry of
//               position j sits at j % (window + 2) and holds slot | e << 31, e the bit
//               that decides the token's eviction when it leaves the window: its own
//               alpha_j (delayed eviction), or alpha_{j+window}, OR-ed in when token
//               j + window arrives (immediate-eviction ablation; 0 until then).  The
//               period is one longer than the window + 1 tokens that must be kept, so
//               the entry read for the token leaving at step j ((j - window - 1) %
//               (window + 2)) and the entry written for the new token (j % (window + 2))
//               are always different words.
//   ctrl        [kCtrlWords] int32               [0] next free page, [1] sticky error.
//   freed       [heads][ring_len] int32          bulk-append scratch (slots freed this call).
//   pieces      [piece_capacity][kPieceFloats]   split-K partial records of the decode.
//   piece_counters [heads] int32                 arrivals per head for the last-CTA combine.
//   head_flags  [layers][heads] u32              completion flags of the cluster kernel.
// heads = batch * kv_heads, indexed b * kv_heads + h.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "dms.h"

namespace dms {

constexpr int kHeadDim = 128;
constexpr int kPageTokens = 64;
constexpr int kRowBytes = kHeadDim * 2;                       // 256
constexpr int kHalfPageBytes = kPageTokens * kRowBytes;       // 16384
constexpr int kPageBytes = 2 * kHalfPageBytes;                // 32768
constexpr int kHalfPageBytesFp8 = 8192;                       // fp8 page: K codes 8 KiB, V^T 8 KiB,
constexpr int kScaleBytes = 2 * kPageTokens * 4;              // then the key and value row scales
constexpr int kPageCodesBytesFp8 = 2 * kHalfPageBytesFp8;     // 16384
constexpr int kPageBytesFp8 = kPageCodesBytesFp8 + kScaleBytes;  // 16896: one bulk copy per page
constexpr int kMaxGroup = 16;                                 // query heads per KV head
constexpr int kMaxHeads = 4096;                               // batch * kv_heads
constexpr int kMaxCtasPerSm = 4;
constexpr uint32_t kAlphaBit = 0x80000000u;
constexpr uint32_t kSlotMask = 0x7fffffffu;
constexpr int64_t kMaxCapacity = (1ll << 30) - 1;  // slots stay below 2^30
constexpr int kPieceFloats = 2 * kMaxGroup + kMaxGroup * kHeadDim;  // m[16] l[16] o[16][128]
constexpr int kCtrlWords = 16;
constexpr int kCtrlPoolNext = 0;
constexpr int kCtrlError = 1;
// A bounded wait gives up after this many nanoseconds of %globaltimer.
constexpr unsigned long long kWaitLimitNs = 2000000000ull;

// The row scales of fp8 page `page` of the pool: [0, 64) the keys', [64, 128) the values'.
__host__ __device__ inline float* page_scales_fp8(uint8_t* pool, int64_t page) {
  return reinterpret_cast<float*>(pool + page * kPageBytesFp8 + kPageCodesBytesFp8);
}

struct Cache {
  int32_t layers = 0, kv_heads = 0, head_dim = 0, window = 0, batch = 0;
  int64_t capacity = 0;
  int32_t heads = 0;        // batch * kv_heads
  int32_t ring_len = 0;     // min(window + 2, capacity)
  int32_t max_pages = 0;    // ceil(capacity / 64)
  int64_t pool_pages = 0;
  int32_t decode_kernel = 0, ctas_per_sm = 1, min_pages_per_cta = 2;
  int32_t eviction_policy = DMS_EVICT_DELAYED;
  int32_t kv_format = DMS_KV_BF16;
  bool fp8() const { return kv_format == DMS_KV_FP8_E4M3; }
  int64_t page_bytes() const { return fp8() ? kPageBytesFp8 : kPageBytes; }
  // Position offset of the token whose decision evicts a given token: 0 for delayed
  // eviction (its own decision), window for the immediate-eviction ablation.
  int64_t decider() const { return eviction_policy == DMS_EVICT_IMMEDIATE ? window : 0; }
  int32_t device = 0, num_sms = 0;
  int64_t piece_capacity = 0;

  uint8_t* pool = nullptr;
  int32_t* pos = nullptr;
  int32_t* page_table = nullptr;
  int32_t* counts = nullptr;
  uint32_t* rings = nullptr;
  int32_t* ctrl = nullptr;
  int32_t* freed = nullptr;
  float* pieces = nullptr;
  int32_t* piece_counters = nullptr;

  int64_t* lengths = nullptr;  // host: tokens appended per layer
  int64_t peak_pages = 0;      // host: largest pages_in_use observed
  // host: layer of the last kernel launched on this cache (-1: none since creation or
  // reset), and whether it was a tiled decode with one CTA per SM.  After such a launch
  // for another layer, a tiled decode may read its layer's state before its dependency
  // wait (DecodeParams::state_ready in dms_decode.cu).
  int32_t last_layer = -1;
  bool last_full_tiled = false;
  // Clusters of C CTAs of the cluster decode kernel resident at once, C = 0..16.
  int32_t max_clusters[17] = {};
  // Per-head completion flags of the cluster kernel's fused append + decode: the launch
  // for length t of layer l stores its sequence number into head_flags[l][h] once head
  // h's cluster has finished every read and write of the layer's state.  Host: the last
  // number published per layer, and whether the layer's state was last written by such
  // a launch (cleared by any other append, a shared prompt or a reset).
  uint32_t* head_flags = nullptr;  // device [layers][heads]
  uint32_t* flag_seq = nullptr;    // host [layers]
  uint8_t* flag_valid = nullptr;   // host [layers]
  // Self-test: the wait limit (ns) of the next cluster launch of layer flag_test_layer (0: none).
  int64_t flag_test_wait_ns = 0;
  int32_t flag_test_layer = -1;

  // Count buffer of `layer` for a layer length of parity `parity`.
  int32_t* counts_at(int32_t layer, int64_t parity) const {
    return counts + ((int64_t)layer * 2 + (parity & 1)) * heads;
  }
};

// Sequence numbers of the completion flags: nonzero (0 marks "no flag to wait for").
inline uint32_t next_flag_seq(uint32_t seq) { return seq + 1u == 0u ? 1u : seq + 1u; }

// Ring period (entries per head cycle) for a sliding window w.
__host__ __device__ __forceinline__ int64_t ring_period(int64_t window) { return window + 2; }

// Sticky device error: the first code written wins.
__device__ __forceinline__ void set_device_error(int32_t* ctrl, int32_t code) {
  atomicCAS(ctrl + kCtrlError, 0, code);
}

// Sec. 3.2: alpha = round(sigmoid(x)) = [x > 0] on the bf16 bit pattern:
// sign bit clear, not +0, and not a NaN (+inf, 0x7f80, counts as > 0).
__device__ __forceinline__ uint32_t decision_from_bf16(uint16_t bits) {
  return (bits != 0u && bits <= 0x7f80u) ? 1u : 0u;
}

// Byte offset of logical 16-byte chunk `chunk` of row `row` inside a half page.
__host__ __device__ __forceinline__ uint32_t swizzled_offset(uint32_t row, uint32_t chunk) {
  return row * kRowBytes + ((chunk ^ (row & 7u)) << 4);
}

// fp8 page format.  Position of logical element d (0..127) of key row `row` (0..63)
// inside the page: k-step kk = d / 16, j = d % 16; thread c = (j & 7) / 2 of an
// m16n8k16 fragment needs j = 2c, 2c + 1, 2c + 8, 2c + 9, stored at bytes 0..3 of word
// kk % 4 of chunk 4 (kk / 4) + c, the chunk XOR-ed with k8_swizzle(row).  A quarter warp
// of the decode loads chunks 4 kg + c (c = 0..3) of two adjacent rows with 16-byte loads;
// the swizzle sends those two rows to different halves of the row's 8 chunks (the second
// term), so the eight loads hit eight different bank groups.
__host__ __device__ __forceinline__ uint32_t fp8_pair_index(uint32_t j) {
  return (j & 1u) | ((j >> 3) << 1);
}
__host__ __device__ __forceinline__ uint32_t k8_swizzle(uint32_t row) {
  return (row & 7u) ^ ((row & 1u) << 2);
}
__host__ __device__ __forceinline__ uint32_t k8_offset(uint32_t row, uint32_t d) {
  const uint32_t kk = d >> 4, j = d & 15u;
  const uint32_t chunk = (4u * (kk >> 2) + ((j & 7u) >> 1)) ^ k8_swizzle(row);
  return row * 128u + (chunk << 4) + 4u * (kk & 3u) + fp8_pair_index(j);
}
// Position of the value of slot `slot` (0..63) at head_dim index d in the V^T half:
// row d of 64 bytes, 16-slot block slot / 16 in chunk (slot / 16) ^ ((d >> 1) & 3), the
// slot's code at byte 4 c + pair index inside it (c, pair index of j = slot % 16 as for K).
__host__ __device__ __forceinline__ uint32_t vt8_offset(uint32_t slot, uint32_t d) {
  const uint32_t j = slot & 15u;
  const uint32_t chunk = (slot >> 4) ^ ((d >> 1) & 3u);
  return (uint32_t)kHalfPageBytesFp8 + d * 64u + (chunk << 4) + 4u * ((j & 7u) >> 1) +
         fp8_pair_index(j);
}

// Launchers (defined in the .cu files).  A decision logit sits at logit[i * logit_stride]
// for entry i = (b * n_tokens + t) * kv_heads + h: stride 1 for a separate logit tensor,
// gqa_group * 128 for the first element of each group's first query head (App. B).
// zero_first: attend with that element of every group's first query head taken as 0.
cudaError_t launch_append_one(const Cache& c, int32_t layer, const void* k, const void* v,
                              const void* logit, int64_t logit_stride, int64_t t0,
                              cudaStream_t stream);
cudaError_t launch_append_bulk(const Cache& c, int32_t layer, const void* k, const void* v,
                               const void* logit, int64_t logit_stride, int64_t t0, int32_t n,
                               cudaStream_t stream);
cudaError_t launch_append_shared_prefix(const Cache& c, int32_t layer, const void* k, const void* v,
                                        const void* logit, int32_t n, cudaStream_t stream);
cudaError_t launch_export_positions(const Cache& c, int32_t layer, int32_t* dev_out,
                                    cudaStream_t stream);
cudaError_t prepare_decode(const Cache& c);
cudaError_t launch_decode_tiled(const Cache& c, int32_t layer, const void* q, void* out,
                                int32_t group, float scale_log2, bool zero_first,
                                cudaStream_t stream);
cudaError_t launch_decode_simple(const Cache& c, int32_t layer, const void* q, void* out,
                                 int32_t group, float scale, bool zero_first, cudaStream_t stream);
bool append_decode_fusable(const Cache& c);
bool tiled_one_cta_per_sm(const Cache& c);  // tiled decode launches use one CTA per SM
cudaError_t prepare_cluster_decode(Cache& c);
// Cluster size of the decode of `group` query heads per KV head (0: the tiled kernel).
int decode_cluster_size(const Cache& c, int group, int64_t tokens);
cudaError_t launch_bounded_wait_probe(int arrive, int64_t limit_ns, int32_t* dev_status,
                                      cudaStream_t stream);
cudaError_t launch_append_decode(const Cache& c, int32_t layer, const void* k, const void* v,
                                 const void* logit, int64_t logit_stride, const void* q, void* out,
                                 int32_t group, float scale_log2, bool zero_first,
                                 cudaStream_t stream);

// Sparse prefill attention (dms_prefill.cu): caller-owned workspace of
// prefill_workspace_bytes(batch * kv_heads, n_tokens) bytes whose first 64 bytes are a
// control block (int32 [kCtrlError] holds the sticky device error).
size_t prefill_workspace_bytes(int64_t heads, int64_t n_tokens);
cudaError_t launch_prefill(const void* q, const void* k, const void* v, const void* logit,
                           int64_t logit_stride, int32_t batch, int32_t n_tokens, int32_t kv_heads,
                           int32_t group, int32_t window, bool immediate, float scale_log2,
                           bool zero_first, int32_t kernel, void* workspace, void* out,
                           cudaStream_t stream);

}  // namespace dms
