// Internal interfaces between the C-ABI layer (api.cu) and the kernels.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <nvtx3/nvToolsExt.h>

#include "../../include/unicache.h"

namespace uc {

// One NVTX range per C-ABI call, named after the call (seen by profilers
// such as nsys when one is attached; a few nanoseconds otherwise).
struct TraceRange {
  explicit TraceRange(const char* name) { nvtxRangePushA(name); }
  ~TraceRange() { nvtxRangePop(); }
  TraceRange(const TraceRange&) = delete;
  TraceRange& operator=(const TraceRange&) = delete;
};
#define UC_TRACE() const ::uc::TraceRange uc_trace_range_(__func__)

struct DevStatus;

void count_launch();
void set_error(const char* fmt, ...);

// Programmatic dependent launch of the decode kernels (uc_set_programmatic_launch).
bool pdl_enabled();

#if defined(__CUDACC__)
// Launch with programmatic stream serialisation when `pdl`, else ordinary.
template <typename... KArgs, typename... Args>
inline void launch_maybe_pdl(bool pdl, void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                             cudaStream_t st, Args&&... args) {
  if (!pdl) {
    kernel<<<grid, block, smem, st>>>(static_cast<Args&&>(args)...);
    return;
  }
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaLaunchKernelEx(&cfg, kernel, static_cast<Args&&>(args)...);
}
#endif

// Limit of the decode kernels' bounded waits and the one-shot test hook that
// makes them run out (uc_set_wait_limit, uc_debug_withhold_tile).
uint64_t wait_limit_ns();
int take_withhold_pos();

// uc_attend's checks before it looks at its workspace (same order and
// statuses); *need: the workspace bytes the call takes.
uc_status attend_precheck(const void* q, int32_t n_q_heads, int32_t n_qtok, const uc_segment* const* segs,
                          int32_t n_seg, const void* out, const char* name, size_t* need);
// Bytes of a uc_attend call's merge counters in its workspace (after the
// 256-byte status word): a block of fixed size that must start at zero.
size_t attend_counter_bytes();

// ------------------------------------------------------------ compression
struct TopkArgs {
  const float* scores;
  int64_t scores_stride, scores_offset;
  int32_t* kept_idx;
  int32_t* n_kept;
  DevStatus* status;
  int n_kv_heads, n_src, n_recent, cap;
  int keep[UC_MAX_BATCH];
  int src_n[UC_MAX_BATCH];  // candidate tokens per sequence (n_src, or a source segment's kept count)
  // NULL: candidate i's score is scores[i]. Otherwise scores[score_idx[i]]
  // (re-compression: the source segment's logical index of stored row i).
  const int32_t* score_idx;
  int64_t score_idx_stride;
  int64_t score_limit;  // logical indices must lie in [0, score_limit)
};

struct GatherArgs {
  const __nv_bfloat16* k_src;
  const __nv_bfloat16* v_src;
  int64_t src_row_stride, src_row_offset;
  const int32_t* kept_idx;
  __nv_bfloat16* k_dst;  // EVICT: compacted rows; quantized: the tail block
  __nv_bfloat16* v_dst;
  int64_t dst_row_stride, dst_row_offset;
  uint64_t wait_ns;  // limit of the quantizer's bounded waits
  int withhold;      // test hook: a group whose K rows are not all copied (-1: none)
  uint8_t* k_codes;
  uint8_t* k_params;
  uint8_t* v_codes;
  uint8_t* v_params;
  DevStatus* status;
  int batch, n_kv_heads, cap, max_chunks;
  int keep[UC_MAX_BATCH];
};

struct AppendArgs {
  const __nv_bfloat16* k_new;
  const __nv_bfloat16* v_new;
  __nv_bfloat16* k;
  __nv_bfloat16* v;
  int64_t row_stride, row_offset;
  int32_t* kept_idx;
  int32_t* n_kept;
  uint8_t* k_codes;
  uint8_t* k_params;
  uint8_t* v_codes;
  uint8_t* v_params;
  DevStatus* status;
  int batch, n_kv_heads, cap, position;
  int position_plus_count;  // 1: logical index = position + n_kept[b] (device)
};

// Rows of a packed segment rebuilt in bf16: x = code * s + z (exact in fp32),
// rounded to nearest even; the bf16 tail copied. Output [nbh][cap][128].
struct DequantArgs {
  const uint8_t* k_codes;
  const uint8_t* k_params;
  const uint8_t* v_codes;
  const uint8_t* v_params;
  const __nv_bfloat16* k_tail;
  const __nv_bfloat16* v_tail;
  const int32_t* n_kept;
  __nv_bfloat16* k_out;
  __nv_bfloat16* v_out;
  int batch, n_kv_heads, cap, bits, max_groups;
};

// kept_idx[i] = src_idx[kept_idx[i]] for the first n_kept[b] entries.
struct ComposeArgs {
  int32_t* kept_idx;
  const int32_t* src_idx;
  const int32_t* n_kept;
  int n_kv_heads, cap, src_cap;
};

void launch_topk(const TopkArgs& a, int n_blocks, bool evict, cudaStream_t st);
void launch_dequant_rows(const DequantArgs& a, cudaStream_t st);
void launch_attention_mass(const float* mass, int batch, int rows, int n_seg, float scale,
                           bool accumulate, float* out, cudaStream_t st);
void launch_compose_idx(const ComposeArgs& a, int nbh, cudaStream_t st);
void launch_gather(const GatherArgs& a, cudaStream_t st);
void launch_quantize(const GatherArgs& a, int bits, cudaStream_t st);
void launch_append(const AppendArgs& a, int bits, cudaStream_t st);

// ---------------------------------------------------------------- scores
struct ScoreArgs {
  CUtensorMap tmap_k;  // bf16 rows of K, box 64 x 64, 128B swizzle
  const __nv_bfloat16* qwin;
  float* scores;
  float* part;         // [B*Hkv*chunks][rows_pad][2] (m, l) in log2 units
  float* lse2;         // [B*Hkv][rows_pad]
  DevStatus* status;
  int64_t k_row_stride;
  int batch, n_q_heads, n_kv_heads, window, n_ctx, chunks, tiles_per_chunk, rows, mtiles;
  float scale_log2;
};

void launch_scores(const ScoreArgs& a, cudaStream_t st);

// Per-token attention probabilities of one decode step, added into a
// heavy-hitter accumulator indexed by logical token.
struct DecodeScoreArgs {
  const __nv_bfloat16* q;   // [B, Hq, T, 128]
  const float* lse;         // [B, Hq, T], natural log
  const __nv_bfloat16* k;   // segment rows: block (b, kvh) at (b*Hkv + kvh)*row_stride + row_offset
  int64_t row_stride, row_offset;
  const int32_t* kept_idx;  // [B, Hkv, cap] logical indices; NULL: row t is token t
  const int32_t* n_kept;    // [B]
  float* acc;               // [B, Hkv, acc_stride]
  int64_t acc_stride, acc_offset;
  DevStatus* status;
  int cap, n_kv_heads, n_q_heads, n_qtok, group, rows;
  float scale;
};
void launch_decode_scores(const DecodeScoreArgs& a, int batch, int max_tokens, cudaStream_t st);
void launch_segment_mass(const float* scores, int batch, int n_kv_heads, int n_ctx,
                         const int32_t* begin, const int32_t* end, int n_seg, float inv_norm,
                         bool accumulate, float* mass, cudaStream_t st);

// ------------------------------------------------------------- attention
struct SegDev {
  int kind, bits, cap, chunk_begin, n_chunks, tiles_per_chunk_hint;
  int64_t row_stride, row_offset;
  const int32_t* n_kept;
  const uint8_t* k_codes;
  const uint8_t* k_params;
  const uint8_t* v_codes;
  const uint8_t* v_params;
};

struct AttnParams {
  CUtensorMap tmap[2 * UC_MAX_SEGMENTS];  // [2s] keys, [2s+1] values (bf16 rows)
  SegDev seg[UC_MAX_SEGMENTS];
  const __nv_bfloat16* q;
  __nv_bfloat16* out;
  float* lse;
  float* mass;
  float* part;       // per item: [rows_pad][128] O, then [rows_pad] m, [rows_pad] l
  int32_t* counters; // [B*Hkv]
  int32_t* sched;    // launch-wide work queue: [0] next item, [1] CTAs done (re-armed to 0)
  DevStatus* status;
  int nseg, batch, n_kv_heads, n_q_heads, n_qtok, group, rows, mtiles, items_per_bh, n_items;
  // processing order: positions [0, n_heavy * nbh) walk the heavy items
  // (bh = pos / n_heavy, local item heavy_local[pos % n_heavy]); the rest
  // walk the light items (bh = pos' / n_light, local light_local[...]):
  // the bf16 tails of packed segments and segments too small for an item of
  // their own
  int n_heavy, n_light;
  int16_t heavy_local[128];
  int16_t light_local[2 * UC_MAX_SEGMENTS];
  int defer_merge;  // 1: the attend launch only leaves partials; a merge kernel follows
  float scale_log2;
  uint64_t wait_ns;  // limit of every bounded wait of the launch (UC_ERR_TIMEOUT past it)
  int withhold_pos;  // test hook: the first tile of the item at this position is never copied (-1: none)
};

// Several decode calls in one launch: the heavy items of every call (call
// order), then their light tail items.
struct MultiAttnParams {
  AttnParams call[UC_MAX_CALLS];
  int heavy_begin[UC_MAX_CALLS + 1];  // prefix over calls of n_heavy * B * Hkv
  int light_begin[UC_MAX_CALLS + 1];  // prefix over calls of n_light * B * Hkv
  int n_calls, n_items;
};

// ------------------------------------------------- dense (many queries)
struct DenseTile {
  int32_t row;       // first row of the tile inside a (b, kvh) block of khi / v
  int32_t lo_row;    // first row inside the klo block, -1 for bf16 segments
  int16_t seg;       // segment index
  int16_t seg_tile;  // tile index inside the segment
};

// Items per (sequence, KV head) whose partial outputs the in-kernel merge of
// a single-n-tile decode call stages in one round trip (two 32 KB ring slots
// of seven (O, m, l) partials each); more take a slower path.
constexpr int kWholeMergeItems = 14;
constexpr int kDenseKeys = 128;     // keys per dense tile
constexpr int kMaxDenseTiles = 512;  // up to 65536 keys per call

struct DenseParams {
  CUtensorMap tmap_khi, tmap_klo, tmap_v;  // fp16 rows, box 64 x 128, 128B swizzle
  SegDev seg[UC_MAX_SEGMENTS];
  const __nv_bfloat16* seg_k[UC_MAX_SEGMENTS];
  const __nv_bfloat16* seg_v[UC_MAX_SEGMENTS];
  DenseTile tiles[kMaxDenseTiles];
  __half* khi;
  __half* klo;
  __half* v;
  const __nv_bfloat16* q;
  __nv_bfloat16* out;
  float* lse;
  float* mass;
  DevStatus* status;
  int64_t rows_per_bh, lo_rows_per_bh;
  int n_tiles, nseg, batch, n_kv_heads, n_q_heads, n_qtok, group;
  int serial_pv;  // 1: wait for P V of a Q tile before its next Q K^T
  float scale_log2;
};

size_t dense_smem_bytes();
void launch_dense(const DenseParams& p, cudaStream_t st);

int attend_ctas_per_sm(int ntiles);
__host__ __device__ size_t attend_part_floats(int mtiles);
void launch_attend(const AttnParams& p, int grid, cudaStream_t st);
void launch_attend_multi(const MultiAttnParams& m, int grid, cudaStream_t st);

}  // namespace uc
