// C-ABI entry points: argument validation, TMA descriptor encoding, work
// planning and kernel launches. No entry point allocates device memory.
#include <cudaTypedefs.h>

#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <climits>
#include <cstring>
#include <mutex>

#include "common.cuh"
#include "internal.h"

namespace uc {

static thread_local char g_err[512] = "";
static std::atomic<uint64_t> g_launches{0};

void set_error(const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err, sizeof(g_err), fmt, ap);
  va_end(ap);
}

void count_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }

static uc_status cuda_check(const char* where) {
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) {
    set_error("%s: %s", where, cudaGetErrorString(e));
    return UC_ERR_CUDA;
  }
  return UC_OK;
}

static bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

// ------------------------------------------------------------ TMA encode
static PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// bf16 rows [rows, 128], box 64 columns x 64 rows, 128-byte swizzle.
static uc_status encode_rows(CUtensorMap* map, const void* base, int64_t rows) {
  auto fn = encode_fn();
  if (fn == nullptr) {
    set_error("cuTensorMapEncodeTiled is not available from the driver");
    return UC_ERR_CUDA;
  }
  if (!aligned(base, 16) || rows <= 0 || rows >= (int64_t(1) << 31)) {
    set_error("TMA rows: base must be 16-byte aligned and 0 < rows < 2^31");
    return UC_ERR_ARG;
  }
  cuuint64_t dims[2] = {(cuuint64_t)kHeadDim, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)kHeadDim * 2};
  cuuint32_t box[2] = {64, 64};
  cuuint32_t estr[2] = {1, 1};
  const CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides,
                        box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    set_error("cuTensorMapEncodeTiled failed (%d)", (int)r);
    return UC_ERR_CUDA;
  }
  return UC_OK;
}

// fp16 rows [rows, 128], box 64 columns x kDenseKeys rows, 128-byte swizzle.
static uc_status encode_rows_f16(CUtensorMap* map, const void* base, int64_t rows) {
  auto fn = encode_fn();
  if (fn == nullptr) {
    set_error("cuTensorMapEncodeTiled is not available from the driver");
    return UC_ERR_CUDA;
  }
  if (!aligned(base, 16) || rows <= 0 || rows >= (int64_t(1) << 31)) {
    set_error("TMA rows: base must be 16-byte aligned and 0 < rows < 2^31");
    return UC_ERR_ARG;
  }
  cuuint64_t dims[2] = {(cuuint64_t)kHeadDim, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)kHeadDim * 2};
  cuuint32_t box[2] = {64, (cuuint32_t)kDenseKeys};
  cuuint32_t estr[2] = {1, 1};
  const CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void*>(base), dims, strides, box,
                        estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    set_error("cuTensorMapEncodeTiled (fp16) failed (%d)", (int)r);
    return UC_ERR_CUDA;
  }
  return UC_OK;
}

// Tensor maps of a segment's bf16 rows, cached inside the segment struct.
static uc_status segment_maps(const uc_segment* seg, CUtensorMap* mk, CUtensorMap* mv) {
  const uint64_t key = reinterpret_cast<uint64_t>(seg->k) * 1000003ull ^
                       reinterpret_cast<uint64_t>(seg->v) * 998244353ull ^ (uint64_t)seg->rows_total * 7ull ^
                       0x5a17ull;
  uc_segment* s = const_cast<uc_segment*>(seg);
  if (s->cache_key != key) {
    CUtensorMap a, b;
    uc_status st = encode_rows(&a, seg->k, seg->rows_total);
    if (st != UC_OK) return st;
    st = encode_rows(&b, seg->v, seg->rows_total);
    if (st != UC_OK) return st;
    memcpy(s->cache, &a, sizeof(CUtensorMap));
    memcpy(s->cache + sizeof(CUtensorMap), &b, sizeof(CUtensorMap));
    s->cache_key = key;
  }
  memcpy(mk, s->cache, sizeof(CUtensorMap));
  memcpy(mv, s->cache + sizeof(CUtensorMap), sizeof(CUtensorMap));
  return UC_OK;
}

static int num_sms() {
  static int n = 0;
  if (n == 0) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (n <= 0) n = 1;
  }
  return n;
}

static bool is_quant(int kind) { return kind == UC_KIND_QUANT || kind == UC_KIND_EVICT_QUANT; }

// Validates the descriptor of a segment (storage pointers included).
static uc_status check_segment(const uc_segment* s, const char* fn) {
  if (s == nullptr) {
    set_error("%s: null segment", fn);
    return UC_ERR_ARG;
  }
  if (s->kind < UC_KIND_FULL || s->kind > UC_KIND_EVICT_QUANT) {
    set_error("%s: bad segment kind %d", fn, s->kind);
    return UC_ERR_ARG;
  }
  if (s->head_dim != UC_HEAD_DIM || s->batch < 1 || s->batch > UC_MAX_BATCH || s->n_kv_heads < 1 ||
      s->n_kv_heads > 8 || s->n_src < 0 || s->cap < 0) {
    set_error("%s: unsupported segment shape (head_dim %d, batch %d, kv heads %d)", fn, s->head_dim,
              s->batch, s->n_kv_heads);
    return UC_ERR_SHAPE;
  }
  if (s->n_kept == nullptr || !aligned(s->n_kept, 4)) {
    set_error("%s: n_kept must be a device int32 array", fn);
    return UC_ERR_ARG;
  }
  if (is_quant(s->kind)) {
    if ((s->bits != 4 && s->bits != 2) || s->cap % 64 != 0) {
      set_error("%s: quantized segments need bits 4 or 2 and cap % 64 == 0", fn);
      return UC_ERR_SHAPE;
    }
    const void* ptrs[] = {s->k_codes, s->k_params, s->v_codes, s->v_params, s->k, s->v};
    for (const void* p : ptrs)
      if (p == nullptr || !aligned(p, 16)) {
        set_error("%s: quantized segment arrays must be non-null and 16-byte aligned", fn);
        return UC_ERR_ARG;
      }
    if (s->kept_idx == nullptr) {
      set_error("%s: quantized segments need kept_idx", fn);
      return UC_ERR_ARG;
    }
    if (s->row_stride != UC_GROUP || s->row_offset != 0 ||
        s->rows_total < (int64_t)s->batch * s->n_kv_heads * UC_GROUP) {
      set_error("%s: the tail of a quantized segment is 32 rows per (b, kvh)", fn);
      return UC_ERR_SHAPE;
    }
  } else {
    if (s->bits != 16) {
      set_error("%s: bf16 segments have bits = 16", fn);
      return UC_ERR_SHAPE;
    }
    if (s->k == nullptr || s->v == nullptr || !aligned(s->k, 16) || !aligned(s->v, 16)) {
      set_error("%s: k / v must be non-null and 16-byte aligned", fn);
      return UC_ERR_ARG;
    }
    if (s->row_stride < 0 || s->row_offset < 0) {
      set_error("%s: negative row stride / offset", fn);
      return UC_ERR_SHAPE;
    }
    if (s->kind == UC_KIND_EVICT && s->kept_idx == nullptr) {
      set_error("%s: EVICT segments need kept_idx", fn);
      return UC_ERR_ARG;
    }
  }
  for (int b = 0; b < s->batch; ++b) {
    const int n = s->n_kept_host[b];
    if (n < 0 || (s->kind != UC_KIND_FULL && n > s->cap)) {
      set_error("%s: n_kept[%d] = %d outside [0, cap = %d]", fn, b, n, s->cap);
      return UC_ERR_SHAPE;
    }
    if (!is_quant(s->kind)) {
      const int64_t last = ((int64_t)(b + 1) * s->n_kv_heads - 1) * s->row_stride + s->row_offset + n;
      if (n > 0 && last > s->rows_total) {
        set_error("%s: rows of sequence %d run past rows_total", fn, b);
        return UC_ERR_SHAPE;
      }
    }
  }
  return UC_OK;
}

}  // namespace uc

using namespace uc;

extern "C" {

const char* uc_last_error(void) { return g_err; }

int32_t uc_version(void) { return 1; }

uint64_t uc_launch_count(void) { return g_launches.load(); }

static std::atomic<int32_t> g_dense_serial_pv{1};
static std::atomic<uint64_t> g_wait_limit_ns{2000000000ull};
static std::atomic<int32_t> g_withhold{-1};
static std::atomic<int32_t> g_pdl{0};

int32_t uc_set_dense_serial_pv(int32_t serial) {
  UC_TRACE();
  return g_dense_serial_pv.exchange(serial != 0 ? 1 : 0);
}

uint64_t uc_set_wait_limit(uint64_t ns) {
  UC_TRACE();
  return g_wait_limit_ns.exchange(ns == 0 ? 2000000000ull : ns);
}

void uc_debug_withhold_tile(int32_t pos) {
  UC_TRACE();
  g_withhold.store(pos < 0 ? -1 : pos);
}

int32_t uc_set_programmatic_launch(int32_t on) {
  UC_TRACE();
  return g_pdl.exchange(on != 0 ? 1 : 0);
}

uc_status uc_workspace_status(void* workspace, void* stream) {
  UC_TRACE();
  if (workspace == nullptr) {
    set_error("uc_workspace_status: null workspace");
    return UC_ERR_ARG;
  }
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  DevStatus h{};
  if (cudaMemcpyAsync(&h, workspace, sizeof(h), cudaMemcpyDeviceToHost, st) != cudaSuccess ||
      cudaStreamSynchronize(st) != cudaSuccess)
    return cuda_check("uc_workspace_status");
  if (h.code != 0) {
    set_error("device reported status %d (detail %d)", h.code, h.detail);
    DevStatus z{};
    cudaMemcpyAsync(workspace, &z, sizeof(z), cudaMemcpyHostToDevice, st);
    cudaStreamSynchronize(st);
    return (uc_status)h.code;
  }
  return UC_OK;
}

uc_status uc_segment_sizes_of(const uc_segment* s, uc_segment_sizes* o) {
  UC_TRACE();
  if (s == nullptr || o == nullptr) {
    set_error("uc_segment_sizes_of: null argument");
    return UC_ERR_ARG;
  }
  if (s->batch < 1 || s->batch > UC_MAX_BATCH || s->n_kv_heads < 1 || s->cap < 0 ||
      (is_quant(s->kind) && (s->cap % 64 || (s->bits != 4 && s->bits != 2)))) {
    set_error("uc_segment_sizes_of: unsupported shape");
    return UC_ERR_SHAPE;
  }
  memset(o, 0, sizeof(*o));
  const uint64_t bh = (uint64_t)s->batch * s->n_kv_heads;
  o->n_kept = 4ull * s->batch;
  if (s->kind != UC_KIND_FULL) o->kept_idx = 4ull * bh * s->cap;
  if (is_quant(s->kind)) {
    o->k = o->v = bh * UC_GROUP * UC_HEAD_DIM * 2;
    o->k_codes = o->v_codes = bh * s->cap * UC_HEAD_DIM * s->bits / 8;
    o->k_params = bh * (s->cap / UC_GROUP) * 512;
    o->v_params = bh * s->cap * 16;
  } else if (s->kind == UC_KIND_EVICT) {
    o->k = o->v = bh * s->cap * UC_HEAD_DIM * 2;
  }
  return UC_OK;
}

// ------------------------------------------------------------------ scores

static int score_mtiles(int rows) { return (rows + 15) / 16; }

// One CTA per SM (tensor memory and shared memory), 128-key tiles: about one
// chunk of keys per SM over all (b, kvh).
static void score_plan(int batch, int hkv, int n_ctx, int* chunks, int* tiles_per_chunk) {
  const int bh = batch * hkv;
  const int n_tiles = (n_ctx + 127) / 128;
  const int sms = num_sms();
  // the fewest chunks per (b, kvh) that keep >= 90 % of the SMs busy in
  // every wave of CTAs (one CTA per SM), else the best fill up to 4 waves
  int c_best = 1;
  double best = -1.0;
  for (int c = 1; c <= std::min(n_tiles, 4 * ((sms + bh - 1) / bh)); ++c) {
    const int tpc = (n_tiles + c - 1) / c;
    const int cc = (n_tiles + tpc - 1) / tpc;  // chunks actually formed
    const double tot = (double)bh * cc;
    const double eff = tot / (std::ceil(tot / sms) * sms);
    if (eff >= 0.9) {
      c_best = c;
      break;
    }
    if (eff > best + 1e-9) {
      best = eff;
      c_best = c;
    }
  }
  *tiles_per_chunk = (n_tiles + c_best - 1) / c_best;
  *chunks = (n_tiles + *tiles_per_chunk - 1) / *tiles_per_chunk;
}

size_t uc_score_workspace_size(int32_t batch, int32_t n_q_heads, int32_t n_kv_heads, int32_t window,
                               int32_t n_ctx) {
  UC_TRACE();
  if (batch <= 0 || n_kv_heads <= 0 || n_q_heads <= 0 || window <= 0 || n_ctx <= 0) return 0;
  const int rows = n_q_heads / n_kv_heads * window;
  int chunks, tpc;
  score_plan(batch, n_kv_heads, n_ctx, &chunks, &tpc);
  const size_t rows_pad = 16 * (size_t)score_mtiles(rows);
  const size_t bh = (size_t)batch * n_kv_heads;
  return 256 + bh * chunks * rows_pad * 2 * 4 + bh * rows_pad * 4;
}

uc_status uc_score_accumulate(const void* qwin, const void* k, int32_t batch, int32_t n_q_heads,
                              int32_t n_kv_heads, int32_t window, int32_t n_ctx, int64_t k_row_stride,
                              float* scores, void* workspace, size_t workspace_bytes, void* stream) {
  UC_TRACE();
  if (qwin == nullptr || k == nullptr || scores == nullptr || workspace == nullptr ||
      !aligned(qwin, 16) || !aligned(k, 16) || !aligned(scores, 4) || !aligned(workspace, 16)) {
    set_error("uc_score_accumulate: null or misaligned pointer");
    return UC_ERR_ARG;
  }
  if (batch < 1 || n_kv_heads < 1 || n_q_heads % n_kv_heads != 0 || window < 1 || n_ctx < 1 ||
      k_row_stride < n_ctx) {
    set_error("uc_score_accumulate: bad sizes");
    return UC_ERR_SHAPE;
  }
  const int rows = n_q_heads / n_kv_heads * window;
  if (rows > 256) {
    set_error("uc_score_accumulate: (Hq / Hkv) * W = %d exceeds 256", rows);
    return UC_ERR_SHAPE;
  }
  const size_t need = uc_score_workspace_size(batch, n_q_heads, n_kv_heads, window, n_ctx);
  if (workspace_bytes < need) {
    set_error("uc_score_accumulate: workspace %zu < %zu bytes", workspace_bytes, need);
    return UC_ERR_OOM;
  }
  ScoreArgs a;
  memset(&a, 0, sizeof(a));
  const int64_t rows_total = (int64_t)batch * n_kv_heads * k_row_stride;
  uc_status st = encode_rows(&a.tmap_k, k, rows_total);
  if (st != UC_OK) return st;
  a.qwin = static_cast<const __nv_bfloat16*>(qwin);
  a.scores = scores;
  a.status = static_cast<DevStatus*>(workspace);
  a.batch = batch;
  a.n_q_heads = n_q_heads;
  a.n_kv_heads = n_kv_heads;
  a.window = window;
  a.n_ctx = n_ctx;
  a.k_row_stride = k_row_stride;
  a.rows = rows;
  a.mtiles = score_mtiles(rows);
  score_plan(batch, n_kv_heads, n_ctx, &a.chunks, &a.tiles_per_chunk);
  const size_t rows_pad = 16 * (size_t)a.mtiles;
  a.part = reinterpret_cast<float*>(static_cast<uint8_t*>(workspace) + 256);
  a.lse2 = a.part + (size_t)batch * n_kv_heads * a.chunks * rows_pad * 2;
  a.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)UC_HEAD_DIM));
  launch_scores(a, reinterpret_cast<cudaStream_t>(stream));
  return cuda_check("uc_score_accumulate");
}

uc_status uc_segment_mass(const float* scores, int32_t batch, int32_t n_kv_heads, int32_t n_ctx,
                          const int32_t* begin, const int32_t* end, int32_t n_seg, int32_t n_q_heads,
                          int32_t window, float weight, int32_t accumulate, float* mass, void* stream) {
  UC_TRACE();
  if (scores == nullptr || begin == nullptr || end == nullptr || mass == nullptr) {
    set_error("uc_segment_mass: null pointer");
    return UC_ERR_ARG;
  }
  if (batch < 1 || n_kv_heads < 1 || n_ctx < 1 || n_seg < 1 || n_seg > UC_MAX_SEGMENTS ||
      n_q_heads < 1 || window < 1) {
    set_error("uc_segment_mass: bad sizes");
    return UC_ERR_SHAPE;
  }
  for (int s = 0; s < n_seg; ++s)
    if (begin[s] < 0 || end[s] < begin[s] || end[s] > n_ctx) {
      set_error("uc_segment_mass: segment %d range [%d, %d) outside [0, %d)", s, begin[s], end[s], n_ctx);
      return UC_ERR_SHAPE;
    }
  if (!std::isfinite(weight)) {
    set_error("uc_segment_mass: weight must be finite");
    return UC_ERR_ARG;
  }
  launch_segment_mass(scores, batch, n_kv_heads, n_ctx, begin, end, n_seg,
                      (float)((double)weight / ((double)n_q_heads * window)), accumulate != 0, mass,
                      reinterpret_cast<cudaStream_t>(stream));
  return cuda_check("uc_segment_mass");
}

uc_status uc_attention_mass(const float* mass, int32_t batch, int32_t n_q_heads, int32_t n_qtok,
                            int32_t n_seg, float weight, int32_t accumulate, float* out, void* stream) {
  UC_TRACE();
  if (mass == nullptr || out == nullptr) {
    set_error("uc_attention_mass: null pointer");
    return UC_ERR_ARG;
  }
  if (batch < 1 || batch > UC_MAX_BATCH || n_q_heads < 1 || n_qtok < 1 || n_seg < 1 ||
      n_seg > UC_MAX_SEGMENTS || (int64_t)n_q_heads * n_qtok > INT32_MAX / UC_MAX_SEGMENTS) {
    set_error("uc_attention_mass: bad sizes");
    return UC_ERR_SHAPE;
  }
  if (!std::isfinite(weight)) {
    set_error("uc_attention_mass: weight must be finite");
    return UC_ERR_ARG;
  }
  const int rows = n_q_heads * n_qtok;
  launch_attention_mass(mass, batch, rows, n_seg, (float)((double)weight / rows), accumulate != 0, out,
                        reinterpret_cast<cudaStream_t>(stream));
  return cuda_check("uc_attention_mass");
}

uc_status uc_accumulate_scores(const void* q, int32_t n_q_heads, int32_t n_qtok, const uc_segment* seg,
                               const float* lse, float* acc, int64_t acc_stride, int64_t acc_offset,
                               void* workspace, size_t workspace_bytes, void* stream) {
  UC_TRACE();
  uc_status st = check_segment(seg, "uc_accumulate_scores");
  if (st != UC_OK) return st;
  if (seg->kind != UC_KIND_FULL && seg->kind != UC_KIND_EVICT) {
    set_error("uc_accumulate_scores: heavy-hitter statistics are kept for bf16 (FULL / EVICT) segments");
    return UC_ERR_ARG;
  }
  if (q == nullptr || lse == nullptr || acc == nullptr || !aligned(q, 16) || !aligned(acc, 4) ||
      workspace == nullptr || workspace_bytes < 256 || !aligned(workspace, 16)) {
    set_error("uc_accumulate_scores: null or misaligned argument / workspace < 256 bytes");
    return UC_ERR_ARG;
  }
  const int hkv = seg->n_kv_heads;
  if (n_qtok < 1 || n_qtok > UC_MAX_QTOKENS || n_q_heads < hkv || n_q_heads % hkv ||
      (n_q_heads / hkv) * n_qtok > UC_MAX_QTOKENS * 8 || acc_offset < 0 || acc_stride <= acc_offset) {
    set_error("uc_accumulate_scores: bad query shape or accumulator extent");
    return UC_ERR_SHAPE;
  }
  int max_n = 0;
  for (int b = 0; b < seg->batch; ++b) max_n = std::max(max_n, seg->n_kept_host[b]);
  if (seg->kind != UC_KIND_FULL && seg->cap > max_n) max_n = seg->cap;  // device counts may run ahead
  DecodeScoreArgs a;
  memset(&a, 0, sizeof(a));
  a.q = static_cast<const __nv_bfloat16*>(q);
  a.lse = lse;
  a.k = static_cast<const __nv_bfloat16*>(seg->k);
  a.row_stride = seg->row_stride;
  a.row_offset = seg->row_offset;
  a.kept_idx = seg->kind == UC_KIND_FULL ? nullptr : seg->kept_idx;
  a.n_kept = seg->n_kept;
  a.acc = acc;
  a.acc_stride = acc_stride;
  a.acc_offset = acc_offset;
  a.status = static_cast<DevStatus*>(workspace);
  a.cap = seg->cap;
  a.n_kv_heads = hkv;
  a.n_q_heads = n_q_heads;
  a.n_qtok = n_qtok;
  a.group = n_q_heads / hkv;
  a.rows = a.group * n_qtok;
  a.scale = (float)(1.0 / std::sqrt((double)UC_HEAD_DIM));
  launch_decode_scores(a, seg->batch, max_n, reinterpret_cast<cudaStream_t>(stream));
  return cuda_check("uc_accumulate_scores");
}

// ------------------------------------------------------------- compression

size_t uc_compress_workspace_size(const uc_segment* seg) {
  UC_TRACE();
  (void)seg;
  return 256;
}

uc_status uc_compress_segment(const void* k_src, const void* v_src, int64_t src_row_stride,
                              int64_t src_row_offset, const float* scores, int64_t scores_stride,
                              int64_t scores_offset, int32_t n_recent, uc_segment* seg, void* workspace,
                              size_t workspace_bytes, void* stream) {
  UC_TRACE();
  uc_status st = check_segment(seg, "uc_compress_segment");
  if (st != UC_OK) return st;
  if (seg->kind == UC_KIND_FULL) {
    set_error("uc_compress_segment: FULL segments are views, there is nothing to compress");
    return UC_ERR_ARG;
  }
  if (k_src == nullptr || v_src == nullptr || !aligned(k_src, 16) || !aligned(v_src, 16) ||
      workspace == nullptr || !aligned(workspace, 16)) {
    set_error("uc_compress_segment: null or misaligned source / workspace");
    return UC_ERR_ARG;
  }
  if (workspace_bytes < uc_compress_workspace_size(seg)) {
    set_error("uc_compress_segment: workspace too small");
    return UC_ERR_OOM;
  }
  const bool evict = seg->kind == UC_KIND_EVICT || seg->kind == UC_KIND_EVICT_QUANT;
  if (evict && (scores == nullptr || scores_stride < seg->n_src || scores_offset < 0)) {
    set_error("uc_compress_segment: eviction needs a score array covering n_src tokens");
    return UC_ERR_ARG;
  }
  if (src_row_stride < seg->n_src + src_row_offset || src_row_offset < 0 || n_recent < 0) {
    set_error("uc_compress_segment: bad source rows");
    return UC_ERR_SHAPE;
  }
  int max_keep = 0;
  for (int b = 0; b < seg->batch; ++b) {
    const int keep = seg->n_kept_host[b];
    if (keep > seg->n_src || keep > seg->cap || (evict && keep < 1) ||
        (!evict && keep != seg->n_src)) {
      set_error("uc_compress_segment: keep[%d] = %d invalid (n_src %d, cap %d)", b, keep, seg->n_src,
                seg->cap);
      return UC_ERR_BUDGET;
    }
    max_keep = std::max(max_keep, keep);
  }
  cudaStream_t cs = reinterpret_cast<cudaStream_t>(stream);
  const int nbh = seg->batch * seg->n_kv_heads;
  DevStatus* dst = static_cast<DevStatus*>(workspace);

  TopkArgs t;
  memset(&t, 0, sizeof(t));
  t.scores = scores;
  t.scores_stride = scores_stride;
  t.scores_offset = scores_offset;
  t.kept_idx = seg->kept_idx;
  t.n_kept = seg->n_kept;
  t.status = dst;
  t.n_kv_heads = seg->n_kv_heads;
  t.n_src = seg->n_src;
  t.n_recent = n_recent;
  t.cap = seg->cap;
  for (int b = 0; b < seg->batch; ++b) {
    t.keep[b] = seg->n_kept_host[b];
    t.src_n[b] = seg->n_src;
  }
  launch_topk(t, nbh, evict, cs);

  GatherArgs g;
  memset(&g, 0, sizeof(g));
  g.k_src = static_cast<const __nv_bfloat16*>(k_src);
  g.v_src = static_cast<const __nv_bfloat16*>(v_src);
  g.src_row_stride = src_row_stride;
  g.src_row_offset = src_row_offset;
  g.kept_idx = seg->kept_idx;
  g.k_dst = static_cast<__nv_bfloat16*>(seg->k);
  g.v_dst = static_cast<__nv_bfloat16*>(seg->v);
  g.dst_row_stride = seg->row_stride;
  g.dst_row_offset = seg->row_offset;
  g.k_codes = static_cast<uint8_t*>(seg->k_codes);
  g.k_params = static_cast<uint8_t*>(seg->k_params);
  g.v_codes = static_cast<uint8_t*>(seg->v_codes);
  g.v_params = static_cast<uint8_t*>(seg->v_params);
  g.status = dst;
  g.batch = seg->batch;
  g.n_kv_heads = seg->n_kv_heads;
  g.cap = seg->cap;
  g.wait_ns = uc::wait_limit_ns();
  for (int b = 0; b < seg->batch; ++b) g.keep[b] = seg->n_kept_host[b];
  g.withhold = -1;
  if (is_quant(seg->kind)) {
    g.max_chunks = std::max(1, max_keep / UC_GROUP);
    g.withhold = uc::take_withhold_pos();
    launch_quantize(g, seg->bits, cs);
  } else {
    g.max_chunks = std::max(1, (max_keep + 31) / 32);
    launch_gather(g, cs);
  }
  return cuda_check("uc_compress_segment");
}

size_t uc_recompress_workspace_size(const uc_segment* src, const uc_segment* dst) {
  UC_TRACE();
  (void)dst;
  if (src == nullptr) return 256;
  size_t n = 256;
  if (is_quant(src->kind))  // rebuilt bf16 K and V rows of every (b, kvh) block
    n += 2 * (size_t)src->batch * src->n_kv_heads * src->cap * UC_HEAD_DIM * 2;
  return n;
}

uc_status uc_recompress_segment(const uc_segment* src, const float* scores, int64_t scores_stride,
                                int64_t scores_offset, int32_t n_recent, uc_segment* dst,
                                void* workspace, size_t workspace_bytes, void* stream) {
  UC_TRACE();
  uc_status st = check_segment(src, "uc_recompress_segment (src)");
  if (st != UC_OK) return st;
  st = check_segment(dst, "uc_recompress_segment (dst)");
  if (st != UC_OK) return st;
  if (dst->kind == UC_KIND_FULL) {
    set_error("uc_recompress_segment: the destination must be a compressed kind");
    return UC_ERR_ARG;
  }
  if (src == dst || src->kept_idx == dst->kept_idx || src->k == dst->k || src->v == dst->v ||
      (is_quant(src->kind) && is_quant(dst->kind) && src->k_codes == dst->k_codes)) {
    set_error("uc_recompress_segment: source and destination must not share storage");
    return UC_ERR_ARG;
  }
  if (src->batch != dst->batch || src->n_kv_heads != dst->n_kv_heads) {
    set_error("uc_recompress_segment: source and destination differ in batch or kv heads");
    return UC_ERR_SHAPE;
  }
  if (workspace == nullptr || !aligned(workspace, 16) ||
      workspace_bytes < uc_recompress_workspace_size(src, dst)) {
    set_error("uc_recompress_segment: null, misaligned or too small workspace");
    return UC_ERR_OOM;
  }
  const bool evict = dst->kind == UC_KIND_EVICT || dst->kind == UC_KIND_EVICT_QUANT;
  if (evict && (scores == nullptr || scores_offset < 0 || scores_stride <= scores_offset)) {
    set_error("uc_recompress_segment: eviction needs a score array");
    return UC_ERR_ARG;
  }
  if (n_recent < 0) {
    set_error("uc_recompress_segment: n_recent < 0");
    return UC_ERR_ARG;
  }
  int max_keep = 0, max_src = 0;
  for (int b = 0; b < dst->batch; ++b) {
    const int have = src->n_kept_host[b], keep = dst->n_kept_host[b];
    if (have < 0 || have > src->cap) {
      set_error("uc_recompress_segment: source n_kept[%d] = %d out of range", b, have);
      return UC_ERR_SHAPE;
    }
    if (keep < 0 || keep > have || keep > dst->cap || (!evict && keep != have)) {
      set_error("uc_recompress_segment: keep[%d] = %d invalid (source holds %d, cap %d)", b, keep, have,
                dst->cap);
      return UC_ERR_BUDGET;
    }
    max_keep = std::max(max_keep, keep);
    max_src = std::max(max_src, have);
  }
  cudaStream_t cs = reinterpret_cast<cudaStream_t>(stream);
  const int nbh = dst->batch * dst->n_kv_heads;
  DevStatus* dstat = static_cast<DevStatus*>(workspace);

  // 1. source rows as bf16: the segment's own rows, or packed groups rebuilt.
  const __nv_bfloat16* k_rows;
  const __nv_bfloat16* v_rows;
  int64_t rows_stride, rows_offset;
  if (is_quant(src->kind)) {
    __nv_bfloat16* kr = reinterpret_cast<__nv_bfloat16*>(static_cast<uint8_t*>(workspace) + 256);
    __nv_bfloat16* vr = kr + (size_t)nbh * src->cap * UC_HEAD_DIM;
    DequantArgs d;
    memset(&d, 0, sizeof(d));
    d.k_codes = static_cast<const uint8_t*>(src->k_codes);
    d.k_params = static_cast<const uint8_t*>(src->k_params);
    d.v_codes = static_cast<const uint8_t*>(src->v_codes);
    d.v_params = static_cast<const uint8_t*>(src->v_params);
    d.k_tail = static_cast<const __nv_bfloat16*>(src->k);
    d.v_tail = static_cast<const __nv_bfloat16*>(src->v);
    d.n_kept = src->n_kept;
    d.k_out = kr;
    d.v_out = vr;
    d.batch = src->batch;
    d.n_kv_heads = src->n_kv_heads;
    d.cap = src->cap;
    d.bits = src->bits;
    d.max_groups = (max_src + UC_GROUP - 1) / UC_GROUP;
    if (d.max_groups > 0) launch_dequant_rows(d, cs);
    k_rows = kr;
    v_rows = vr;
    rows_stride = src->cap;
    rows_offset = 0;
  } else {
    k_rows = static_cast<const __nv_bfloat16*>(src->k);
    v_rows = static_cast<const __nv_bfloat16*>(src->v);
    rows_stride = src->row_stride;
    rows_offset = src->row_offset;
  }

  // 2. rows to keep, as indices into the source's stored rows.
  TopkArgs t;
  memset(&t, 0, sizeof(t));
  t.scores = scores;
  t.scores_stride = scores_stride;
  t.scores_offset = scores_offset;
  t.kept_idx = dst->kept_idx;
  t.n_kept = dst->n_kept;
  t.status = dstat;
  t.n_kv_heads = dst->n_kv_heads;
  t.n_src = src->n_src;
  t.n_recent = n_recent;
  t.cap = dst->cap;
  t.score_idx = src->kept_idx;  // NULL for FULL sources: stored row i is token i
  t.score_idx_stride = src->cap;
  t.score_limit = scores_stride - scores_offset;
  for (int b = 0; b < dst->batch; ++b) {
    t.keep[b] = dst->n_kept_host[b];
    t.src_n[b] = src->n_kept_host[b];
  }
  launch_topk(t, nbh, evict, cs);

  // 3. gather or quantize the kept rows into the destination.
  GatherArgs g;
  memset(&g, 0, sizeof(g));
  g.k_src = k_rows;
  g.v_src = v_rows;
  g.src_row_stride = rows_stride;
  g.src_row_offset = rows_offset;
  g.kept_idx = dst->kept_idx;
  g.k_dst = static_cast<__nv_bfloat16*>(dst->k);
  g.v_dst = static_cast<__nv_bfloat16*>(dst->v);
  g.dst_row_stride = dst->row_stride;
  g.dst_row_offset = dst->row_offset;
  g.k_codes = static_cast<uint8_t*>(dst->k_codes);
  g.k_params = static_cast<uint8_t*>(dst->k_params);
  g.v_codes = static_cast<uint8_t*>(dst->v_codes);
  g.v_params = static_cast<uint8_t*>(dst->v_params);
  g.status = dstat;
  g.batch = dst->batch;
  g.n_kv_heads = dst->n_kv_heads;
  g.cap = dst->cap;
  g.wait_ns = uc::wait_limit_ns();
  for (int b = 0; b < dst->batch; ++b) g.keep[b] = dst->n_kept_host[b];
  g.withhold = -1;
  if (is_quant(dst->kind)) {
    g.max_chunks = std::max(1, max_keep / UC_GROUP);
    g.withhold = uc::take_withhold_pos();
    launch_quantize(g, dst->bits, cs);
  } else {
    g.max_chunks = std::max(1, (max_keep + 31) / 32);
    launch_gather(g, cs);
  }

  // 4. stored-row indices -> the source's logical token indices.
  if (src->kept_idx != nullptr) {
    ComposeArgs c;
    c.kept_idx = dst->kept_idx;
    c.src_idx = src->kept_idx;
    c.n_kept = dst->n_kept;
    c.n_kv_heads = dst->n_kv_heads;
    c.cap = dst->cap;
    c.src_cap = src->cap;
    launch_compose_idx(c, nbh, cs);
  }
  return cuda_check("uc_recompress_segment");
}

// --------------------------------------------------------------- attention

namespace {

struct AttnPlan {
  int items_per_bh, n_items, grid, mtiles, n_heavy, n_light;
  int chunk_begin[UC_MAX_SEGMENTS], n_chunks[UC_MAX_SEGMENTS];
  int16_t heavy_local[128], light_local[2 * UC_MAX_SEGMENTS];
};

int groups_per_tile(int bits) { return bits == 2 ? 8 : 4; }

// Many items per (sequence, KV head) (a few long sequences): merge them in a
// kernel of their own, spread over many SMs (the in-launch merge of one
// (b, kvh) runs on one SM; 128K batch 2, 54 items: 10 us of a 55 us
// launch). Below 33 items the second launch costs more than it saves.
constexpr int kMergeKernelItems = 32;

int seg_tiles_host(const uc_segment* s, int n) {
  if (!is_quant(s->kind)) return (n + 63) / 64;
  const int ng = n / 32, tg = groups_per_tile(s->bits);
  return (ng + tg - 1) / tg + ((n % 32) ? 1 : 0);
}

double tile_bytes_host(const uc_segment* s) {
  if (!is_quant(s->kind)) return 32768.0;
  return groups_per_tile(s->bits) * (2.0 * 32 * 128 * s->bits / 8 + 1024);
}

// Stored bytes one (sequence, KV head) of a call streams (longest sequence).
double call_cost(const uc_segment* const* segs, int nseg) {
  double total = 0.0;
  for (int s = 0; s < nseg; ++s) {
    int mx = 0;
    for (int b = 0; b < segs[s]->batch; ++b) mx = std::max(mx, segs[s]->n_kept_host[b]);
    total += seg_tiles_host(segs[s], mx) * tile_bytes_host(segs[s]);
  }
  return total;
}

// nbh_launch: (sequence, KV head) pairs of every call sharing the launch.
// forced_ipb > 0 fixes the items per (sequence, KV head) instead of
// searching for the count that fills whole rounds of CTA slots.
// slots_in > 0: resident CTAs to plan for (no device query).
AttnPlan plan_attend(const uc_segment* const* segs, int nseg, int mtiles, int nbh_launch, int forced_ipb = 0,
                     int slots_in = 0) {
  AttnPlan p;
  memset(&p, 0, sizeof(p));
  p.mtiles = mtiles;
  const int B = segs[0]->batch, hkv = segs[0]->n_kv_heads;
  const int nbh = B * hkv;
  const int slots = slots_in > 0 ? slots_in : std::max(1, attend_ctas_per_sm(mtiles)) * num_sms();
  // heavy tiles of each segment (a packed segment's bf16 tail is a light
  // item of its own) and their bytes
  int htiles[UC_MAX_SEGMENTS];
  double tbytes[UC_MAX_SEGMENTS], hbytes[UC_MAX_SEGMENTS];
  bool heavy[UC_MAX_SEGMENTS];
  for (int s = 0; s < nseg; ++s) {
    int mx = 0;
    for (int b = 0; b < B; ++b) mx = std::max(mx, segs[s]->n_kept_host[b]);
    const int nt = seg_tiles_host(segs[s], mx);
    htiles[s] = is_quant(segs[s]->kind) ? nt - ((mx % UC_GROUP) ? 1 : 0) : nt;
    tbytes[s] = tile_bytes_host(segs[s]);
    hbytes[s] = htiles[s] * tbytes[s];
    heavy[s] = htiles[s] > 0;
  }
  // Heavy items per (b, kvh): the fewest (at least one per heavy segment, at
  // most 56 and at most 64 with the light items, the partials one merge
  // stages) that keep >= 90 % of the CTA slots busy in every round, else the
  // count with the best fill. Few long items amortise each item's start,
  // cross-warp reduction and split-K merge. A segment under half an average
  // heavy item (a few generated tokens next to a long context) becomes a
  // light item: as a heavy item of its own it would take an item from the
  // long segments and lengthen theirs; light items run last, on the CTAs
  // whose heavy items finished early.
  int H = 0;
  for (int pass = 0; pass <= nseg; ++pass) {
    int nh = 0, nl = 0;
    double tot = 0.0;
    for (int s = 0; s < nseg; ++s) {
      const bool q = is_quant(segs[s]->kind);
      if (heavy[s]) {
        ++nh;
        tot += hbytes[s];
        nl += q ? 1 : 0;
      } else {
        nl += (q && htiles[s] > 0) ? 2 : 1;
      }
    }
    const int hmax = std::max(nh, std::min(56, 64 - nl));
    H = forced_ipb;
    if (nh == 0) {
      H = 0;
    } else if (H <= 0) {
      double best_eff = -1.0;
      for (int h = nh; h <= hmax; ++h) {
        const double all = (double)h * nbh_launch;
        const double eff = all / (std::ceil(all / slots) * slots);
        if (eff >= 0.9) {
          H = h;
          break;
        }
        if (eff > best_eff + 1e-9) {
          best_eff = eff;
          H = h;
        }
      }
    }
    H = std::min(std::max(H, nh), hmax);
    // single-n-tile calls: items that the in-kernel merge stages in one
    // round trip, if they still keep >= 80 % of the slots busy (8K
    // understanding layer: 15 -> 14 items, 21.0 -> 19.5 us)
    if (mtiles == 1 && forced_ipb <= 0 && H + nl > kWholeMergeItems && kWholeMergeItems - nl >= nh) {
      const int hw = kWholeMergeItems - nl;
      const double all = (double)hw * nbh_launch;
      if (all / (std::ceil(all / slots) * slots) >= 0.8) H = hw;
    }
    // calls whose merge is the separate kernel: there an item costs no
    // merge work, so take the most heavy items that still start in the
    // first round (128K batch 2: 52 -> 56 heavy items, 50.3 -> 47.8 us)
    if (forced_ipb <= 0 && H + nl > kMergeKernelItems) {
      const int hr = std::min(hmax, slots / std::max(1, nbh_launch));
      if (hr > H) H = hr;
    }
    bool changed = false;
    for (int s = 0; s < nseg; ++s)
      if (heavy[s] && H > 0 && hbytes[s] < 0.5 * tot / H) {
        heavy[s] = false;
        changed = true;
      }
    if (!changed) break;
  }
  // split them among the heavy segments so that the largest item is
  // smallest (one more item at a time to the segment whose items are
  // largest). Where the launch merges its own partials, drop then the items
  // that do not shrink a segment's largest item: each would only bring its
  // start, cross-warp reduction and merge share (8K understanding layer: text
  // 8 tiles as 4 items of 2 instead of 5 items of 1-2, 13 items per (b, kvh)
  // instead of 14, 12694 -> 13221 tokens/s). With the separate merge kernel
  // an item is cheap and more of them even out the SMs' loads.
  int hc[UC_MAX_SEGMENTS], nh = 0;
  for (int s = 0; s < nseg; ++s) {
    hc[s] = heavy[s] ? 1 : 0;
    nh += hc[s];
  }
  for (int left = H - nh; left > 0; --left) {
    int pick = -1;
    double worst = 0.0;
    for (int s = 0; s < nseg; ++s) {
      if (!heavy[s] || hc[s] >= htiles[s]) continue;
      const double item = std::ceil((double)htiles[s] / hc[s]) * tbytes[s];
      if (item > worst) {
        worst = item;
        pick = s;
      }
    }
    if (pick < 0) break;
    ++hc[pick];
  }
  {
    int trimmed[UC_MAX_SEGMENTS], items = 0;
    for (int s = 0; s < nseg; ++s) {
      trimmed[s] = hc[s];
      if (heavy[s]) {
        const int per = (htiles[s] + hc[s] - 1) / hc[s];  // tiles of the segment's largest item
        trimmed[s] = (htiles[s] + per - 1) / per;          // the fewest items of at most that many
        items += hc[s] + (is_quant(segs[s]->kind) ? 1 : 0);
      } else {
        items += (is_quant(segs[s]->kind) && htiles[s] > 0) ? 2 : 1;
      }
    }
    if (items <= kMergeKernelItems)
      for (int s = 0; s < nseg; ++s) hc[s] = trimmed[s];
  }
  // chunks: a heavy segment's items (+ the tail of a packed one); a light
  // packed segment's packed tiles and its tail; a light bf16 segment whole
  int assigned = 0;
  for (int s = 0; s < nseg; ++s) {
    const bool q = is_quant(segs[s]->kind);
    if (heavy[s])
      p.n_chunks[s] = hc[s] + (q ? 1 : 0);
    else
      p.n_chunks[s] = (q && htiles[s] > 0) ? 2 : 1;
    assigned += p.n_chunks[s];
  }
  int cb = 0;
  for (int s = 0; s < nseg; ++s) {
    p.chunk_begin[s] = cb;
    for (int c = 0; c < p.n_chunks[s]; ++c) {
      const bool light = !heavy[s] || (is_quant(segs[s]->kind) && c == p.n_chunks[s] - 1);
      if (light)
        p.light_local[p.n_light++] = (int16_t)(cb + c);
      else
        p.heavy_local[p.n_heavy++] = (int16_t)(cb + c);
    }
    cb += p.n_chunks[s];
  }
  p.items_per_bh = assigned;  // at most 64 (the merge staging)
  p.n_items = assigned * nbh;
  p.grid = std::min(p.n_items, slots);
  return p;
}

}  // namespace

namespace {

// Dense calls: every segment's rows padded to kDenseKeys-key tiles; packed segments
// also get fp16 lo rows for their keys.
struct DensePlan {
  int n_tiles;
  int64_t rows_per_bh, lo_rows_per_bh;
  DenseTile tiles[kMaxDenseTiles];
};

bool plan_dense(const uc_segment* const* segs, int nseg, DensePlan* dp) {
  dp->n_tiles = 0;
  dp->rows_per_bh = dp->lo_rows_per_bh = 0;
  for (int s = 0; s < nseg; ++s) {
    int mx = 0;
    for (int b = 0; b < segs[s]->batch; ++b) mx = std::max(mx, segs[s]->n_kept_host[b]);
    const int nt = (mx + kDenseKeys - 1) / kDenseKeys;
    for (int t = 0; t < nt; ++t) {
      if (dp->n_tiles >= kMaxDenseTiles) return false;
      DenseTile& tl = dp->tiles[dp->n_tiles++];
      tl.row = (int32_t)(dp->rows_per_bh + kDenseKeys * t);
      tl.lo_row = is_quant(segs[s]->kind) ? (int32_t)(dp->lo_rows_per_bh + kDenseKeys * t) : -1;
      tl.seg = (int16_t)s;
      tl.seg_tile = (int16_t)t;
    }
    dp->rows_per_bh += (int64_t)kDenseKeys * nt;
    if (is_quant(segs[s]->kind)) dp->lo_rows_per_bh += (int64_t)kDenseKeys * nt;
  }
  return true;
}

// The dense path's rebuilt rows start past the status word, the decode work
// queue and the largest decode merge-counter block (UC_MAX_BATCH * 8 KV
// heads), so decode and dense calls may share one workspace.
constexpr size_t kDenseRowsOffset = 4096;

size_t dense_workspace(const DensePlan& dp, int nbh) {
  const size_t rows = (size_t)nbh * dp.rows_per_bh, lo = (size_t)nbh * dp.lo_rows_per_bh;
  return kDenseRowsOffset + 2 * rows * UC_HEAD_DIM * 2 + lo * UC_HEAD_DIM * 2 + 1024;
}

}  // namespace

namespace {

// Checks shared by uc_attend and uc_attend_batch.
uc_status check_call(const void* q, int32_t n_q_heads, int32_t n_qtok, const uc_segment* const* segs,
                     int32_t n_seg, const void* out, const char* name) {
  if (q == nullptr || out == nullptr || segs == nullptr || !aligned(q, 16) || !aligned(out, 16)) {
    set_error("%s: null or misaligned pointer", name);
    return UC_ERR_ARG;
  }
  if (n_seg < 1 || n_seg > UC_MAX_SEGMENTS || n_qtok < 1) {
    set_error("%s: need 1..%d segments and at least one query token", name, UC_MAX_SEGMENTS);
    return UC_ERR_SHAPE;
  }
  for (int s = 0; s < n_seg; ++s) {
    const uc_status st = check_segment(segs[s], name);
    if (st != UC_OK) return st;
    if (segs[s]->batch != segs[0]->batch || segs[s]->n_kv_heads != segs[0]->n_kv_heads) {
      set_error("%s: segments disagree on batch / KV heads", name);
      return UC_ERR_SHAPE;
    }
  }
  const int B = segs[0]->batch, hkv = segs[0]->n_kv_heads;
  if (n_q_heads < hkv || n_q_heads % hkv) {
    set_error("%s: query heads %d not a multiple of KV heads %d", name, n_q_heads, hkv);
    return UC_ERR_SHAPE;
  }
  for (int b = 0; b < B; ++b) {
    int64_t tot = 0;
    for (int s = 0; s < n_seg; ++s) tot += segs[s]->n_kept_host[b];
    if (tot <= 0) {
      set_error("%s: sequence %d has no cached tokens", name, b);
      return UC_ERR_SHAPE;
    }
  }
  return UC_OK;
}

int decode_mtiles(int n_q_heads, int hkv, int n_qtok) { return (n_q_heads / hkv * n_qtok + 7) / 8; }

int merge_kernel_for(int items_per_bh) { return items_per_bh > kMergeKernelItems ? 1 : 0; }

// A decode call's merge counters (one per (b, kvh)) live in a block of fixed
// size at a fixed place of the workspace, whatever the call's shape: every
// counter a call uses is re-armed to zero by its merge, so a block that calls
// of any layout share stays zero between calls (counters placed by the
// call's own layout could land on an earlier call's partial outputs).
constexpr size_t kCounterBlock = (size_t)UC_MAX_BATCH * 8 * 4;
static_assert(kCounterBlock % 256 == 0, "counter block alignment");

// Partial outputs of one decode call.
size_t decode_part_bytes(const uc_segment* const* segs, int n_seg, int mtiles, int nbh_launch,
                         int forced_ipb = 0) {
  const AttnPlan p = plan_attend(segs, n_seg, mtiles, nbh_launch, forced_ipb);
  return ((size_t)p.n_items * attend_part_floats(mtiles) * 4 + 255) / 256 * 256;
}

// Kernel parameters of one checked decode call whose counters start at
// `counters` (a kCounterBlock) and partial outputs at `parts`.
uc_status build_decode_call(const void* q, int32_t n_q_heads, int32_t n_qtok, const uc_segment* const* segs,
                            int32_t n_seg, void* out, float* lse, float* mass, int nbh_launch, int forced_ipb,
                            uint8_t* counters, uint8_t* parts, DevStatus* status, AttnParams* p,
                            AttnPlan* plan) {
  memset(p, 0, sizeof(*p));
  const int B = segs[0]->batch, hkv = segs[0]->n_kv_heads;
  const int group = n_q_heads / hkv;
  const int rows = group * n_qtok;
  const int mtiles = (rows + 7) / 8;
  *plan = plan_attend(segs, n_seg, mtiles, nbh_launch, forced_ipb);
  for (int s = 0; s < n_seg; ++s) {
    const uc_segment* sg = segs[s];
    SegDev& d = p->seg[s];
    d.kind = sg->kind;
    d.bits = sg->bits;
    d.cap = sg->cap;
    d.chunk_begin = plan->chunk_begin[s];
    d.n_chunks = plan->n_chunks[s];
    d.row_stride = sg->row_stride;
    d.row_offset = sg->row_offset;
    d.n_kept = sg->n_kept;
    d.k_codes = static_cast<const uint8_t*>(sg->k_codes);
    d.k_params = static_cast<const uint8_t*>(sg->k_params);
    d.v_codes = static_cast<const uint8_t*>(sg->v_codes);
    d.v_params = static_cast<const uint8_t*>(sg->v_params);
    const uc_status st = segment_maps(sg, &p->tmap[2 * s], &p->tmap[2 * s + 1]);
    if (st != UC_OK) return st;
  }
  const size_t nbh = (size_t)B * hkv;
  p->status = status;
  p->sched = reinterpret_cast<int32_t*>(reinterpret_cast<uint8_t*>(status) + 128);
  p->counters = reinterpret_cast<int32_t*>(counters);
  p->part = reinterpret_cast<float*>(parts);
  p->q = static_cast<const __nv_bfloat16*>(q);
  p->out = static_cast<__nv_bfloat16*>(out);
  p->lse = lse;
  p->mass = mass;
  p->nseg = n_seg;
  p->batch = B;
  p->n_kv_heads = hkv;
  p->n_q_heads = n_q_heads;
  p->n_qtok = n_qtok;
  p->group = group;
  p->rows = rows;
  p->mtiles = mtiles;
  p->items_per_bh = plan->items_per_bh;
  p->n_items = plan->n_items;
  p->n_heavy = plan->n_heavy;
  p->n_light = plan->n_light;
  for (int i = 0; i < plan->n_heavy; ++i) p->heavy_local[i] = plan->heavy_local[i];
  for (int i = 0; i < plan->n_light; ++i) p->light_local[i] = plan->light_local[i];
  p->scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)UC_HEAD_DIM));
  p->wait_ns = uc::wait_limit_ns();
  p->withhold_pos = uc::take_withhold_pos();
  return UC_OK;
}

// Items per (sequence, KV head) of each call of a batch: every call's items
// carry about the same number of bytes, about one item per CTA slot overall.
void batch_items(const uc_attend_call* calls, int n_calls, int mtiles, int* ipb) {
  const int slots = std::max(1, attend_ctas_per_sm(mtiles)) * num_sms();
  double cost[UC_MAX_CALLS], total = 0.0;
  for (int c = 0; c < n_calls; ++c) {
    cost[c] = call_cost(calls[c].segs, calls[c].n_seg);
    total += cost[c] * calls[c].segs[0]->batch * calls[c].segs[0]->n_kv_heads;
  }
  for (int c = 0; c < n_calls; ++c) {
    const int x = total > 0 ? (int)std::lround(slots * cost[c] / total) : 1;
    ipb[c] = std::max(calls[c].n_seg, std::min(56, x));
  }
}

}  // namespace
}  // extern "C"

namespace uc {

// Everything uc_attend checks before it looks at its workspace, in the same
// order and with the same statuses; *need receives the workspace bytes the
// call takes. Shared with uc_attend_static, which has no workspace.
size_t attend_counter_bytes() { return kCounterBlock; }

uc_status attend_precheck(const void* q, int32_t n_q_heads, int32_t n_qtok, const uc_segment* const* segs,
                          int32_t n_seg, const void* out, const char* name, size_t* need) {
  uc_status st = check_call(q, n_q_heads, n_qtok, segs, n_seg, out, name);
  if (st != UC_OK) return st;
  const int hkv = segs[0]->n_kv_heads;
  if (n_qtok > UC_MAX_QTOKENS) {
    static thread_local DensePlan dp;
    if (!plan_dense(segs, n_seg, &dp)) {
      set_error("%s: more than %d key tiles of %d", name, kMaxDenseTiles, kDenseKeys);
      return UC_ERR_SHAPE;
    }
    *need = dense_workspace(dp, segs[0]->batch * hkv);
    return UC_OK;
  }
  if (decode_mtiles(n_q_heads, hkv, n_qtok) > 8) {
    set_error("%s: (Hq / Hkv) * T = %d rows exceed 64", name, n_q_heads / hkv * n_qtok);
    return UC_ERR_SHAPE;
  }
  *need = 256 + kCounterBlock + decode_part_bytes(segs, n_seg, decode_mtiles(n_q_heads, hkv, n_qtok), segs[0]->batch * hkv);
  return UC_OK;
}

uint64_t wait_limit_ns() { return g_wait_limit_ns.load(); }
bool pdl_enabled() { return g_pdl.load() != 0; }
int take_withhold_pos() { return g_withhold.exchange(-1); }

}  // namespace uc

extern "C" {


size_t uc_attend_workspace_size(const uc_segment* const* segs, int32_t n_seg, int32_t n_q_heads,
                                int32_t n_qtok) {
  UC_TRACE();
  if (segs == nullptr || n_seg < 1 || n_seg > UC_MAX_SEGMENTS || segs[0] == nullptr || n_qtok < 1 ||
      n_q_heads < 1)
    return 0;
  if (n_qtok > UC_MAX_QTOKENS) {
    static thread_local DensePlan dp;
    if (!plan_dense(segs, n_seg, &dp)) return 0;
    return dense_workspace(dp, segs[0]->batch * segs[0]->n_kv_heads);
  }
  const int hkv = segs[0]->n_kv_heads;
  if (hkv < 1 || n_q_heads % hkv) return 0;
  const int mtiles = decode_mtiles(n_q_heads, hkv, n_qtok);
  return 256 + kCounterBlock + decode_part_bytes(segs, n_seg, mtiles, segs[0]->batch * hkv);
}

uc_status uc_attend_plan(const uc_segment* const* segs, int32_t n_seg, int32_t n_q_heads, int32_t n_qtok,
                         int32_t slots, uc_attend_plan_info* out) {
  UC_TRACE();
  if (segs == nullptr || out == nullptr) {
    set_error("uc_attend_plan: null pointer");
    return UC_ERR_ARG;
  }
  if (n_seg < 1 || n_seg > UC_MAX_SEGMENTS || n_qtok < 1 || n_qtok > UC_MAX_QTOKENS) {
    set_error("uc_attend_plan: need 1..%d segments and 1..%d query tokens", UC_MAX_SEGMENTS, UC_MAX_QTOKENS);
    return UC_ERR_SHAPE;
  }
  for (int s = 0; s < n_seg; ++s) {
    const uc_segment* g = segs[s];
    if (g == nullptr) {
      set_error("uc_attend_plan: segment %d is null", s);
      return UC_ERR_ARG;
    }
    const bool q = is_quant(g->kind);
    if (g->batch < 1 || g->batch > UC_MAX_BATCH || g->n_kv_heads < 1 || g->batch != segs[0]->batch ||
        g->n_kv_heads != segs[0]->n_kv_heads || g->kind < UC_KIND_FULL || g->kind > UC_KIND_EVICT_QUANT ||
        (q && g->bits != 2 && g->bits != 4)) {
      set_error("uc_attend_plan: segment %d has an invalid kind, width, batch or head count", s);
      return UC_ERR_SHAPE;
    }
    for (int b = 0; b < g->batch; ++b)
      if (g->n_kept_host[b] < 0) {
        set_error("uc_attend_plan: segment %d holds a negative count", s);
        return UC_ERR_SHAPE;
      }
  }
  const int hkv = segs[0]->n_kv_heads;
  if (n_q_heads < hkv || n_q_heads % hkv) {
    set_error("uc_attend_plan: query heads %d not a multiple of KV heads %d", n_q_heads, hkv);
    return UC_ERR_SHAPE;
  }
  const int mtiles = decode_mtiles(n_q_heads, hkv, n_qtok);
  if (mtiles > 8) {
    set_error("uc_attend_plan: (Hq / Hkv) * T = %d rows exceed 64", n_q_heads / hkv * n_qtok);
    return UC_ERR_SHAPE;
  }
  const AttnPlan p = plan_attend(segs, n_seg, mtiles, segs[0]->batch * hkv, 0, slots);
  memset(out, 0, sizeof(*out));
  out->items_per_bh = p.items_per_bh;
  out->n_heavy = p.n_heavy;
  out->n_light = p.n_light;
  out->grid = p.grid;
  out->merge_kernel = merge_kernel_for(p.items_per_bh);
  for (int s = 0; s < n_seg; ++s) {
    out->n_chunks[s] = p.n_chunks[s];
    bool any_heavy = false;
    for (int i = 0; i < p.n_heavy; ++i)
      any_heavy |= p.heavy_local[i] >= p.chunk_begin[s] && p.heavy_local[i] < p.chunk_begin[s] + p.n_chunks[s];
    out->light[s] = any_heavy ? 0 : 1;
  }
  return UC_OK;
}

uc_status uc_attend(const void* q, int32_t n_q_heads, int32_t n_qtok, const uc_segment* const* segs,
                    int32_t n_seg, void* out, float* lse, float* mass, void* workspace,
                    size_t workspace_bytes, void* stream) {
  UC_TRACE();
  if (workspace == nullptr || !aligned(workspace, 16)) {
    set_error("uc_attend: null or misaligned workspace");
    return UC_ERR_ARG;
  }
  size_t need_checked = 0;
  uc_status st = uc::attend_precheck(q, n_q_heads, n_qtok, segs, n_seg, out, "uc_attend", &need_checked);
  if (st != UC_OK) return st;
  const int B = segs[0]->batch, hkv = segs[0]->n_kv_heads;
  const int group = n_q_heads / hkv;
  if (n_qtok > UC_MAX_QTOKENS) {
    // many query tokens (denoising / editing): tensor-core dense path
    static thread_local DensePlan dp;
    if (!plan_dense(segs, n_seg, &dp)) {
      set_error("uc_attend: more than %d key tiles of %d", kMaxDenseTiles, kDenseKeys);
      return UC_ERR_SHAPE;
    }
    const int nbh = B * hkv;
    const size_t need = dense_workspace(dp, nbh);
    if (workspace_bytes < need) {
      set_error("uc_attend: workspace %zu < %zu bytes", workspace_bytes, need);
      return UC_ERR_OOM;
    }
    static thread_local DenseParams d;
    memset(&d, 0, sizeof(d));
    uint8_t* ws = static_cast<uint8_t*>(workspace);
    const size_t rows = (size_t)nbh * dp.rows_per_bh, lo = (size_t)nbh * dp.lo_rows_per_bh;
    d.status = reinterpret_cast<DevStatus*>(ws);
    d.khi = reinterpret_cast<__half*>(ws + kDenseRowsOffset);
    d.v = d.khi + rows * UC_HEAD_DIM;
    d.klo = d.v + rows * UC_HEAD_DIM;
    st = encode_rows_f16(&d.tmap_khi, d.khi, (int64_t)rows);
    if (st == UC_OK) st = encode_rows_f16(&d.tmap_v, d.v, (int64_t)rows);
    if (st == UC_OK) st = encode_rows_f16(&d.tmap_klo, lo > 0 ? (void*)d.klo : (void*)d.khi,
                                          (int64_t)(lo > 0 ? lo : rows));
    if (st != UC_OK) return st;
    for (int s = 0; s < n_seg; ++s) {
      const uc_segment* sg = segs[s];
      SegDev& sd = d.seg[s];
      sd.kind = sg->kind;
      sd.bits = sg->bits;
      sd.cap = sg->cap;
      sd.row_stride = sg->row_stride;
      sd.row_offset = sg->row_offset;
      sd.n_kept = sg->n_kept;
      sd.k_codes = static_cast<const uint8_t*>(sg->k_codes);
      sd.k_params = static_cast<const uint8_t*>(sg->k_params);
      sd.v_codes = static_cast<const uint8_t*>(sg->v_codes);
      sd.v_params = static_cast<const uint8_t*>(sg->v_params);
      d.seg_k[s] = static_cast<const __nv_bfloat16*>(sg->k);
      d.seg_v[s] = static_cast<const __nv_bfloat16*>(sg->v);
    }
    memcpy(d.tiles, dp.tiles, sizeof(DenseTile) * dp.n_tiles);
    d.n_tiles = dp.n_tiles;
    d.rows_per_bh = dp.rows_per_bh;
    d.lo_rows_per_bh = dp.lo_rows_per_bh;
    d.q = static_cast<const __nv_bfloat16*>(q);
    d.out = static_cast<__nv_bfloat16*>(out);
    d.lse = lse;
    d.mass = mass;
    d.nseg = n_seg;
    d.batch = B;
    d.n_kv_heads = hkv;
    d.n_q_heads = n_q_heads;
    d.n_qtok = n_qtok;
    d.group = group;
    d.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)UC_HEAD_DIM));
    d.serial_pv = g_dense_serial_pv.load();
    launch_dense(d, reinterpret_cast<cudaStream_t>(stream));
    return cuda_check("uc_attend (dense)");
  }
  const int mtiles = decode_mtiles(n_q_heads, hkv, n_qtok);
  if (mtiles > 8) {
    set_error("uc_attend: (Hq / Hkv) * T = %d rows exceed 64", group * n_qtok);
    return UC_ERR_SHAPE;
  }
  const size_t need = uc_attend_workspace_size(segs, n_seg, n_q_heads, n_qtok);
  if (workspace_bytes < need) {
    set_error("uc_attend: workspace %zu < %zu bytes", workspace_bytes, need);
    return UC_ERR_OOM;
  }
  static thread_local AttnParams p;
  AttnPlan plan;
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  st = build_decode_call(q, n_q_heads, n_qtok, segs, n_seg, out, lse, mass, B * hkv, 0, ws + 256,
                         ws + 256 + kCounterBlock, reinterpret_cast<DevStatus*>(ws), &p, &plan);
  if (st != UC_OK) return st;
  p.defer_merge = merge_kernel_for(plan.items_per_bh);
  launch_attend(p, plan.grid, reinterpret_cast<cudaStream_t>(stream));
  return cuda_check("uc_attend");
}

size_t uc_attend_batch_workspace_size(const uc_attend_call* calls, int32_t n_calls) {
  UC_TRACE();
  if (calls == nullptr || n_calls < 1 || n_calls > UC_MAX_CALLS) return 0;
  int nbh_launch = 0;
  for (int c = 0; c < n_calls; ++c) {
    const uc_attend_call& k = calls[c];
    if (k.segs == nullptr || k.n_seg < 1 || k.n_seg > UC_MAX_SEGMENTS || k.segs[0] == nullptr ||
        k.n_qtok < 1 || k.n_qtok > UC_MAX_QTOKENS || k.segs[0]->n_kv_heads < 1 ||
        k.n_q_heads % k.segs[0]->n_kv_heads)
      return 0;
    nbh_launch += k.segs[0]->batch * k.segs[0]->n_kv_heads;
  }
  const int mt0 = decode_mtiles(calls[0].n_q_heads, calls[0].segs[0]->n_kv_heads, calls[0].n_qtok);
  int ipb[UC_MAX_CALLS];
  batch_items(calls, n_calls, mt0, ipb);
  size_t n = 256 + UC_MAX_CALLS * kCounterBlock;  // every call's counters at a fixed place, then the partials
  for (int c = 0; c < n_calls; ++c) {
    const uc_attend_call& k = calls[c];
    const int mt = decode_mtiles(k.n_q_heads, k.segs[0]->n_kv_heads, k.n_qtok);
    n += decode_part_bytes(k.segs, k.n_seg, mt, nbh_launch, ipb[c]);
  }
  return n;
}

uc_status uc_attend_batch(const uc_attend_call* calls, int32_t n_calls, void* workspace, size_t workspace_bytes,
                          void* stream) {
  UC_TRACE();
  if (calls == nullptr || workspace == nullptr || !aligned(workspace, 16)) {
    set_error("uc_attend_batch: null calls or null / misaligned workspace");
    return UC_ERR_ARG;
  }
  if (n_calls < 1 || n_calls > UC_MAX_CALLS) {
    set_error("uc_attend_batch: 1..%d calls per launch", UC_MAX_CALLS);
    return UC_ERR_SHAPE;
  }
  int mtiles = -1, nbh_launch = 0;
  for (int c = 0; c < n_calls; ++c) {
    const uc_attend_call& k = calls[c];
    const uc_status st = check_call(k.q, k.n_q_heads, k.n_qtok, k.segs, k.n_seg, k.out, "uc_attend_batch");
    if (st != UC_OK) return st;
    if (k.n_qtok > UC_MAX_QTOKENS) {
      set_error("uc_attend_batch: call %d has %d query tokens; batches take decode-shaped calls (<= %d)", c,
                k.n_qtok, UC_MAX_QTOKENS);
      return UC_ERR_SHAPE;
    }
    const int mt = decode_mtiles(k.n_q_heads, k.segs[0]->n_kv_heads, k.n_qtok);
    if (mt > 8 || (mtiles >= 0 && mt != mtiles)) {
      set_error("uc_attend_batch: call %d has %d query-row tiles of 8; every call of a batch needs the same "
                "number (<= 8)", c, mt);
      return UC_ERR_SHAPE;
    }
    mtiles = mt;
    nbh_launch += k.segs[0]->batch * k.segs[0]->n_kv_heads;
  }
  const size_t need = uc_attend_batch_workspace_size(calls, n_calls);
  if (need == 0 || workspace_bytes < need) {
    set_error("uc_attend_batch: workspace %zu < %zu bytes", workspace_bytes, need);
    return UC_ERR_OOM;
  }
  int ipb[UC_MAX_CALLS];
  batch_items(calls, n_calls, mtiles, ipb);
  static thread_local MultiAttnParams m;
  memset(&m, 0, sizeof(m));
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  DevStatus* status = reinterpret_cast<DevStatus*>(ws);
  size_t off = 256 + UC_MAX_CALLS * kCounterBlock;
  int heavy = 0, light = 0, grid = 0;
  for (int c = 0; c < n_calls; ++c) {
    const uc_attend_call& k = calls[c];
    AttnPlan plan;
    const uc_status st = build_decode_call(k.q, k.n_q_heads, k.n_qtok, k.segs, k.n_seg, k.out, k.lse, k.mass,
                                           nbh_launch, ipb[c], ws + 256 + c * kCounterBlock, ws + off, status,
                                           &m.call[c], &plan);
    if (st != UC_OK) return st;
    off += decode_part_bytes(k.segs, k.n_seg, mtiles, nbh_launch, ipb[c]);
    const int nbh = k.segs[0]->batch * k.segs[0]->n_kv_heads;
    m.heavy_begin[c] = heavy;
    m.light_begin[c] = light;
    heavy += plan.n_heavy * nbh;
    light += plan.n_light * nbh;
    grid = std::max(grid, plan.grid);
  }
  m.heavy_begin[n_calls] = heavy;
  m.light_begin[n_calls] = light;
  m.n_calls = n_calls;
  m.n_items = heavy + light;
  const int slots = std::max(1, attend_ctas_per_sm(mtiles)) * num_sms();
  launch_attend_multi(m, std::min(m.n_items, slots), reinterpret_cast<cudaStream_t>(stream));
  return cuda_check("uc_attend_batch");
}

// ------------------------------------------------------------------ append

static uc_status append_common(uc_segment* seg, const void* k_new, const void* v_new, int32_t position,
                               bool device_position, void* workspace, size_t workspace_bytes, void* stream,
                               const char* name) {
  uc_status st = check_segment(seg, name);
  if (st != UC_OK) return st;
  if (k_new == nullptr || v_new == nullptr || !aligned(k_new, 16) || !aligned(v_new, 16) ||
      workspace == nullptr || workspace_bytes < 256 || !aligned(workspace, 16)) {
    set_error("%s: null or misaligned argument / workspace < 256 bytes", name);
    return UC_ERR_ARG;
  }
  if (seg->kind == UC_KIND_FULL) {
    set_error("%s: FULL segments are read-only views", name);
    return UC_ERR_ARG;
  }
  if (!device_position)
    for (int b = 0; b < seg->batch; ++b)
      if (seg->n_kept_host[b] >= seg->cap) {
        set_error("%s: sequence %d is at capacity %d", name, b, seg->cap);
        return UC_ERR_BUDGET;
      }
  AppendArgs a;
  memset(&a, 0, sizeof(a));
  a.k_new = static_cast<const __nv_bfloat16*>(k_new);
  a.v_new = static_cast<const __nv_bfloat16*>(v_new);
  a.k = static_cast<__nv_bfloat16*>(seg->k);
  a.v = static_cast<__nv_bfloat16*>(seg->v);
  a.row_stride = seg->row_stride;
  a.row_offset = seg->row_offset;
  a.kept_idx = seg->kept_idx;
  a.n_kept = seg->n_kept;
  a.k_codes = static_cast<uint8_t*>(seg->k_codes);
  a.k_params = static_cast<uint8_t*>(seg->k_params);
  a.v_codes = static_cast<uint8_t*>(seg->v_codes);
  a.v_params = static_cast<uint8_t*>(seg->v_params);
  a.status = static_cast<DevStatus*>(workspace);
  a.batch = seg->batch;
  a.n_kv_heads = seg->n_kv_heads;
  a.cap = seg->cap;
  a.position = position;
  a.position_plus_count = device_position ? 1 : 0;
  launch_append(a, seg->bits, reinterpret_cast<cudaStream_t>(stream));
  st = cuda_check(name);
  if (st == UC_OK && !device_position)
    for (int b = 0; b < seg->batch; ++b) seg->n_kept_host[b] += 1;
  return st;
}

uc_status uc_append(uc_segment* seg, const void* k_new, const void* v_new, int32_t position,
                    void* workspace, size_t workspace_bytes, void* stream) {
  UC_TRACE();
  return append_common(seg, k_new, v_new, position, false, workspace, workspace_bytes, stream, "uc_append");
}

uc_status uc_append_next(uc_segment* seg, const void* k_new, const void* v_new, int32_t base_position,
                         void* workspace, size_t workspace_bytes, void* stream) {
  UC_TRACE();
  return append_common(seg, k_new, v_new, base_position, true, workspace, workspace_bytes, stream,
                       "uc_append_next");
}

}  // extern "C"
