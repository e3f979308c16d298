// Library-owned segments: the budget form of segment compression and its
// release (the problem statement of §3.4 / App. E, "per-segment compression
// under a budget": compress_segment(K, V, scores, budget) -> segment).
//
// uc_compress_budget maps one cache type's per-sequence budget tables (the
// output of Eq. 2, uc_allocate_budget) to the batch's segment configuration
// (uc_plan_batch), allocates the segment's storage and the call's workspace
// through the caller's allocator hook (by default cudaMallocAsync /
// cudaFreeAsync on the call's stream), compresses with uc_compress_segment
// and hands the segment out; uc_segment_free returns the storage. These are
// the only entry points that allocate device memory; every other call works
// on caller-owned storage.
#include <cuda_runtime.h>

#include <algorithm>
#include <cstring>
#include <mutex>
#include <unordered_map>

#include "internal.h"

namespace {

constexpr int kMaxOwnedArrays = 8;

struct Owned {
  uc_segment seg;                 // handed out as &seg
  uc_allocator alloc;             // the caller's hooks (alloc == NULL: stream-ordered CUDA allocator)
  void* stream;                   // stream the storage was allocated on and is released on
  void* ptrs[kMaxOwnedArrays];
  int n_ptrs;
};

std::mutex g_mu;

std::unordered_map<const uc_segment*, Owned*>& registry() {
  static std::unordered_map<const uc_segment*, Owned*> m;
  return m;
}

void* dev_alloc(const uc_allocator& a, size_t bytes, void* stream) {
  if (bytes == 0) return nullptr;
  if (a.alloc != nullptr) return a.alloc(bytes, stream, a.ctx);
  void* p = nullptr;
  if (cudaMallocAsync(&p, bytes, reinterpret_cast<cudaStream_t>(stream)) != cudaSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  return p;
}

void dev_free(const uc_allocator& a, void* p, void* stream) {
  if (p == nullptr) return;
  if (a.free != nullptr)
    a.free(p, stream, a.ctx);
  else
    cudaFreeAsync(p, reinterpret_cast<cudaStream_t>(stream));
}

void release(Owned* o) {
  for (int i = 0; i < o->n_ptrs; ++i) dev_free(o->alloc, o->ptrs[i], o->stream);
  delete o;
}

// Allocates `bytes` for one array of the segment (nullptr for 0 bytes);
// false when the allocator fails or returns storage that is not 16-byte
// aligned.
bool take(Owned* o, size_t bytes, void** slot) {
  *slot = nullptr;
  if (bytes == 0) return true;
  void* p = dev_alloc(o->alloc, bytes, o->stream);
  if (p == nullptr) return false;
  o->ptrs[o->n_ptrs++] = p;
  if (reinterpret_cast<uintptr_t>(p) % 16 != 0) return false;
  *slot = p;
  return true;
}

}  // namespace

extern "C" {

uc_status uc_compress_budget(const void* k_src, const void* v_src, int32_t batch, int32_t n_kv_heads,
                             int32_t n_src, int64_t src_row_stride, int64_t src_row_offset, const float* scores,
                             int64_t scores_stride, int64_t scores_offset, int32_t n_recent,
                             const uc_segment_table* tables, int32_t type, const uc_allocator* allocator,
                             void* stream, uc_segment** out) {
  UC_TRACE();
  if (out == nullptr) {
    uc::set_error("uc_compress_budget: null output");
    return UC_ERR_ARG;
  }
  *out = nullptr;
  if (k_src == nullptr || v_src == nullptr || tables == nullptr) {
    uc::set_error("uc_compress_budget: null source or tables");
    return UC_ERR_ARG;
  }
  if (allocator != nullptr && ((allocator->alloc == nullptr) != (allocator->free == nullptr))) {
    uc::set_error("uc_compress_budget: an allocator needs both alloc and free (or neither)");
    return UC_ERR_ARG;
  }
  if (batch < 1 || batch > UC_MAX_BATCH || n_kv_heads < 1 || n_kv_heads > 8 || n_src < 0) {
    uc::set_error("uc_compress_budget: unsupported shape (batch %d, kv heads %d, n_src %d)", batch, n_kv_heads,
                  n_src);
    return UC_ERR_SHAPE;
  }
  if (tables[0].n_types < 1 || tables[0].n_types > UC_MAX_SEGMENTS || type < 0 || type >= tables[0].n_types) {
    uc::set_error("uc_compress_budget: type %d outside the tables' %d types", type, tables[0].n_types);
    return UC_ERR_ARG;
  }
  if (tables[0].n_tokens[type] != n_src) {
    uc::set_error("uc_compress_budget: the tables give %d tokens for type %d, the source %d",
                  tables[0].n_tokens[type], type, n_src);
    return UC_ERR_SHAPE;
  }
  if (src_row_offset < 0 || src_row_stride < (int64_t)n_src + src_row_offset) {
    uc::set_error("uc_compress_budget: bad source rows");
    return UC_ERR_SHAPE;
  }
  int32_t keep[UC_MAX_BATCH];
  uc_type_config cfg;
  uc_status st = uc_plan_batch(tables, batch, type, keep, &cfg);
  if (st != UC_OK) return st;

  Owned* o = new Owned();
  memset(&o->seg, 0, sizeof(o->seg));
  o->alloc = allocator != nullptr ? *allocator : uc_allocator{nullptr, nullptr, nullptr};
  o->stream = stream;
  o->n_ptrs = 0;
  uc_segment& s = o->seg;
  s.batch = batch;
  s.n_kv_heads = n_kv_heads;
  s.head_dim = UC_HEAD_DIM;
  s.n_src = n_src;
  s.label = type;
  cudaStream_t cs = reinterpret_cast<cudaStream_t>(stream);
  const int64_t nbh = (int64_t)batch * n_kv_heads;

  if (cfg.full_view) {
    // every sequence keeps every token in bf16: a view of the source rows
    s.kind = UC_KIND_FULL;
    s.bits = 16;
    s.cap = n_src;
    s.k = const_cast<void*>(k_src);
    s.v = const_cast<void*>(v_src);
    s.row_stride = src_row_stride;
    s.row_offset = src_row_offset;
    s.rows_total = nbh * src_row_stride;
    for (int b = 0; b < batch; ++b) s.n_kept_host[b] = n_src;
    void* nk = nullptr;
    if (!take(o, 4ull * batch, &nk)) {
      release(o);
      uc::set_error("uc_compress_budget: allocation failed");
      return UC_ERR_OOM;
    }
    s.n_kept = static_cast<int32_t*>(nk);
    // pageable source: staged before the call returns
    if (cudaMemcpyAsync(s.n_kept, s.n_kept_host, 4ull * batch, cudaMemcpyHostToDevice, cs) != cudaSuccess) {
      release(o);
      uc::set_error("uc_compress_budget: %s", cudaGetErrorString(cudaGetLastError()));
      return UC_ERR_CUDA;
    }
  } else {
    s.kind = cfg.kind;
    s.bits = cfg.bits;
    s.cap = std::max(64, (cfg.max_keep + 63) / 64 * 64);
    uc_segment_sizes sz;
    st = uc_segment_sizes_of(&s, &sz);
    if (st != UC_OK) {
      release(o);
      return st;
    }
    void* p[8];
    const uint64_t bytes[8] = {sz.n_kept, sz.kept_idx, sz.k, sz.v, sz.k_codes, sz.k_params, sz.v_codes, sz.v_params};
    for (int i = 0; i < 8; ++i)
      if (!take(o, bytes[i], &p[i])) {
        release(o);
        uc::set_error("uc_compress_budget: allocation of %llu bytes failed or is not 16-byte aligned",
                      (unsigned long long)bytes[i]);
        return UC_ERR_OOM;
      }
    s.n_kept = static_cast<int32_t*>(p[0]);
    s.kept_idx = static_cast<int32_t*>(p[1]);
    s.k = p[2];
    s.v = p[3];
    s.k_codes = p[4];
    s.k_params = p[5];
    s.v_codes = p[6];
    s.v_params = p[7];
    const bool packed = s.kind == UC_KIND_QUANT || s.kind == UC_KIND_EVICT_QUANT;
    s.row_stride = packed ? UC_GROUP : s.cap;
    s.row_offset = 0;
    s.rows_total = nbh * s.row_stride;
    for (int b = 0; b < batch; ++b) s.n_kept_host[b] = keep[b];
    if (cfg.max_keep == 0) {
      // nothing kept anywhere: an empty segment
      if (cudaMemsetAsync(s.n_kept, 0, 4ull * batch, cs) != cudaSuccess) {
        release(o);
        uc::set_error("uc_compress_budget: %s", cudaGetErrorString(cudaGetLastError()));
        return UC_ERR_CUDA;
      }
    } else {
      const size_t wbytes = uc_compress_workspace_size(&s);
      void* ws = dev_alloc(o->alloc, wbytes, stream);
      if (ws == nullptr || reinterpret_cast<uintptr_t>(ws) % 16 != 0) {
        dev_free(o->alloc, ws, stream);
        release(o);
        uc::set_error("uc_compress_budget: workspace allocation failed or is not 16-byte aligned");
        return UC_ERR_OOM;
      }
      // the status word the kernels report through starts clean
      if (cudaMemsetAsync(ws, 0, 16, cs) != cudaSuccess) {
        dev_free(o->alloc, ws, stream);
        release(o);
        uc::set_error("uc_compress_budget: %s", cudaGetErrorString(cudaGetLastError()));
        return UC_ERR_CUDA;
      }
      st = uc_compress_segment(k_src, v_src, src_row_stride, src_row_offset, scores, scores_stride, scores_offset,
                               n_recent, &s, ws, wbytes, stream);
      if (st == UC_OK) st = uc_workspace_status(ws, stream);  // synchronises the stream
      dev_free(o->alloc, ws, stream);
      if (st != UC_OK) {
        release(o);
        return st;
      }
    }
  }
  {
    std::lock_guard<std::mutex> lock(g_mu);
    registry()[&o->seg] = o;
  }
  *out = &o->seg;
  return UC_OK;
}

void uc_segment_free(uc_segment* seg) {
  UC_TRACE();
  if (seg == nullptr) return;
  Owned* o = nullptr;
  {
    std::lock_guard<std::mutex> lock(g_mu);
    auto it = registry().find(seg);
    if (it == registry().end()) {
      uc::set_error("uc_segment_free: not a segment uc_compress_budget returned (left untouched)");
      return;
    }
    o = it->second;
    registry().erase(it);
  }
  release(o);
}

}  // extern "C"
