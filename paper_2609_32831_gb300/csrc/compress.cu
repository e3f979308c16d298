// Segment compression kernels (§3.4; App. E "Physical, type-aware KV
// storage" and "Batched GQA token selection") and the decode-time append.
//
//  topk_select     exact per-(sequence, KV head) top-k by radix select on
//                  order-preserving score keys, ties to the lower index,
//                  kept indices written in ascending order
//  gather_rows     compaction of the kept bf16 rows (eviction)
//  quantize_groups int4 / int2 group quantization of the kept sequence
//  copy_tail       the bf16 residual tail (n_kept mod 32 last kept tokens)
//  append_token    one decode token per sequence into a segment
#include <algorithm>

#include <cooperative_groups.h>

#include "internal.h"
#include "quant.cuh"

namespace cg = cooperative_groups;

namespace uc {

// ------------------------------------------------------------------ top-k

// Order-preserving key of an fp32 score (ascending key <=> ascending value),
// with -0.0 folded onto +0.0.
__device__ __forceinline__ uint32_t score_key(float f) {
  uint32_t u = __float_as_uint(f);
  if (f == 0.0f) u = 0u;
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

constexpr int kTopkThreads = 1024;

// Block-wide exclusive scan of one flag per thread; returns the prefix and
// writes the block total to *total. Uses `scratch` [32] ints.
__device__ __forceinline__ int block_excl_scan(int flag, int* scratch, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const unsigned bal = __ballot_sync(0xffffffffu, flag);
  const int in_warp = __popc(bal & ((1u << lane) - 1u));
  if (lane == 0) scratch[warp] = __popc(bal);
  __syncthreads();
  int before = 0, sum = 0;
  for (int w = 0; w < kTopkThreads / 32; ++w) {
    const int c = scratch[w];
    before += (w < warp) ? c : 0;
    sum += c;
  }
  __syncthreads();
  *total = sum;
  return before + in_warp;
}

// Score of candidate i: scores[i], or scores[idx[i]] through the source's
// logical indices; an index outside the score array flags UC_ERR_RANGE and
// reads nothing.
__device__ __forceinline__ float candidate_score(const float* s, const int32_t* idx, int64_t limit, int i,
                                                 int* bad) {
  if (idx == nullptr) return s[i];
  const int32_t t = idx[i];
  if (t < 0 || t >= limit) {
    *bad = 1;
    return 0.f;
  }
  return s[t];
}

__global__ void __launch_bounds__(kTopkThreads) topk_select_kernel(TopkArgs a) {
  const int bh = blockIdx.x;
  const int b = bh / a.n_kv_heads;
  const int keep = a.keep[b];
  const float* s = a.scores + (int64_t)bh * a.scores_stride + a.scores_offset;
  int32_t* out = a.kept_idx + (int64_t)bh * a.cap;
  const int32_t* sidx = a.score_idx ? a.score_idx + (int64_t)bh * a.score_idx_stride : nullptr;
  const int r = min(a.n_recent, keep);
  const int n_old = a.src_n[b] - r;
  const int k_old = keep - r;

  __shared__ uint32_t hist[256];
  __shared__ uint32_t sh_prefix, sh_mask, sh_remaining;
  __shared__ int scratch[32];
  __shared__ int sh_nan;

  if (threadIdx.x == 0) {
    sh_prefix = 0;
    sh_mask = 0;
    sh_remaining = (uint32_t)k_old;
    sh_nan = 0;
  }
  __syncthreads();

  if (k_old > 0) {
    for (int shift = 24; shift >= 0; shift -= 8) {
      for (int i = threadIdx.x; i < 256; i += kTopkThreads) hist[i] = 0;
      __syncthreads();
      const uint32_t prefix = sh_prefix, mask = sh_mask;
      for (int i = threadIdx.x; i < n_old; i += kTopkThreads) {
        int bad = 0;
        const float f = candidate_score(s, sidx, a.score_limit, i, &bad);
        if (shift == 24 && (isnan(f) || bad)) sh_nan = bad ? 2 : 1;
        const uint32_t key = score_key(f);
        if ((key & mask) == prefix) atomicAdd(&hist[(key >> shift) & 255u], 1u);
      }
      __syncthreads();
      if (threadIdx.x == 0) {
        uint32_t rem = sh_remaining, cum = 0;
        int digit = 0;
        for (int d = 255; d >= 0; --d) {
          const uint32_t h = hist[d];
          if (cum + h >= rem) {
            digit = d;
            break;
          }
          cum += h;
        }
        sh_remaining = rem - cum;
        sh_prefix = prefix | ((uint32_t)digit << shift);
        sh_mask = mask | (255u << shift);
      }
      __syncthreads();
    }
  }
  if (sh_nan) {
    // the result is undefined, but later kernels of the call must still find
    // in-range row indices: keep rows 0 .. keep-1
    for (int t = threadIdx.x; t < keep; t += kTopkThreads) out[t] = t;
    if (bh % a.n_kv_heads == 0 && threadIdx.x == 0) a.n_kept[b] = keep;
    if (threadIdx.x == 0) set_status(a.status, UC_ERR_RANGE, sh_nan);
    return;
  }
  const uint32_t thr = sh_prefix;
  const int need_eq = (int)sh_remaining;
  int out_base = 0, eq_base = 0;
  if (k_old > 0) {
    for (int base = 0; base < n_old; base += kTopkThreads) {
      const int i = base + threadIdx.x;
      uint32_t key = 0;
      int bad = 0;
      if (i < n_old) key = score_key(candidate_score(s, sidx, a.score_limit, i, &bad));
      const int gt = (i < n_old) && key > thr;
      const int eq = (i < n_old) && key == thr;
      int eq_total, take_total;
      const int eq_rank = eq_base + block_excl_scan(eq, scratch, &eq_total);
      const int take = gt || (eq && eq_rank < need_eq);
      const int pos = out_base + block_excl_scan(take, scratch, &take_total);
      if (take) out[pos] = i;
      eq_base += eq_total;
      out_base += take_total;
    }
  }
  for (int t = threadIdx.x; t < r; t += kTopkThreads) out[k_old + t] = n_old + t;
  if (bh % a.n_kv_heads == 0 && threadIdx.x == 0) a.n_kept[b] = keep;
}

// The same selection for long candidate lists (the long-context workloads:
// ~118K image tokens per (sequence, KV head) at 128K context): one cluster of
// kTopkCluster CTAs per (sequence, KV head), each CTA histogramming its share
// of the candidates into rank 0's shared-memory histogram (distributed shared
// memory) between cluster barriers, then counting its (greater, equal) keys
// so that each CTA writes its kept indices at their global rank. Every CTA
// runs every cluster barrier, and none leaves while another may still read
// its shared memory.
constexpr int kTopkCluster = 8;
// The cluster kernel serves calls with long candidate lists and few (sequence,
// KV head) pairs (128K context, batch 2: 8 pairs x 118K candidates, 405 ->
// 109 us); with many pairs one CTA each already fills the GPU (32K context,
// batch 16: 64 pairs x 29K candidates, 150 us single vs 236 us clustered).
constexpr int kTopkClusterMinN = 16384;
constexpr int kTopkClusterMaxPairs = 32;

__device__ __forceinline__ int block_sum(int v, int* scratch) {
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  if ((threadIdx.x & 31) == 0) scratch[threadIdx.x >> 5] = v;
  __syncthreads();
  int s = 0;
  for (int w = 0; w < kTopkThreads / 32; ++w) s += scratch[w];
  __syncthreads();
  return s;
}

__global__ void __cluster_dims__(kTopkCluster, 1, 1) __launch_bounds__(kTopkThreads)
    topk_cluster_kernel(TopkArgs a) {
  cg::cluster_group cluster = cg::this_cluster();
  const int rank = (int)cluster.block_rank();
  const int bh = blockIdx.x / kTopkCluster;
  const int b = bh / a.n_kv_heads;
  const int keep = a.keep[b];
  const float* s = a.scores + (int64_t)bh * a.scores_stride + a.scores_offset;
  int32_t* out = a.kept_idx + (int64_t)bh * a.cap;
  const int32_t* sidx = a.score_idx ? a.score_idx + (int64_t)bh * a.score_idx_stride : nullptr;
  const int r = min(a.n_recent, keep);
  const int n_old = a.src_n[b] - r;
  const int k_old = keep - r;
  const int lo = (int)((int64_t)n_old * rank / kTopkCluster);
  const int hi = (int)((int64_t)n_old * (rank + 1) / kTopkCluster);
  const int tid = threadIdx.x;

  __shared__ uint32_t hist[256];   // this CTA's histogram of the pass
  __shared__ uint32_t ghist[256];  // the cluster's histogram (rank 0's copy)
  __shared__ uint32_t sh_prefix, sh_mask, sh_remaining;
  __shared__ int sh_nan;
  __shared__ int counts[kTopkCluster][2];  // rank 0: (greater, equal) keys per CTA
  __shared__ int scratch[32];
  uint32_t* g_hist = cluster.map_shared_rank(ghist, 0);
  int* g_nan = cluster.map_shared_rank(&sh_nan, 0);

  for (int i = tid; i < 256; i += kTopkThreads) ghist[i] = 0;
  if (tid == 0) {
    sh_prefix = 0;
    sh_mask = 0;
    sh_remaining = (uint32_t)max(k_old, 0);
    sh_nan = 0;
  }
  cluster.sync();  // every CTA's shared memory is set before any other adds into it

  uint32_t prefix = 0, mask = 0;
  if (k_old > 0) {  // the same for every CTA of the cluster (one sequence)
    for (int shift = 24; shift >= 0; shift -= 8) {
      for (int i = tid; i < 256; i += kTopkThreads) hist[i] = 0;
      __syncthreads();
      for (int i = lo + tid; i < hi; i += kTopkThreads) {
        int bad = 0;
        const float f = candidate_score(s, sidx, a.score_limit, i, &bad);
        if (shift == 24 && (isnan(f) || bad)) atomicOr(g_nan, bad ? 2 : 1);
        const uint32_t key = score_key(f);
        if ((key & mask) == prefix) atomicAdd(&hist[(key >> shift) & 255u], 1u);
      }
      __syncthreads();
      for (int i = tid; i < 256; i += kTopkThreads)
        if (hist[i]) atomicAdd(&g_hist[i], hist[i]);
      cluster.sync();
      if (rank == 0) {
        if (tid == 0) {
          uint32_t rem = sh_remaining, cum = 0;
          int digit = 0;
          for (int d = 255; d >= 0; --d) {
            const uint32_t h = ghist[d];
            if (cum + h >= rem) {
              digit = d;
              break;
            }
            cum += h;
          }
          sh_remaining = rem - cum;
          sh_prefix |= (uint32_t)digit << shift;
          sh_mask |= 255u << shift;
        }
        __syncthreads();
        for (int i = tid; i < 256; i += kTopkThreads) ghist[i] = 0;
      }
      cluster.sync();
      prefix = *cluster.map_shared_rank(&sh_prefix, 0);
      mask = *cluster.map_shared_rank(&sh_mask, 0);
    }
  }
  const int nan = *g_nan;
  const uint32_t thr = prefix;
  const int need_eq = (int)*cluster.map_shared_rank(&sh_remaining, 0);
  if (nan) {
    // the result is undefined, but later kernels of the call must still find
    // in-range row indices: keep rows 0 .. keep-1
    if (rank == 0) {
      for (int t = tid; t < keep; t += kTopkThreads) out[t] = t;
      if (bh % a.n_kv_heads == 0 && tid == 0) a.n_kept[b] = keep;
      if (tid == 0) set_status(a.status, UC_ERR_RANGE, nan);
    }
  } else if (k_old > 0) {
    // this CTA's (greater, equal) counts, then the global rank of its first take
    int gt = 0, eq = 0;
    for (int i = lo + tid; i < hi; i += kTopkThreads) {
      int bad = 0;
      const uint32_t key = score_key(candidate_score(s, sidx, a.score_limit, i, &bad));
      gt += key > thr;
      eq += key == thr;
    }
    gt = block_sum(gt, scratch);
    eq = block_sum(eq, scratch);
    if (tid == 0) {
      int* c = cluster.map_shared_rank(&counts[0][0], 0);
      c[2 * rank] = gt;
      c[2 * rank + 1] = eq;
    }
    cluster.sync();
    int eq_base = 0, out_base = 0;
    for (int q = 0; q < rank; ++q) {
      const int* c = cluster.map_shared_rank(&counts[q][0], 0);
      const int g_q = c[0], e_q = c[1];
      out_base += g_q + min(e_q, max(0, need_eq - eq_base));
      eq_base += e_q;
    }
    for (int base = lo; base < hi; base += kTopkThreads) {
      const int i = base + tid;
      uint32_t key = 0;
      int bad = 0;
      if (i < hi) key = score_key(candidate_score(s, sidx, a.score_limit, i, &bad));
      const int g1 = (i < hi) && key > thr;
      const int e1 = (i < hi) && key == thr;
      int eq_total, take_total;
      const int eq_rank = eq_base + block_excl_scan(e1, scratch, &eq_total);
      const int take = g1 || (e1 && eq_rank < need_eq);
      const int pos = out_base + block_excl_scan(take, scratch, &take_total);
      if (take) out[pos] = i;
      eq_base += eq_total;
      out_base += take_total;
    }
  }
  if (!nan && rank == 0) {
    for (int t = tid; t < r; t += kTopkThreads) out[k_old + t] = n_old + t;
    if (bh % a.n_kv_heads == 0 && tid == 0) a.n_kept[b] = keep;
  }
  if (nan || k_old <= 0) cluster.sync();  // the count exchange's barrier of the other path
  cluster.sync();  // no CTA leaves while another may still read its shared memory
}

// Kept indices of a segment that keeps every token (QUANT).
__global__ void iota_kernel(TopkArgs a) {
  const int bh = blockIdx.x;
  const int b = bh / a.n_kv_heads;
  int32_t* out = a.kept_idx + (int64_t)bh * a.cap;
  for (int t = threadIdx.x; t < a.keep[b]; t += blockDim.x) out[t] = t;
  if (bh % a.n_kv_heads == 0 && threadIdx.x == 0) a.n_kept[b] = a.keep[b];
}

// -------------------------------------------------- re-compression helpers

// One warp per (b, kvh, 32 kept tokens) of a packed segment: rebuild the K and
// V rows in bf16 (x = code * s + z, exact in fp32, rounded to nearest even);
// the residual tail rows are copied. Lane L handles channels 4L .. 4L + 3.
template <int BITS>
__global__ void dequant_rows_kernel(DequantArgs a) {
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  const int nbh = a.batch * a.n_kv_heads;
  if (warp >= nbh * a.max_groups) return;
  const int bh = warp / a.max_groups, g = warp % a.max_groups;
  const int b = bh / a.n_kv_heads;
  const int n = a.n_kept[b];
  const int ng = n / kGroup;
  if (g * kGroup >= n) return;
  __nv_bfloat16* ko = a.k_out + ((size_t)bh * a.cap + (size_t)g * kGroup) * kHeadDim;
  __nv_bfloat16* vo = a.v_out + ((size_t)bh * a.cap + (size_t)g * kGroup) * kHeadDim;
  if (g >= ng) {  // the tail block (n mod 32 rows)
    const __nv_bfloat16* kt = a.k_tail + (size_t)bh * kGroup * kHeadDim;
    const __nv_bfloat16* vt = a.v_tail + (size_t)bh * kGroup * kHeadDim;
    for (int t = 0; t < n - g * kGroup; ++t) {
      reinterpret_cast<uint2*>(ko + t * kHeadDim)[lane] = reinterpret_cast<const uint2*>(kt + t * kHeadDim)[lane];
      reinterpret_cast<uint2*>(vo + t * kHeadDim)[lane] = reinterpret_cast<const uint2*>(vt + t * kHeadDim)[lane];
    }
    return;
  }
  constexpr uint32_t mask = (1u << BITS) - 1u;
  const size_t blk = (size_t)bh * a.cap * kHeadDim * BITS / 8;
  const uint8_t* kc = a.k_codes + blk;
  const uint8_t* vc = a.v_codes + blk;
  const uint8_t* kp = a.k_params + (size_t)bh * (a.cap / kGroup) * 512 + (size_t)g * 512;
  const uint8_t* vp = a.v_params + (size_t)bh * a.cap * 16;
  for (int tg = 0; tg < kGroup; ++tg) {
    const int t = g * kGroup + tg;
    float kx[4], vx[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int c = 4 * lane + e;
      // key code (token tg of group g, channel c) in the fragment layout
      const int nt = tg >> 3, nn = tg & 7, i = c >> 4, cc = c & 15;
      const int j = (cc & 7) >> 1, sub = cc >> 3, ee = cc & 1;
      const int pr = BITS == 4 ? 2 * (i & 1) + sub : 2 * (i & 3) + sub;
      const int wq = BITS == 4 ? (i >> 1) : (i >> 2);
      const uint32_t w =
          *reinterpret_cast<const uint32_t*>(kc + ((size_t)(g * 4 + nt) * 32 + nn * 4 + j) * (BITS * 4) + 4 * wq);
      const uint32_t code = (w >> (BITS * pr + 16 * ee)) & mask;
      const __half* kpar = reinterpret_cast<const __half*>(kp + (i * 4 + j) * 16);
      kx[e] = __fmaf_rn((float)code, __half2float(kpar[sub * 2 + ee]), __half2float(kpar[4 + sub * 2 + ee]));
      // value code (token t, channel c): 16-token tile, lane (c % 8, token pair)
      const int t16 = t >> 4, tt = t & 15, m = c >> 3, gq = c & 7;
      const int vsub = tt >> 3, vj = (tt & 7) >> 1, ve = tt & 1;
      const int vpr = BITS == 4 ? 2 * (m & 1) + vsub : 2 * (m & 3) + vsub;
      const int vwq = BITS == 4 ? (m >> 1) : (m >> 2);
      const uint32_t vw =
          *reinterpret_cast<const uint32_t*>(vc + ((size_t)t16 * 32 + gq * 4 + vj) * (BITS * 8) + 4 * vwq);
      const uint32_t vcode = (vw >> (BITS * vpr + 16 * ve)) & mask;
      const __half* vpar = reinterpret_cast<const __half*>(vp + (size_t)t16 * 256 + ((c >> 5) * 4 + vj) * 16);
      vx[e] = __fmaf_rn((float)vcode, __half2float(vpar[vsub * 2 + ve]), __half2float(vpar[4 + vsub * 2 + ve]));
    }
    const uint2 kw = make_uint2(pack_bf16(kx[0], kx[1]), pack_bf16(kx[2], kx[3]));
    const uint2 vw2 = make_uint2(pack_bf16(vx[0], vx[1]), pack_bf16(vx[2], vx[3]));
    reinterpret_cast<uint2*>(ko + tg * kHeadDim)[lane] = kw;
    reinterpret_cast<uint2*>(vo + tg * kHeadDim)[lane] = vw2;
  }
}

__global__ void compose_idx_kernel(ComposeArgs a) {
  const int bh = blockIdx.x;
  const int b = bh / a.n_kv_heads;
  int32_t* idx = a.kept_idx + (int64_t)bh * a.cap;
  const int32_t* src = a.src_idx + (int64_t)bh * a.src_cap;
  for (int t = threadIdx.x; t < a.n_kept[b]; t += blockDim.x) idx[t] = src[idx[t]];
}

// ----------------------------------------------------------------- gather

// One warp per (b, kvh, 32 kept tokens): copy the kept K and V rows into the
// compacted bf16 storage (rows_per_block = cap, offset 0).
__global__ void gather_rows_kernel(GatherArgs a) {
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  const int per_bh = a.max_chunks;
  const int bh = warp / per_bh;
  if (bh >= a.batch * a.n_kv_heads) return;
  const int b = bh / a.n_kv_heads;
  const int t0 = (warp % per_bh) * 32;
  const int n = a.keep[b];
  if (t0 >= n) return;
  const int32_t* idx = a.kept_idx + (int64_t)bh * a.cap;
  const int64_t src_base = (int64_t)bh * a.src_row_stride + a.src_row_offset;
  const int64_t dst_base = (int64_t)bh * a.dst_row_stride + a.dst_row_offset;
  const int cnt = min(32, n - t0);
  // two rows per pass: lanes 0..15 row 2q, lanes 16..31 row 2q+1
  for (int q = 0; q < (cnt + 1) / 2; ++q) {
    const int t = t0 + 2 * q + (lane >> 4);
    if (t < t0 + cnt) {
      const int64_t sr = src_base + idx[t];
      const int64_t dr = dst_base + t;
      const int c = (lane & 15) * 8;
      *reinterpret_cast<uint4*>(a.k_dst + dr * kHeadDim + c) =
          *reinterpret_cast<const uint4*>(a.k_src + sr * kHeadDim + c);
      *reinterpret_cast<uint4*>(a.v_dst + dr * kHeadDim + c) =
          *reinterpret_cast<const uint4*>(a.v_src + sr * kHeadDim + c);
    }
  }
}

// ---------------------------------------------------------- quantization

// Persistent: each warp quantizes the groups gw, gw + W, ... (W warps in the
// grid), consecutive warps taking consecutive groups of a (b, kvh). A warp
// stages a group's 32 K rows and 32 V rows in shared memory with one bulk
// copy per row (rows gathered through the kept-index list, 272 bytes apart
// so that rows of the fragment-order reads fall in different banks).
// kQuantBufs = 1 (used): one buffer takes the K rows, then the V rows; each
// warp waits for every copy, but 10 KB of shared memory per warp fits 21
// warps per SM, which cover each other's waits (32K layer, batch 16: int2
// 376 us, int4 383 us). kQuantBufs = 2: K and V rows have buffers of their
// own and each copy is requested half a group ahead, but only 12 warps fit
// (403 / 414 us).
constexpr int kQuantBufs = 1;
constexpr int kQuantWarps = kQuantBufs == 2 ? 6 : 7;
constexpr int kQuantCtasPerSm = kQuantBufs == 2 ? 2 : 3;
constexpr int kQuantRowBytes = 272;

struct QuantWarpSmem {
  uint8_t rows[kQuantBufs][32 * kQuantRowBytes];
  QuantStats st;
  uint64_t bar[kQuantBufs];
};
constexpr size_t kQuantSmemBytes = kQuantWarps * sizeof(QuantWarpSmem);

template <int BITS>
__global__ void __launch_bounds__(kQuantWarps * 32, kQuantCtasPerSm) quantize_groups_kernel(GatherArgs a) {
  extern __shared__ __align__(16) uint8_t quant_smem[];
  QuantWarpSmem& sm = reinterpret_cast<QuantWarpSmem*>(quant_smem)[threadIdx.x >> 5];
  const int lane = threadIdx.x & 31;
  const int n_warps = gridDim.x * kQuantWarps;
  const int per_bh = a.max_chunks;
  const int total = a.batch * a.n_kv_heads * per_bh;
  // the first valid group at or after w (groups past a sequence's full
  // groups are skipped)
  auto valid_from = [&](int w) {
    for (; w < total; w += n_warps) {
      const int b = (w / per_bh) / a.n_kv_heads;
      if (w % per_bh < a.keep[b] / kGroup) break;
    }
    return w;
  };
  if (lane == 0) {
    for (int k = 0; k < kQuantBufs; ++k) mbar_init(&sm.bar[k], 1);
    fence_barrier_init();
  }
  __syncwarp();
  // kept index of this lane's row of group w (loaded a group ahead, so that
  // the request does not wait for it)
  auto row_index = [&](int w) {
    return w < total ? a.kept_idx[(int64_t)(w / per_bh) * a.cap + (w % per_bh) * kGroup + lane] : 0;
  };
  // rows of group w (K if kv == 0, else V) into buffer `buf`
  auto request = [&](int w, int buf, int kv, int32_t idx) {
    const int64_t row = (int64_t)(w / per_bh) * a.src_row_stride + a.src_row_offset + idx;
    if (lane == 0) mbar_arrive_expect_tx(&sm.bar[buf], kGroup * kHeadDim * 2);
    __syncwarp();
    if (w == a.withhold && kv == 0 && lane == 0) return;  // test hook: one K row is never copied
    bulk_load(sm.rows[buf] + lane * kQuantRowBytes, (kv ? a.v_src : a.k_src) + row * kHeadDim, kHeadDim * 2,
              &sm.bar[buf]);
  };
  constexpr int kVBuf = kQuantBufs - 1;
  auto krow = [&](int t) { return reinterpret_cast<const __nv_bfloat16*>(sm.rows[0] + t * kQuantRowBytes); };
  auto vrow = [&](int t) { return reinterpret_cast<const __nv_bfloat16*>(sm.rows[kVBuf] + t * kQuantRowBytes); };
  int w = valid_from(blockIdx.x * kQuantWarps + (threadIdx.x >> 5));
  if (w >= total) return;
  int32_t idx = row_index(w);
  request(w, 0, 0, idx);
  if constexpr (kQuantBufs == 2) request(w, 1, 1, idx);
  // phase of the next completion of each buffer's barrier
  uint32_t ph_k = 0, ph_v = 0;
  bool failed = false;
  while (w < total) {
    const int next = valid_from(w + n_warps);
    const int32_t next_idx = row_index(next);
    const int bh = w / per_bh, g = w % per_bh;
    QuantOut out;
    out.k_codes = a.k_codes + (size_t)bh * a.cap * kHeadDim * BITS / 8;
    out.k_params = a.k_params + (size_t)bh * (a.cap / kGroup) * 512;
    out.v_codes = a.v_codes + (size_t)bh * a.cap * kHeadDim * BITS / 8;
    out.v_params = a.v_params + (size_t)bh * a.cap * 16;
    if (!__all_sync(0xffffffffu, mbar_wait(&sm.bar[0], ph_k, a.status, 20, a.wait_ns))) {
      failed = true;
      break;
    }
    ph_k ^= 1u;
    const bool ok = quantize_keys<BITS>(krow, g, out, sm.st);
    // every lane has read this group's K rows: the buffer takes the next rows
    if constexpr (kQuantBufs == 2) {
      if (next < total) request(next, 0, 0, next_idx);
    } else {
      request(w, 0, 1, idx);
      ph_v = ph_k;
    }
    if (!__all_sync(0xffffffffu, mbar_wait(&sm.bar[kVBuf], ph_v, a.status, 21, a.wait_ns))) {
      failed = true;
      break;
    }
    ph_v ^= 1u;
    if (!ok || !quantize_values<BITS>(vrow, g, out, sm.st)) {
      if (lane == 0) set_status(a.status, UC_ERR_RANGE, 2);
    }
    if constexpr (kQuantBufs == 2) {
      if (next < total) request(next, 1, 1, next_idx);
    } else {
      if (next < total) request(next, 0, 0, next_idx);
      ph_k = ph_v;
    }
    idx = next_idx;
    w = next;
  }
  if (failed) {
    // copies still in flight must land before the warp's shared memory is
    // released: wait for each barrier's pending phase (bounded again)
    mbar_wait(&sm.bar[0], ph_k, nullptr, 0, a.wait_ns);
    if constexpr (kQuantBufs == 2) mbar_wait(&sm.bar[1], ph_v, nullptr, 0, a.wait_ns);
  }
}

// The residual tail: the last (n mod 32) kept tokens, copied to the bf16
// tail block (32 rows per (b, kvh)). One warp per (b, kvh).
__global__ void copy_tail_kernel(GatherArgs a) {
  const int bh = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (bh >= a.batch * a.n_kv_heads) return;
  const int b = bh / a.n_kv_heads;
  const int n = a.keep[b];
  const int t0 = (n / kGroup) * kGroup;
  const int32_t* idx = a.kept_idx + (int64_t)bh * a.cap;
  const int64_t src_base = (int64_t)bh * a.src_row_stride + a.src_row_offset;
  for (int t = t0 + (lane >> 4); t < n; t += 2) {
    const int64_t sr = src_base + idx[t];
    const int64_t dr = (int64_t)bh * kGroup + (t - t0);
    const int c = (lane & 15) * 8;
    *reinterpret_cast<uint4*>(a.k_dst + dr * kHeadDim + c) =
        *reinterpret_cast<const uint4*>(a.k_src + sr * kHeadDim + c);
    *reinterpret_cast<uint4*>(a.v_dst + dr * kHeadDim + c) =
        *reinterpret_cast<const uint4*>(a.v_src + sr * kHeadDim + c);
  }
}

// ---------------------------------------------------------------- append

// One CTA per sequence, one warp per KV head.
template <int BITS>
__global__ void append_token_kernel(AppendArgs a) {
  // Launched programmatically, an append waits for nothing: it writes only
  // its own segment, which the launches it may overlap do not read (the
  // caller orders them so: uc_set_programmatic_launch).
  griddep_launch_dependents();
  const int b = blockIdx.x;
  const int j = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  __shared__ int sh_n;
  if (threadIdx.x == 0) sh_n = a.n_kept[b];
  __syncthreads();
  const int n = sh_n;
  if (n >= a.cap) {
    if (threadIdx.x == 0) set_status(a.status, UC_ERR_BUDGET, 3);
    return;
  }
  if (j < a.n_kv_heads) {
    const int bh = b * a.n_kv_heads + j;
    const __nv_bfloat16* kn = a.k_new + (int64_t)bh * kHeadDim;
    const __nv_bfloat16* vn = a.v_new + (int64_t)bh * kHeadDim;
    int64_t row;
    if (BITS == 16)
      row = (int64_t)bh * a.row_stride + a.row_offset + n;
    else
      row = (int64_t)bh * kGroup + (n % kGroup);
    reinterpret_cast<uint2*>(a.k + row * kHeadDim)[lane] = reinterpret_cast<const uint2*>(kn)[lane];
    reinterpret_cast<uint2*>(a.v + row * kHeadDim)[lane] = reinterpret_cast<const uint2*>(vn)[lane];
    if (a.kept_idx != nullptr && lane == 0)
      a.kept_idx[(int64_t)bh * a.cap + n] = a.position + (a.position_plus_count ? n : 0);
    if (BITS != 16 && (n % kGroup) == kGroup - 1) {
      __syncwarp();
      __threadfence_block();
      const __nv_bfloat16* kt = a.k + (int64_t)bh * kGroup * kHeadDim;
      const __nv_bfloat16* vt = a.v + (int64_t)bh * kGroup * kHeadDim;
      auto krow = [&](int t) { return kt + t * kHeadDim; };
      auto vrow = [&](int t) { return vt + t * kHeadDim; };
      __shared__ QuantStats smem[8];
      QuantOut out;
      out.k_codes = a.k_codes + (size_t)bh * a.cap * kHeadDim * (BITS > 0 ? BITS : 1) / 8;
      out.k_params = a.k_params + (size_t)bh * (a.cap / kGroup) * 512;
      out.v_codes = a.v_codes + (size_t)bh * a.cap * kHeadDim * (BITS > 0 ? BITS : 1) / 8;
      out.v_params = a.v_params + (size_t)bh * a.cap * 16;
      if (!quantize_group_warp<(BITS == 16 ? 4 : BITS)>(krow, vrow, n / kGroup, out, smem[j]))
        if (lane == 0) set_status(a.status, UC_ERR_RANGE, 4);
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) a.n_kept[b] = n + 1;
}

// ---------------------------------------------------------------- launchers

void launch_topk(const TopkArgs& a, int n_blocks, bool evict, cudaStream_t st) {
  int max_src = 0;
  for (int b = 0; b < UC_MAX_BATCH; ++b) max_src = std::max(max_src, a.src_n[b]);
  if (evict && max_src >= kTopkClusterMinN && n_blocks <= kTopkClusterMaxPairs)
    topk_cluster_kernel<<<n_blocks * kTopkCluster, kTopkThreads, 0, st>>>(a);
  else if (evict)
    topk_select_kernel<<<n_blocks, kTopkThreads, 0, st>>>(a);
  else
    iota_kernel<<<n_blocks, 256, 0, st>>>(a);
  count_launch();
}

void launch_dequant_rows(const DequantArgs& a, cudaStream_t st) {
  const int warps = a.batch * a.n_kv_heads * a.max_groups;
  if (a.bits == 4)
    dequant_rows_kernel<4><<<(warps + 3) / 4, 128, 0, st>>>(a);
  else
    dequant_rows_kernel<2><<<(warps + 3) / 4, 128, 0, st>>>(a);
  count_launch();
}

void launch_compose_idx(const ComposeArgs& a, int nbh, cudaStream_t st) {
  compose_idx_kernel<<<nbh, 256, 0, st>>>(a);
  count_launch();
}

void launch_gather(const GatherArgs& a, cudaStream_t st) {
  const int warps = a.batch * a.n_kv_heads * a.max_chunks;
  gather_rows_kernel<<<(warps + 3) / 4, 128, 0, st>>>(a);
  count_launch();
}

void launch_quantize(const GatherArgs& a, int bits, cudaStream_t st) {
  static int sms = 0;
  static bool attr4 = false, attr2 = false;
  if (sms == 0) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    sms = std::max(sms, 1);
  }
  const int warps = a.batch * a.n_kv_heads * a.max_chunks;
  const int blocks = std::min((warps + kQuantWarps - 1) / kQuantWarps, kQuantCtasPerSm * sms);
  if (blocks > 0) {
    if (bits == 4) {
      if (!attr4)
        attr4 = cudaFuncSetAttribute(quantize_groups_kernel<4>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)kQuantSmemBytes) == cudaSuccess;
      quantize_groups_kernel<4><<<blocks, kQuantWarps * 32, kQuantSmemBytes, st>>>(a);
    } else {
      if (!attr2)
        attr2 = cudaFuncSetAttribute(quantize_groups_kernel<2>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)kQuantSmemBytes) == cudaSuccess;
      quantize_groups_kernel<2><<<blocks, kQuantWarps * 32, kQuantSmemBytes, st>>>(a);
    }
    count_launch();
  }
  const int tw = a.batch * a.n_kv_heads;
  copy_tail_kernel<<<(tw + 3) / 4, 128, 0, st>>>(a);
  count_launch();
}

void launch_append(const AppendArgs& a, int bits, cudaStream_t st) {
  const int threads = 32 * ((a.n_kv_heads + 0) > 8 ? 8 : a.n_kv_heads);
  const bool pdl = pdl_enabled();
  if (bits == 4)
    launch_maybe_pdl(pdl, append_token_kernel<4>, a.batch, threads, 0, st, a);
  else if (bits == 2)
    launch_maybe_pdl(pdl, append_token_kernel<2>, a.batch, threads, 0, st, a);
  else
    launch_maybe_pdl(pdl, append_token_kernel<16>, a.batch, threads, 0, st, a);
  count_launch();
}

}  // namespace uc
