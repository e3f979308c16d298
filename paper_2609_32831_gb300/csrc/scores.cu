// Observation-window attention scores (§3.3 Eq. 1's P, summed per KV head as
// in App. E "Batched GQA token selection"):
//   scores[b, j, t] = sum over the g query heads of KV head j and the W window
//                     queries of softmax_t(q . k_t / sqrt(128))
//
// Two passes over K, both on the 5th-generation tensor cores (tcgen05.mma,
// bf16 operands from shared memory, fp32 accumulators in tensor memory):
//   pass 1: per query row, an online max / sum of exp2 over this CTA's keys;
//   merge : per row, log2-sum-exp over the key chunks;
//   pass 2: recompute the logits (transposed, one key per TMEM lane) and add
//           exp2(x - lse) over each key's query rows.
// K tiles of 128 tokens stream through a 3-stage TMA ring (128-byte swizzle);
// the window queries sit in shared memory for the whole CTA.
#include <mutex>

#include "common.cuh"
#include "internal.h"
#include "tcgen05.cuh"

namespace uc {

constexpr int kScTile = 128;     // keys per tile
constexpr int kScStages = 3;     // K ring
constexpr int kScCompute = 16;   // compute warps: four warpgroups
constexpr int kScThreads = 32 * (kScCompute + 2);  // + warp 16: TMA, 17: MMA
constexpr int kScTmaWarp = kScCompute, kScMmaWarp = kScCompute + 1;
constexpr int kScMaxRows = 256;
constexpr uint32_t kScTmemCols = 512;

// Shared memory: window queries as a K-major, 128-byte-swizzled operand
// ([channel half][256 rows][128 B]), the K ring ([channel half][128 keys]
// [128 B] per slot, as TMA writes it), pass 2's per-key partial sums and
// per-row lse.
struct ScoreSmem {
  uint8_t q[2][kScMaxRows * 128];
  uint8_t k[kScStages][2][kScTile * 128];
  float part[2][2][kScTile];      // pass 2: per pair, the second half's key sums (double-buffered)
  float2 ml[2][kScMaxRows];       // pass 1: (max, sum) of each row's two key halves
  float lse2[kScMaxRows];
  uint64_t k_full[kScStages], k_empty[kScStages];
  uint64_t s_full[2], s_free[2];
  uint32_t tmem_base;
};

__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

__device__ __forceinline__ void sc_sync() { asm volatile("bar.sync 1, 512;" ::: "memory"); }
// the 256 threads of compute pair p
__device__ __forceinline__ void sc_pair_sync(int p) { asm volatile("bar.sync %0, 256;" ::"r"(2 + p) : "memory"); }

__device__ __forceinline__ bool sc_wait_warp(uint64_t* bar, uint32_t parity, DevStatus* st, int where,
                                             bool& aborted) {
  if (!aborted && !mbar_wait(bar, parity, st, where)) aborted = true;
  aborted = __any_sync(0xffffffffu, aborted);
  return !aborted;
}

// D = A B^T over the 8 K steps of d = 128 (16 channels each): A and B step
// 32 B inside their 128-B swizzled rows, then jump to their second channel
// half (offsets in units of 16 B).
template <int AH, int BH>
__device__ __forceinline__ void sc_issue(uint32_t d, uint32_t a_lo, uint32_t b_lo, uint32_t hi, uint32_t idesc) {
  umma_ss_off<0, 0, 0>(d, a_lo, b_lo, hi, idesc);
  umma_ss_off<2, 2, 1>(d, a_lo, b_lo, hi, idesc);
  umma_ss_off<4, 4, 1>(d, a_lo, b_lo, hi, idesc);
  umma_ss_off<6, 6, 1>(d, a_lo, b_lo, hi, idesc);
  umma_ss_off<AH, BH, 1>(d, a_lo, b_lo, hi, idesc);
  umma_ss_off<AH + 2, BH + 2, 1>(d, a_lo, b_lo, hi, idesc);
  umma_ss_off<AH + 4, BH + 4, 1>(d, a_lo, b_lo, hi, idesc);
  umma_ss_off<AH + 6, BH + 6, 1>(d, a_lo, b_lo, hi, idesc);
}

// Both passes on the 5th-generation tensor cores, bf16 operands, fp32 in
// tensor memory. One CTA per (b, kvh, chunk of 128-key tiles).
//   pass 1: S = Q K^T, M = 128 query rows per tile (two tiles cover up to
//           256 rows), N = 128 keys; each compute thread owns one query row
//           (= TMEM lane) of every other key tile and keeps an online max /
//           sum of exp2; the row's two sets of tiles meet in shared memory;
//   pass 2: S^T = K Q^T, M = 128 keys, N = 256 query rows; each thread owns
//           one key of every other tile and sums exp2(x - lse) over its
//           warpgroup's half of the query rows; the halves meet in shared
//           memory.
// S is double-buffered in TMEM (512 columns) so the next tile's MMAs run
// while this tile is read.
template <bool PASS2>
__global__ void __launch_bounds__(kScThreads, 1) score_kernel(const __grid_constant__ ScoreArgs a) {
  extern __shared__ uint8_t dyn_smem[];
  ScoreSmem& sm = *reinterpret_cast<ScoreSmem*>(
      (reinterpret_cast<uintptr_t>(dyn_smem) + 1023) & ~static_cast<uintptr_t>(1023));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int bh = blockIdx.x / a.chunks, chunk = blockIdx.x % a.chunks;
  const int b = bh / a.n_kv_heads, kvh = bh % a.n_kv_heads;
  const int group = a.n_q_heads / a.n_kv_heads;
  const int n_tiles = (a.n_ctx + kScTile - 1) / kScTile;
  const int t_begin = chunk * a.tiles_per_chunk;
  const int t_end = min(n_tiles, t_begin + a.tiles_per_chunk);
  const int rows_pad = 16 * a.mtiles;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kScStages; ++s) {
      mbar_init(&sm.k_full[s], 1);
      mbar_init(&sm.k_empty[s], 1);
    }
    for (int x = 0; x < 2; ++x) {
      mbar_init(&sm.s_full[x], 1);
      mbar_init(&sm.s_free[x], kScCompute / 2);  // the pair that reads buffer x
    }
    fence_barrier_init();
  }
  if (warp == kScMmaWarp) tmem_alloc(&sm.tmem_base, kScTmemCols);
  if (warp < kScCompute) {
    // window queries -> shared memory: row r = hl * W + w (zero past the
    // window rows), K-major with the 128-byte swizzle the MMA reads
    for (int idx = threadIdx.x; idx < kScMaxRows * 16; idx += 32 * kScCompute) {
      const int r = idx >> 4, c = idx & 15;
      uint4 v = make_uint4(0, 0, 0, 0);
      if (r < a.rows) {
        const int hl = r / a.window, w = r % a.window;
        v = *reinterpret_cast<const uint4*>(
            a.qwin + ((size_t)(b * a.n_q_heads + kvh * group + hl) * a.window + w) * kHeadDim + c * 8);
      }
      *reinterpret_cast<uint4*>(sm.q[c >> 3] + r * 128 + (((c & 7) ^ (r & 7)) << 4)) = v;
    }
    if (PASS2)
      for (int r = threadIdx.x; r < kScMaxRows; r += 32 * kScCompute)
        sm.lse2[r] = r < a.rows ? a.lse2[(size_t)bh * rows_pad + r] : INFINITY;
    fence_proxy_async_smem();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sm.tmem_base;
  bool aborted = false;

  if (warp == kScTmaWarp) {
    if (lane == 0) {
      // ------------------------------------------------------ TMA producer
      prefetch_tmap(&a.tmap_k);
      uint32_t seq = 0;
      for (int t = t_begin; t < t_end; ++t, ++seq) {
        const int slot = seq % kScStages;
        if (seq >= kScStages && !mbar_wait(&sm.k_empty[slot], ((seq / kScStages) - 1) & 1, a.status, 20)) break;
        const int row = (int)((int64_t)bh * a.k_row_stride + (int64_t)t * kScTile);
        mbar_arrive_expect_tx(&sm.k_full[slot], 2 * kScTile * 128);
        tma_load_2d(sm.k[slot][0], &a.tmap_k, 0, row, &sm.k_full[slot]);
        tma_load_2d(sm.k[slot][0] + 64 * 128, &a.tmap_k, 0, row + 64, &sm.k_full[slot]);
        tma_load_2d(sm.k[slot][1], &a.tmap_k, 64, row, &sm.k_full[slot]);
        tma_load_2d(sm.k[slot][1] + 64 * 128, &a.tmap_k, 64, row + 64, &sm.k_full[slot]);
      }
    }
  } else if (warp == kScMmaWarp) {
    if (lane == 0) {
      // ------------------------------------------------------ MMA issue
      const uint32_t hi = (uint32_t)(smem_desc_sw128(0, 16) >> 32);
      const uint32_t q_lo = (uint32_t)smem_desc_sw128(smem_u32(sm.q[0]), 16);
      const int xt = (a.rows + 127) / 128;  // query-row tiles of pass 1
      uint32_t seq = 0;
      for (int t = t_begin; t < t_end; ++t, ++seq) {
        const int slot = seq % kScStages, buf = seq & 1;
        if (!mbar_wait(&sm.k_full[slot], (seq / kScStages) & 1, a.status, 22)) break;
        if (seq >= 2 && !mbar_wait(&sm.s_free[buf], ((seq >> 1) - 1) & 1, a.status, 23)) break;
        tc_fence_after();
        const uint32_t k_lo = (uint32_t)smem_desc_sw128(smem_u32(sm.k[slot][0]), 16);
        const uint32_t d = tmem + buf * 256;
        if (!PASS2) {
          constexpr uint32_t id = idesc_bf16(128, kScTile, 0, 0);
          // Q rows 128x .. : 16 KB further in each channel half (32 KB apart)
          sc_issue<2048, 1024>(d, q_lo, k_lo, hi, id);
          if (xt > 1) sc_issue<2048, 1024>(d + 128, q_lo + (16384 >> 4), k_lo, hi, id);
        } else {
          constexpr uint32_t id = idesc_bf16(kScTile, kScMaxRows, 0, 0);
          sc_issue<1024, 2048>(d, k_lo, q_lo, hi, id);
        }
        umma_commit(&sm.k_empty[slot]);
        umma_commit(&sm.s_full[buf]);
      }
    }
  } else {
    // ------------------------------------------------------ compute warps
    // Four warpgroups in two pairs: pair p reads the S tiles in TMEM buffer p
    // (every other tile), so one pair's tensor-memory loads overlap the
    // other pair's exp2 work. Pass 1: warpgroup w takes row tile w % 2 of its
    // pair's tiles; pass 2: the query rows (columns of S^T) 128 (w % 2) ..
    // 128 (w % 2) + 127. Each tile is read in two 64-column chunks.
    const int wg = warp >> 2, par = wg >> 1, hw = wg & 1;
    const uint32_t lane_off = (uint32_t)(32 * (warp & 3)) << 16;
    const float sl2 = a.scale_log2;
    if (!PASS2) {
      const int row = hw * 128 + 32 * (warp & 3) + lane;  // query row = TMEM lane of S tile hw
      const bool active = hw * 128 + 32 * (warp & 3) < a.rows;
      float m_ref = -INFINITY, l = 0.f;
      uint32_t seq = par;
      for (int t = t_begin + par; t < t_end; t += 2, seq += 2) {
        const int buf = par;
        if (!sc_wait_warp(&sm.s_full[buf], (seq >> 1) & 1, a.status, 24, aborted)) break;
        tc_fence_after();
        const int valid_t = min(kScTile, a.n_ctx - t * kScTile);
        if (active) {
#pragma unroll 1
          for (int kh = 0; kh < 2; ++kh) {
            const int valid = valid_t - 64 * kh;
            if (valid <= 0) break;
            uint32_t sr[2][32];
#pragma unroll
            for (int c = 0; c < 2; ++c) tmem_ld32(tmem + lane_off + buf * 256 + hw * 128 + kh * 64 + 32 * c, sr[c]);
            tmem_wait_ld();
            // the chunk's max on the raw logits (sl2 > 0), two per 3-input max
            if (valid < 64) {
#pragma unroll
              for (int c = 0; c < 2; ++c)
#pragma unroll
                for (int e = 0; e < 32; ++e)
                  if (32 * c + e >= valid) sr[c][e] = __float_as_uint(-INFINITY);
            }
            float mr[2] = {-INFINITY, -INFINITY};
#pragma unroll
            for (int c = 0; c < 2; ++c)
#pragma unroll
              for (int e = 0; e < 32; e += 2)
                mr[c] = fmax3(mr[c], __uint_as_float(sr[c][e]), __uint_as_float(sr[c][e + 1]));
            const float mx = fmaxf(mr[0], mr[1]) * sl2;
            // reference max moved only when exceeded by more than 8
            if (mx > m_ref + 8.f) {
              l = (m_ref == -INFINITY) ? 0.f : l * ex2_approx(m_ref - mx);
              m_ref = mx;
            }
            const float nm = -m_ref;
            float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
            for (int c = 0; c < 2; ++c)
#pragma unroll
              for (int e = 0; e < 32; ++e)
                acc[(c << 1) | (e & 1)] += ex2_approx(fmaf(__uint_as_float(sr[c][e]), sl2, nm));
            l += (acc[0] + acc[1]) + (acc[2] + acc[3]);
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&sm.s_free[buf]);
      }
      // the row's two pairs meet in shared memory
      sm.ml[par][row] = make_float2(m_ref, l);
      sc_sync();
      if (par == 0 && row < rows_pad) {
        const float2 o = sm.ml[1][row];
        const float m = fmaxf(m_ref, o.x);
        const float mu = (m == -INFINITY) ? 0.f : m;
        const float lt = (m_ref == -INFINITY ? 0.f : l * exp2f(m_ref - mu)) + (o.x == -INFINITY ? 0.f : o.y * exp2f(o.x - mu));
        float* pp = a.part + ((size_t)blockIdx.x * rows_pad + row) * 2;
        pp[0] = m;
        pp[1] = lt;
      }
    } else {
      const int key = 32 * (warp & 3) + lane;  // TMEM lane of S^T
      uint32_t seq = par;
      for (int t = t_begin + par; t < t_end; t += 2, seq += 2) {
        const int buf = par;
        // on a timeout the loop still runs to the end without waiting, so
        // that both warpgroups of the pair take the same number of barriers
        const bool ok = sc_wait_warp(&sm.s_full[buf], (seq >> 1) & 1, a.status, 25, aborted);
        tc_fence_after();
        float sum = 0.f;
        if (ok) {
#pragma unroll 1
          for (int ch = 0; ch < 2; ++ch) {
            const int col0 = 128 * hw + 64 * ch;  // query rows of this chunk (lse = +inf past the window)
            if (col0 >= a.rows) break;
            uint32_t sr[2][32];
#pragma unroll
            for (int c = 0; c < 2; ++c) tmem_ld32(tmem + lane_off + buf * 256 + col0 + 32 * c, sr[c]);
            tmem_wait_ld();
            float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
            for (int c = 0; c < 2; ++c)
#pragma unroll
              for (int e = 0; e < 32; ++e)
                acc[(c << 1) | (e & 1)] += ex2_approx(fmaf(__uint_as_float(sr[c][e]), sl2, -sm.lse2[col0 + 32 * c + e]));
            sum += (acc[0] + acc[1]) + (acc[2] + acc[3]);
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&sm.s_free[buf]);
        // the pair's two row halves of the key meet in shared memory (double
        // buffered: one warpgroup of the pair is at most one tile ahead)
        const int pb = (seq >> 1) & 1;
        if (hw == 1) sm.part[par][pb][key] = sum;
        sc_pair_sync(par);
        const int valid = min(kScTile, a.n_ctx - t * kScTile);
        if (ok && hw == 0 && key < valid)
          a.scores[(size_t)bh * a.n_ctx + (size_t)t * kScTile + key] = sum + sm.part[par][pb][key];
      }
    }
  }
  __syncwarp();
  __syncthreads();
  if (warp == kScMmaWarp) {
    tc_fence_after();
    tmem_dealloc(tmem, kScTmemCols);
  }
}

// Per (b, kvh, row): log2-sum-exp over the key chunks; rows past the window
// get +inf so that pass 2 gives them zero probability.
__global__ void score_merge_kernel(const __grid_constant__ ScoreArgs a) {
  const int bh = blockIdx.x;
  const int rows_pad = 16 * a.mtiles;
  for (int r = threadIdx.x; r < rows_pad; r += blockDim.x) {
    float out = INFINITY;
    if (r < a.rows) {
      float M = -INFINITY;
      for (int c = 0; c < a.chunks; ++c)
        M = fmaxf(M, a.part[((size_t)(bh * a.chunks + c) * rows_pad + r) * 2]);
      float L = 0.f;
      for (int c = 0; c < a.chunks; ++c) {
        const float* pp = a.part + ((size_t)(bh * a.chunks + c) * rows_pad + r) * 2;
        if (pp[0] != -INFINITY) L += pp[1] * exp2f(pp[0] - M);
      }
      out = M + log2f(L);
    }
    a.lse2[(size_t)bh * rows_pad + r] = out;
  }
}

// mass[b, s] = sum_{j, t in [begin_s, end_s)} scores[b, j, t] * inv_norm
struct MassArgs {
  const float* scores;
  float* mass;
  int n_kv_heads, n_ctx, n_seg;
  int begin[UC_MAX_SEGMENTS], end[UC_MAX_SEGMENTS];
  float inv_norm;
  int accumulate;
};

// One block per (sequence, segment); 8 independent partial sums per thread
// keep enough loads in flight. Summation order is fixed (deterministic).
__global__ void __launch_bounds__(1024) segment_mass_kernel(const __grid_constant__ MassArgs a) {
  const int b = blockIdx.x / a.n_seg, s = blockIdx.x % a.n_seg;
  const int lo = a.begin[s], n = a.end[s] - a.begin[s];
  float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  for (int j = 0; j < a.n_kv_heads; ++j) {
    const float* row = a.scores + (size_t)(b * a.n_kv_heads + j) * a.n_ctx + lo;
    for (int t0 = threadIdx.x; t0 < n; t0 += 8 * blockDim.x) {
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int t = t0 + u * blockDim.x;
        if (t < n) acc[u] += row[t];
      }
    }
  }
  float tot = ((acc[0] + acc[1]) + (acc[2] + acc[3])) + ((acc[4] + acc[5]) + (acc[6] + acc[7]));
  __shared__ float red[32];
  for (int o = 16; o > 0; o >>= 1) tot += __shfl_xor_sync(0xffffffffu, tot, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = tot;
  __syncthreads();
  if (threadIdx.x == 0) {
    float t = 0.f;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) t += red[w];
    const float v = t * a.inv_norm;
    a.mass[blockIdx.x] = a.accumulate ? a.mass[blockIdx.x] + v : v;
  }
}

// Eq. 1 from the attention call's own probabilities: one block per sequence
// b sums mass[b, h, t, s] over all (h, t) for each segment s.
__global__ void __launch_bounds__(512) attention_mass_kernel(const float* __restrict__ mass, int rows,
                                                             int n_seg, float scale, int accumulate,
                                                             float* __restrict__ out) {
  const int b = blockIdx.x;
  const float* m = mass + (size_t)b * rows * n_seg;
  float acc[UC_MAX_SEGMENTS];
#pragma unroll
  for (int s = 0; s < UC_MAX_SEGMENTS; ++s) acc[s] = 0.f;
  for (int i = threadIdx.x; i < rows; i += blockDim.x) {
#pragma unroll
    for (int s = 0; s < UC_MAX_SEGMENTS; ++s)
      if (s < n_seg) acc[s] += m[(size_t)i * n_seg + s];
  }
  __shared__ float red[16][UC_MAX_SEGMENTS];
#pragma unroll
  for (int s = 0; s < UC_MAX_SEGMENTS; ++s) {
    float v = acc[s];
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5][s] = v;
  }
  __syncthreads();
  if (threadIdx.x < n_seg) {
    float t = 0.f;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) t += red[w][threadIdx.x];
    float* o = out + (size_t)b * n_seg + threadIdx.x;
    *o = accumulate ? *o + t * scale : t * scale;
  }
}

// Heavy-hitter statistics of one decode step: one CTA per (b, kvh, 64-token
// chunk) stages the g * T query rows and their lse in shared memory; a warp
// takes one stored token at a time (lane L holds channels 4L .. 4L + 3),
// forms every row's logit with a shuffle reduction and adds
// sum_rows exp(logit - lse) to the token's accumulator slot. Each token has
// one writer, so the result does not depend on scheduling.
constexpr int kDsTokens = 64;
constexpr int kDsMaxRows = UC_MAX_QTOKENS * 8;

__global__ void __launch_bounds__(256) decode_score_kernel(const __grid_constant__ DecodeScoreArgs a) {
  __shared__ float qs[kDsMaxRows][kHeadDim];
  __shared__ float lse[kDsMaxRows];
  const int bh = blockIdx.x;
  const int b = bh / a.n_kv_heads, kvh = bh % a.n_kv_heads;
  const int n = a.n_kept[b];
  const int t0 = blockIdx.y * kDsTokens;
  if (t0 >= n) return;
  for (int x = threadIdx.x; x < a.rows * kHeadDim; x += blockDim.x) {
    const int r = x / kHeadDim, c = x % kHeadDim;
    const int h = kvh * a.group + r / a.n_qtok, tau = r % a.n_qtok;
    qs[r][c] = __bfloat162float(a.q[(((size_t)b * a.n_q_heads + h) * a.n_qtok + tau) * kHeadDim + c]) * a.scale;
  }
  for (int r = threadIdx.x; r < a.rows; r += blockDim.x) {
    const int h = kvh * a.group + r / a.n_qtok, tau = r % a.n_qtok;
    lse[r] = a.lse[((size_t)b * a.n_q_heads + h) * a.n_qtok + tau];
  }
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int t_end = min(n, t0 + kDsTokens);
  for (int t = t0 + warp; t < t_end; t += blockDim.x >> 5) {
    const uint2 raw = *reinterpret_cast<const uint2*>(
        a.k + ((int64_t)bh * a.row_stride + a.row_offset + t) * kHeadDim + 4 * lane);
    const __nv_bfloat162 k01 = *reinterpret_cast<const __nv_bfloat162*>(&raw.x);
    const __nv_bfloat162 k23 = *reinterpret_cast<const __nv_bfloat162*>(&raw.y);
    const float k0 = __low2float(k01), k1 = __high2float(k01), k2 = __low2float(k23), k3 = __high2float(k23);
    float p = 0.f;
    for (int r = 0; r < a.rows; ++r) {
      const float4 qv = *reinterpret_cast<const float4*>(&qs[r][4 * lane]);
      float d = fmaf(qv.x, k0, fmaf(qv.y, k1, fmaf(qv.z, k2, qv.w * k3)));
      for (int o = 16; o > 0; o >>= 1) d += __shfl_xor_sync(0xffffffffu, d, o);
      p += expf(d - lse[r]);
    }
    if (lane == 0) {
      const int64_t idx = a.kept_idx ? (int64_t)a.kept_idx[(int64_t)bh * a.cap + t] : (int64_t)t;
      const int64_t slot = a.acc_offset + idx;
      if (idx < 0 || slot >= a.acc_stride)
        set_status(a.status, UC_ERR_RANGE, 3);
      else
        a.acc[(int64_t)bh * a.acc_stride + slot] += p;
    }
  }
}

void launch_decode_scores(const DecodeScoreArgs& a, int batch, int max_tokens, cudaStream_t st) {
  if (max_tokens <= 0) return;
  dim3 grid(batch * a.n_kv_heads, (max_tokens + kDsTokens - 1) / kDsTokens);
  decode_score_kernel<<<grid, 256, 0, st>>>(a);
  count_launch();
}

void launch_attention_mass(const float* mass, int batch, int rows, int n_seg, float scale,
                           bool accumulate, float* out, cudaStream_t st) {
  attention_mass_kernel<<<batch, 512, 0, st>>>(mass, rows, n_seg, scale, accumulate ? 1 : 0, out);
  count_launch();
}

void launch_scores(const ScoreArgs& a, cudaStream_t st) {
  const size_t smem = sizeof(ScoreSmem) + 1024;
  static std::once_flag once;
  std::call_once(once, [smem] {
    cudaFuncSetAttribute(score_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    cudaFuncSetAttribute(score_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  });
  const int grid = a.batch * a.n_kv_heads * a.chunks;
  score_kernel<false><<<grid, kScThreads, smem, st>>>(a);
  count_launch();
  score_merge_kernel<<<a.batch * a.n_kv_heads, 256, 0, st>>>(a);
  count_launch();
  score_kernel<true><<<grid, kScThreads, smem, st>>>(a);
  count_launch();
}

void launch_segment_mass(const float* scores, int batch, int n_kv_heads, int n_ctx,
                         const int32_t* begin, const int32_t* end, int n_seg, float inv_norm,
                         bool accumulate, float* mass, cudaStream_t st) {
  MassArgs a;
  a.scores = scores;
  a.mass = mass;
  a.n_kv_heads = n_kv_heads;
  a.n_ctx = n_ctx;
  a.n_seg = n_seg;
  for (int s = 0; s < n_seg; ++s) {
    a.begin[s] = begin[s];
    a.end[s] = end[s];
  }
  a.inv_norm = inv_norm;
  a.accumulate = accumulate ? 1 : 0;
  segment_mass_kernel<<<batch * n_seg, 1024, 0, st>>>(a);
  count_launch();
}

}  // namespace uc
