// Observation-window attention scores (§3.3 Eq. 1's P, summed per KV head as
// in App. E "Batched GQA token selection"):
//   scores[b, j, t] = sum over the g query heads of KV head j and the W window
//                     queries of softmax_t(q . k_t / sqrt(128))
//
// Two passes over K, both on the tensor cores (mma.sync m16n8k16, bf16 in,
// fp32 accumulate):
//   pass 1: per query row, an online max / sum of exp2 over this CTA's keys;
//   merge : per row, log2-sum-exp over the key chunks;
//   pass 2: recompute the logits and add exp2(x - lse) down each key's column.
// K tiles of 64 tokens stream through a 3-stage TMA ring (128-byte swizzle);
// the window queries sit in shared memory for the whole CTA.
#include <mutex>

#include "common.cuh"
#include "internal.h"

namespace uc {

constexpr int kScTile = 64;
constexpr int kScStages = 3;
constexpr int kScConsumers = 8;
constexpr int kScThreads = 32 * (kScConsumers + 1);
constexpr int kScMaxRows = 256;

struct ScoreSmem {
  uint8_t ring[kScStages][16384];
  uint8_t q[kScMaxRows * 256];
  float colsum[2][kScConsumers][kScTile];  // pass 2: double-buffered per tile
  uint64_t full[kScStages];
  uint64_t empty[kScStages];
};

__device__ __forceinline__ void sc_sync() { asm volatile("bar.sync 1, 256;" ::: "memory"); }

__device__ __forceinline__ uint32_t sc_swz(uint32_t base, int key, int chunk) {
  return base + (chunk >> 3) * 8192 + key * 128 + ((((chunk & 7) ^ (key & 7))) << 4);
}

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

  if (threadIdx.x == 0) {
    for (int s = 0; s < kScStages; ++s) {
      mbar_init(&sm.full[s], 1);
      mbar_init(&sm.empty[s], kScConsumers);
    }
    fence_barrier_init();
  }
  __syncthreads();

  if (warp == kScConsumers) {
    if (lane == 0) {
      prefetch_tmap(&a.tmap_k);
      uint32_t seq = 0;
      for (int t = t_begin; t < t_end; ++t, ++seq) {
        const int slot = seq % kScStages;
        if (seq >= kScStages && !mbar_wait(&sm.empty[slot], ((seq / kScStages) - 1) & 1, a.status, 20))
          return;
        const int row = (int)((int64_t)bh * a.k_row_stride + (int64_t)t * kScTile);
        mbar_arrive_expect_tx(&sm.full[slot], 16384);
        tma_load_2d(sm.ring[slot], &a.tmap_k, 0, row, &sm.full[slot]);
        tma_load_2d(sm.ring[slot] + 8192, &a.tmap_k, 64, row, &sm.full[slot]);
      }
    }
    return;
  }

  // window queries -> shared memory, rows r = hl * W + w, swizzled 16-B chunks
  const int rows_pad = 16 * a.mtiles;
  for (int idx = threadIdx.x; idx < rows_pad * 16; idx += 32 * kScConsumers) {
    const int r = idx >> 4, c = idx & 15;
    uint4 v = make_uint4(0, 0, 0, 0);
    if (r < a.rows) {
      const int hl = r / a.window, w = r % a.window;
      const __nv_bfloat16* src =
          a.qwin + ((size_t)(b * a.n_q_heads + kvh * group + hl) * a.window + w) * kHeadDim + c * 8;
      v = *reinterpret_cast<const uint4*>(src);
    }
    *reinterpret_cast<uint4*>(sm.q + r * 256 + ((c ^ (r & 7)) << 4)) = v;
  }
  sc_sync();

  const int g = lane >> 2, j = lane & 3, mi = lane >> 3, rr = lane & 7;
  const int mt0 = 2 * warp;
  const bool has0 = mt0 < a.mtiles, has1 = mt0 + 1 < a.mtiles;
  const uint32_t qbase = smem_u32(sm.q);

  // A fragments of the warp's two m-tiles
  uint32_t qa[2][8][4];
#pragma unroll
  for (int m = 0; m < 2; ++m) {
    const int row = (mt0 + m) * 16 + 8 * (mi & 1) + rr;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      if ((m == 0 && has0) || (m == 1 && has1)) {
        const int c = 2 * i + (mi >> 1);
        ldsm_x4(qbase + row * 256 + ((c ^ (row & 7)) << 4), qa[m][i][0], qa[m][i][1], qa[m][i][2],
                qa[m][i][3]);
      } else {
        qa[m][i][0] = qa[m][i][1] = qa[m][i][2] = qa[m][i][3] = 0u;
      }
    }
  }

  // per-thread rows: (m, half) -> row (mt0 + m) * 16 + g + 8 * half
  float rm[2][2], rl[2][2], lse[2][2];
#pragma unroll
  for (int m = 0; m < 2; ++m)
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      rm[m][h] = -INFINITY;
      rl[m][h] = 0.f;
      lse[m][h] = INFINITY;
      if (PASS2) {
        const int row = (mt0 + m) * 16 + g + 8 * h;
        if (row < a.rows) lse[m][h] = a.lse2[(size_t)bh * rows_pad + row];
      }
    }

  uint32_t seq = 0;
  for (int t = t_begin; t < t_end; ++t, ++seq) {
    const int slot = seq % kScStages;
    bool ok = mbar_wait(&sm.full[slot], (seq / kScStages) & 1, a.status, 21);
    const uint32_t kbase = smem_u32(sm.ring[slot]);
    const int valid = min(kScTile, a.n_ctx - t * kScTile);
    if (ok && has0) {
#pragma unroll 1
      for (int u = 0; u < 4; ++u) {
        float s[2][2][4];
#pragma unroll
        for (int m = 0; m < 2; ++m)
#pragma unroll
          for (int nt = 0; nt < 2; ++nt) s[m][nt][0] = s[m][nt][1] = s[m][nt][2] = s[m][nt][3] = 0.f;
        const int kk = 16 * u + 8 * (mi >> 1) + rr;
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          uint32_t b0, b1, b2, b3;
          ldsm_x4(sc_swz(kbase, kk, 2 * i + (mi & 1)), b0, b1, b2, b3);
          mma_bf16(s[0][0], qa[0][i], b0, b1);
          mma_bf16(s[0][1], qa[0][i], b2, b3);
          if (has1) {
            mma_bf16(s[1][0], qa[1][i], b0, b1);
            mma_bf16(s[1][1], qa[1][i], b2, b3);
          }
        }
        float cs[2][2] = {{0.f, 0.f}, {0.f, 0.f}};  // pass 2: column sums (n-tile, e)
#pragma unroll
        for (int m = 0; m < 2; ++m) {
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            float x[4];
#pragma unroll
            for (int nt = 0; nt < 2; ++nt)
#pragma unroll
              for (int e = 0; e < 2; ++e) {
                const bool kv = 16 * u + 8 * nt + 2 * j + e < valid;
                x[2 * nt + e] = kv ? s[m][nt][2 * h + e] * a.scale_log2 : -INFINITY;
              }
            if (!PASS2) {
              // online sum with a reference max that moves only when a row's
              // max exceeds it by more than 8 (terms <= 2^8, rescaled rarely)
              float mx = fmaxf(fmaxf(x[0], x[1]), fmaxf(x[2], x[3]));
              mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
              mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
              if (mx > rm[m][h] + 8.f) {
                rl[m][h] = (rm[m][h] == -INFINITY) ? 0.f : rl[m][h] * ex2_approx(rm[m][h] - mx);
                rm[m][h] = mx;
              }
              const float um = (rm[m][h] == -INFINITY) ? 0.f : rm[m][h];
              rl[m][h] += (ex2_approx(x[0] - um) + ex2_approx(x[1] - um)) + (ex2_approx(x[2] - um) + ex2_approx(x[3] - um));
            } else {
#pragma unroll
              for (int nt = 0; nt < 2; ++nt)
#pragma unroll
                for (int e = 0; e < 2; ++e) cs[nt][e] += ex2_approx(x[2 * nt + e] - lse[m][h]);
            }
          }
        }
        if (PASS2) {
#pragma unroll
          for (int nt = 0; nt < 2; ++nt)
#pragma unroll
            for (int e = 0; e < 2; ++e) {
              float c = cs[nt][e];
              c += __shfl_xor_sync(0xffffffffu, c, 4);
              c += __shfl_xor_sync(0xffffffffu, c, 8);
              c += __shfl_xor_sync(0xffffffffu, c, 16);
              if (g == 0) sm.colsum[seq & 1][warp][16 * u + 8 * nt + 2 * j + e] = c;
            }
        }
      }
    } else if (PASS2) {
      if (lane < 16)
        for (int u = 0; u < 4; ++u) sm.colsum[seq & 1][warp][16 * u + lane] = 0.f;
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&sm.empty[slot]);
    if (PASS2) {
      // one barrier per tile: the sums of tile t are read while tile t + 1
      // writes the other buffer (a warp can be at most one tile ahead)
      sc_sync();
      if (threadIdx.x < kScTile && threadIdx.x < valid) {
        float sum = 0.f;
#pragma unroll
        for (int w = 0; w < kScConsumers; ++w) sum += sm.colsum[seq & 1][w][threadIdx.x];
        a.scores[(size_t)bh * a.n_ctx + (size_t)t * kScTile + threadIdx.x] = sum;
      }
    }
  }

  if (!PASS2) {
#pragma unroll
    for (int m = 0; m < 2; ++m)
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        float l = rl[m][h];
        l += __shfl_xor_sync(0xffffffffu, l, 1);
        l += __shfl_xor_sync(0xffffffffu, l, 2);
        const int row = (mt0 + m) * 16 + g + 8 * h;
        if (j == 0 && row < rows_pad && ((m == 0 && has0) || (m == 1 && has1))) {
          float* pp = a.part + ((size_t)blockIdx.x * rows_pad + row) * 2;
          pp[0] = rm[m][h];
          pp[1] = l;
        }
      }
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
