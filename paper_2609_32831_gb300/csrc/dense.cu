// Dense multi-query attention over heterogeneous segments (App. E "Attention
// over heterogeneous cache segments"; the denoising / editing calls where
// thousands of latent queries attend to the compressed cache and to
// themselves) on the 5th-generation tensor cores.
//
// 1. materialize_kernel rebuilds every (sequence, KV head) cache as fp16
//    rows, once per call: bf16 rows convert exactly; packed rows dequantize
//    in fp32 (x = code * s + z) and store as fp16 hi + lo parts for keys
//    (~22 bits, so the logits carry no fp16 rounding) and fp16 for values.
//    The pass reads each packed byte once and is amortised over every query
//    row of the KV head (7 heads x thousands of queries).
// 2. dense_kernel: one CTA per 256 query rows (two Q tiles of 128) of one
//    query head; keys in tiles of 128. Warpgroup roles:
//      WG0, WG1   softmax of Q tile 0 / 1: one query row per thread (= one
//                 TMEM lane); S read from TMEM, P = 2^(S - m) written back
//                 over S as fp16 pairs; online softmax with a lazily moved
//                 reference max (O is rescaled only when a row's max grows
//                 by more than 2^8, so P <= 256 stays exact enough in fp16);
//      WG2        warp 8: TMA producer of K hi / K lo tiles (3-slot ring) and
//                 V tiles (2-slot ring); warp 9: allocates TMEM and issues
//                 every tcgen05.mma from one thread, alternating the Q tiles:
//                 S_x = Q_x K^T (M=128, N=128, K=128, both from shared
//                 memory) and O_x += P_x V (A = P from TMEM, B = V from shared
//                 memory), so that one tile's softmax overlaps the other
//                 tile's MMAs. TMEM: S/P and O of both tiles, 512 columns.
//    The warpgroups rebalance registers with setmaxnreg (softmax 216, the
//    producer / MMA group 56).
#include <mutex>

#include "common.cuh"
#include "internal.h"
#include "tcgen05.cuh"

namespace uc {

// S_x = Q_x K^T over the 8 K steps of d = 128 (16 channels each): the A
// (Q) and B (K) offsets step 32 B inside a 128-B swizzled row, then 16 KB
// to the second 64-channel block.
template <int ACC0>
__device__ __forceinline__ void issue_qk(uint32_t d, uint32_t q_lo, uint32_t k_lo, uint32_t hi, uint32_t idesc) {
  umma_ss_off<0, 0, ACC0>(d, q_lo, k_lo, hi, idesc);
  umma_ss_off<2, 2, 1>(d, q_lo, k_lo, hi, idesc);
  umma_ss_off<4, 4, 1>(d, q_lo, k_lo, hi, idesc);
  umma_ss_off<6, 6, 1>(d, q_lo, k_lo, hi, idesc);
  umma_ss_off<1024, 1024, 1>(d, q_lo, k_lo, hi, idesc);
  umma_ss_off<1026, 1026, 1>(d, q_lo, k_lo, hi, idesc);
  umma_ss_off<1028, 1028, 1>(d, q_lo, k_lo, hi, idesc);
  umma_ss_off<1030, 1030, 1>(d, q_lo, k_lo, hi, idesc);
}


// Two fp32 lanes in one 64-bit register: packed FMA / add (sm_100 family).
__device__ __forceinline__ uint64_t f2_pack(float a, float b) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(a), "f"(b));
  return r;
}
__device__ __forceinline__ void f2_unpack(uint64_t r, float& a, float& b) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(a), "=f"(b) : "l"(r));
}
__device__ __forceinline__ uint64_t f2_fma(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ uint64_t f2_add(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

// Non-blocking test of an mbarrier phase (issued early; its result is used
// later, so the check overlaps the MMAs queued meanwhile).
__device__ __forceinline__ bool mbar_test(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n"
      ".reg .pred p;\n"
      "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      "selp.u32 %0, 1, 0, p;\n"
      "}\n"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

template <int N>
__device__ __forceinline__ void setmaxnreg_inc() {
  asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(N));
}
template <int N>
__device__ __forceinline__ void setmaxnreg_dec() {
  asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(N));
}

// Named barrier over the 256 softmax threads (warps 0-7).
__device__ __forceinline__ void softmax_bar() { asm volatile("bar.sync 1, 256;" ::: "memory"); }

// ------------------------------------------------------------ parameters
constexpr int kDQ = 128;           // query rows per Q tile (= TMEM lanes)
constexpr int kDQT = 2;            // Q tiles per CTA (ping-pong softmax warpgroups)
constexpr int kDK = kDenseKeys;    // keys per tile
constexpr int kDKSlots = 3;        // K ring (hi and lo tiles each take one slot)
constexpr int kDVSlots = 2;        // V ring
constexpr int kDThreads = 384;     // WG0, WG1: softmax of Q tile 0, 1; WG2: TMA warp, MMA warp, 2 idle
// Registers per thread after the warpgroups rebalance (launch: 168 each, 384
// threads = 64512; after: 256 x 216 + 128 x 56 = 62464 <= 64512).
constexpr int kRegSoftmax = 216;
constexpr int kRegOther = 56;
static_assert(2 * 128 * kRegSoftmax + 128 * kRegOther <= kDThreads * 168, "register split");
constexpr int kTmemCols = 512;     // per Q tile X: S/P [256X, 256X+128), O [256X+128, 256X+256)
constexpr float kDNegInf = -INFINITY;
// Issue S(j+1) of a Q tile only after P(j) V(j) of that tile has completed
// (P(j) lives in S's TMEM columns). false: rely on the in-order execution of
// the tensor pipe for that write-after-read.

struct DenseSmem {
  uint8_t q[kDQT][2][16384];       // Q fp16 [128 rows][2 x 64 cols], K-major, 128B swizzle
  uint8_t k[kDKSlots][2][16384];   // K hi or K lo [128 keys][2 x 64 cols]
  uint8_t v[kDVSlots][2][16384];   // V [128 keys][2 x 64 cols] (MN-major B operand)
  uint8_t valid[kMaxDenseTiles];   // keys of tile j present for this sequence
  uint8_t tseg[kMaxDenseTiles];    // segment of tile j
  uint8_t tlo[kMaxDenseTiles];     // 1 if tile j has K lo rows (packed segment)
  uint64_t k_full[kDKSlots], k_empty[kDKSlots], v_full[kDVSlots], v_empty[kDVSlots];
  uint64_t s_full[kDQT], p_full[kDQT], q_full[kDQT], o_full[kDQT];
  uint64_t pv_done[kDQT];  // serial order only: P V of the Q tile completed
  uint32_t tmem_base;
};
static_assert(sizeof(DenseSmem) + 1024 <= 232448, "dense kernel shared memory");

__device__ __forceinline__ bool dwait(uint64_t* bar, uint32_t parity, DevStatus* st, int where, bool& aborted) {
  if (aborted) return false;
  if (!mbar_wait(bar, parity, st, where)) aborted = true;
  return !aborted;
}

// The same for all 32 lanes of a warp: the outcome is made warp-uniform, so
// the warp-collective tcgen05.ld / st that follow never run divergently.
__device__ __forceinline__ bool dwait_warp(uint64_t* bar, uint32_t parity, DevStatus* st, int where,
                                           bool& aborted) {
  if (!aborted && !mbar_wait(bar, parity, st, where)) aborted = true;
  aborted = __any_sync(0xffffffffu, aborted);
  return !aborted;
}

// ------------------------------------------------------------ materialize
// Writes fp16 K hi / K lo / V rows of every tile of every (b, kvh). One warp
// per 32 rows of a tile of kDK rows (a quantization group of a packed
// segment); a tile never spans two segments. Rows past the sequence's kept
// count are written as zeros.
//
// A full quantization group of a packed segment (32 tokens) is decoded the
// way it is stored: each lane reads its own fragment-ordered code words and
// the parameter entries that belong to exactly its channels (keys) or tokens
// (values), rebuilds x = code * s + z in fp32, and writes fp16 into a
// 32-row staging block in shared memory (rows 272 bytes apart: conflict-free
// for both fragment patterns); the block then goes out as whole rows, 16
// bytes per lane. bf16 rows, the residual tail and the zero rows past the
// kept count are converted row by row.
constexpr int kMatWarps = 4;
constexpr int kMatRow = 136;  // halves per staged row (272 bytes)
struct MatStage {
  __half r[2][32][kMatRow];  // K hi, K lo; then V in r[0]
};

// 32 staged rows -> global rows dst[0 .. 31] (128 halves each), 16 B per lane
__device__ __forceinline__ void mat_store_rows(__half* dst, const __half (*src)[kMatRow]) {
  const int lane = threadIdx.x & 31;
#pragma unroll 4
  for (int k = lane; k < 32 * 16; k += 32) {
    const int row = k >> 4, c = k & 15;
    *reinterpret_cast<uint4*>(dst + (size_t)row * kHeadDim + 8 * c) =
        *reinterpret_cast<const uint4*>(&src[row][8 * c]);
  }
}

template <int BITS>
__device__ void mat_packed_group(const SegDev& sd, int bh, int g, __half* khi, __half* klo, __half* vv,
                                 MatStage& st) {
  const int lane = threadIdx.x & 31;
  constexpr uint32_t mask = (1u << BITS) - 1u;
  constexpr int kb = 8 / BITS;  // 16-channel (K) / 8-channel (V) blocks per code word
  const size_t blk_codes = (size_t)bh * sd.cap * kHeadDim * BITS / 8;
  // ---- keys: lane (n, j) holds tokens 8 nt + n, channels 16 i + 2 j + {0, 1, 8, 9}
  {
    const int n = lane >> 2, j = lane & 3;
    uint32_t w[4][BITS];
#pragma unroll
    for (int nt = 0; nt < 4; ++nt) {
      const uint8_t* src = sd.k_codes + blk_codes + ((size_t)(g * 4 + nt) * 32 + lane) * (BITS * 4);
      if constexpr (BITS == 4) {
        const uint4 x = *reinterpret_cast<const uint4*>(src);
        w[nt][0] = x.x; w[nt][BITS > 1 ? 1 : 0] = x.y; w[nt][BITS > 2 ? 2 : 0] = x.z; w[nt][BITS > 3 ? 3 : 0] = x.w;
      } else {
        const uint2 x = *reinterpret_cast<const uint2*>(src);
        w[nt][0] = x.x; w[nt][BITS > 1 ? 1 : 0] = x.y;
      }
    }
    const uint8_t* kp = sd.k_params + (size_t)bh * (sd.cap / kGroup) * 512 + (size_t)g * 512;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const uint4 e = *reinterpret_cast<const uint4*>(kp + (i * 4 + j) * 16);  // s01, s89, z01, z89
      const float2 s01 = __half22float2(*reinterpret_cast<const __half2*>(&e.x));
      const float2 s89 = __half22float2(*reinterpret_cast<const __half2*>(&e.y));
      const float2 z01 = __half22float2(*reinterpret_cast<const __half2*>(&e.z));
      const float2 z89 = __half22float2(*reinterpret_cast<const __half2*>(&e.w));
      const int q = i / kb, p = 2 * (i % kb);
      const int c = 16 * i + 2 * j;
#pragma unroll
      for (int nt = 0; nt < 4; ++nt) {
        const uint32_t word = w[nt][q];
        const float x0 = __fmaf_rn((float)((word >> (BITS * p)) & mask), s01.x, z01.x);
        const float x1 = __fmaf_rn((float)((word >> (16 + BITS * p)) & mask), s01.y, z01.y);
        const float x8 = __fmaf_rn((float)((word >> (BITS * (p + 1))) & mask), s89.x, z89.x);
        const float x9 = __fmaf_rn((float)((word >> (16 + BITS * (p + 1))) & mask), s89.y, z89.y);
        const __half2 h01 = __floats2half2_rn(x0, x1), h89 = __floats2half2_rn(x8, x9);
        const float2 f01 = __half22float2(h01), f89 = __half22float2(h89);
        const int row = 8 * nt + n;
        *reinterpret_cast<__half2*>(&st.r[0][row][c]) = h01;
        *reinterpret_cast<__half2*>(&st.r[0][row][c + 8]) = h89;
        *reinterpret_cast<__half2*>(&st.r[1][row][c]) = __floats2half2_rn(x0 - f01.x, x1 - f01.y);
        *reinterpret_cast<__half2*>(&st.r[1][row][c + 8]) = __floats2half2_rn(x8 - f89.x, x9 - f89.y);
      }
    }
    __syncwarp();
    mat_store_rows(khi, st.r[0]);
    mat_store_rows(klo, st.r[1]);
    __syncwarp();
  }
  // ---- values: lane (gq, j) holds, in 16-token tile kt, tokens 2 j + 8 sub
  // + {0, 1}, channels 8 m + gq
  {
    const int gq = lane >> 2, j = lane & 3;
    const uint8_t* vp = sd.v_params + (size_t)bh * sd.cap * 16;
#pragma unroll
    for (int kt = 0; kt < 2; ++kt) {
      uint32_t w[2 * BITS];
      const uint8_t* src = sd.v_codes + blk_codes + ((size_t)(g * 2 + kt) * 32 + lane) * (BITS * 8);
#pragma unroll
      for (int q = 0; q < 2 * BITS; q += 4) {
        const uint4 x = *reinterpret_cast<const uint4*>(src + 4 * q);
        w[q] = x.x; w[q + 1] = x.y; w[q + 2] = x.z; w[q + 3] = x.w;
      }
#pragma unroll
      for (int grp = 0; grp < 4; ++grp) {
        const uint4 e = *reinterpret_cast<const uint4*>(vp + (size_t)(g * 2 + kt) * 256 + (grp * 4 + j) * 16);
        const float2 s01 = __half22float2(*reinterpret_cast<const __half2*>(&e.x));  // tokens 2j, 2j + 1
        const float2 s89 = __half22float2(*reinterpret_cast<const __half2*>(&e.y));  // 2j + 8, 2j + 9
        const float2 z01 = __half22float2(*reinterpret_cast<const __half2*>(&e.z));
        const float2 z89 = __half22float2(*reinterpret_cast<const __half2*>(&e.w));
#pragma unroll
        for (int mm = 0; mm < 4; ++mm) {
          const int m = 4 * grp + mm;
          const uint32_t word = w[m / kb];
          const int p = 2 * (m % kb);
          const int ch = 8 * m + gq, t0 = 16 * kt + 2 * j;
          st.r[0][t0][ch] = __float2half_rn(__fmaf_rn((float)((word >> (BITS * p)) & mask), s01.x, z01.x));
          st.r[0][t0 + 1][ch] = __float2half_rn(__fmaf_rn((float)((word >> (16 + BITS * p)) & mask), s01.y, z01.y));
          st.r[0][t0 + 8][ch] =
              __float2half_rn(__fmaf_rn((float)((word >> (BITS * (p + 1))) & mask), s89.x, z89.x));
          st.r[0][t0 + 9][ch] =
              __float2half_rn(__fmaf_rn((float)((word >> (16 + BITS * (p + 1))) & mask), s89.y, z89.y));
        }
      }
    }
    __syncwarp();
    mat_store_rows(vv, st.r[0]);
    __syncwarp();
  }
}

__global__ void __launch_bounds__(32 * kMatWarps) materialize_kernel(const __grid_constant__ DenseParams p) {
  extern __shared__ __align__(16) uint8_t mat_smem[];
  MatStage& stg = reinterpret_cast<MatStage*>(mat_smem)[threadIdx.x >> 5];
  // one warp per (b, kvh, tile, 32-row quarter of the tile)
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  const int nbh = p.batch * p.n_kv_heads;
  constexpr int kQuarters = kDK / kGroup;
  if (warp >= nbh * p.n_tiles * kQuarters) return;
  const int qr = warp % kQuarters;
  const int bh = warp / (p.n_tiles * kQuarters), ti = (warp / kQuarters) % p.n_tiles;
  const int b = bh / p.n_kv_heads;
  const DenseTile tl = p.tiles[ti];
  const SegDev& sd = p.seg[tl.seg];
  const int n = sd.n_kept[b];
  const int r_lo = qr * kGroup;            // first row of this quarter inside the tile
  const int t0 = tl.seg_tile * kDK;
  __half* khi = p.khi + ((size_t)bh * p.rows_per_bh + tl.row) * kHeadDim;
  __half* vv = p.v + ((size_t)bh * p.rows_per_bh + tl.row) * kHeadDim;
  __half* klo = tl.lo_row >= 0 ? p.klo + ((size_t)bh * p.lo_rows_per_bh + tl.lo_row) * kHeadDim : nullptr;
  const bool bf16_kind = sd.kind == UC_KIND_FULL || sd.kind == UC_KIND_EVICT;
  const int ng = bf16_kind ? 0 : n / kGroup;
  // a full packed group (quantized segments always have a K lo block)
  if (!bf16_kind && klo != nullptr && (t0 + r_lo) / kGroup < ng) {
    const int g = (t0 + r_lo) / kGroup;
    if (sd.bits == 4)
      mat_packed_group<4>(sd, bh, g, khi + (size_t)r_lo * kHeadDim, klo + (size_t)r_lo * kHeadDim,
                          vv + (size_t)r_lo * kHeadDim, stg);
    else
      mat_packed_group<2>(sd, bh, g, khi + (size_t)r_lo * kHeadDim, klo + (size_t)r_lo * kHeadDim,
                          vv + (size_t)r_lo * kHeadDim, stg);
    return;
  }
  const int r_first = r_lo, r_end = r_lo + kGroup;
  // the rest row by row, eight rows' loads in flight at once: bf16 rows, the
  // residual tail, zeros past the kept count. Lane: channels 4 lane .. 4 lane + 3.
  for (int rb = r_first; rb < r_end; rb += 8) {
    uint2 ka[8], va[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const int t = t0 + rb + u;
      ka[u] = make_uint2(0u, 0u);
      va[u] = make_uint2(0u, 0u);
      if (t < n) {
        int64_t row;
        if (bf16_kind)
          row = (int64_t)bh * sd.row_stride + sd.row_offset + t;
        else
          row = (int64_t)bh * kGroup + (t - ng * kGroup);  // the residual tail (t >= ng * 32 here)
        ka[u] = *reinterpret_cast<const uint2*>(p.seg_k[tl.seg] + row * kHeadDim + 4 * lane);
        va[u] = *reinterpret_cast<const uint2*>(p.seg_v[tl.seg] + row * kHeadDim + 4 * lane);
      }
    }
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const int r = rb + u;
      const float kx[4] = {bf16_lo(ka[u].x), bf16_hi(ka[u].x), bf16_lo(ka[u].y), bf16_hi(ka[u].y)};
      const float vx[4] = {bf16_lo(va[u].x), bf16_hi(va[u].x), bf16_lo(va[u].y), bf16_hi(va[u].y)};
      __half hk[4], hv[4], lk[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        hk[e] = __float2half_rn(kx[e]);
        lk[e] = __float2half_rn(kx[e] - __half2float(hk[e]));
        hv[e] = __float2half_rn(vx[e]);
      }
      *reinterpret_cast<uint2*>(khi + r * kHeadDim + 4 * lane) =
          make_uint2(pack_h2(hk[0], hk[1]), pack_h2(hk[2], hk[3]));
      *reinterpret_cast<uint2*>(vv + r * kHeadDim + 4 * lane) =
          make_uint2(pack_h2(hv[0], hv[1]), pack_h2(hv[2], hv[3]));
      if (klo != nullptr)
        *reinterpret_cast<uint2*>(klo + r * kHeadDim + 4 * lane) =
            make_uint2(pack_h2(lk[0], lk[1]), pack_h2(lk[2], lk[3]));
    }
  }
}

// ---------------------------------------------------------------- dense
// MAXSEG: segments whose softmax mass is accumulated in registers (>= nseg).
template <int MAXSEG>
__global__ void __launch_bounds__(kDThreads, 1) dense_kernel(const __grid_constant__ DenseParams p) {
  extern __shared__ uint8_t dyn_smem[];
  DenseSmem& sm = *reinterpret_cast<DenseSmem*>(
      (reinterpret_cast<uintptr_t>(dyn_smem) + 1023) & ~static_cast<uintptr_t>(1023));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n_qp = (p.n_qtok + kDQ * kDQT - 1) / (kDQ * kDQT);
  const int qp = blockIdx.x % n_qp;
  const int bhq = blockIdx.x / n_qp;  // b * Hq + h
  const int b = bhq / p.n_q_heads, h = bhq % p.n_q_heads;
  const int kvh = h / p.group;
  const int bh = b * p.n_kv_heads + kvh;
  const int T = p.n_tiles;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kDKSlots; ++s) {
      mbar_init(&sm.k_full[s], 1);
      mbar_init(&sm.k_empty[s], 1);
    }
    for (int s = 0; s < kDVSlots; ++s) {
      mbar_init(&sm.v_full[s], 1);
      mbar_init(&sm.v_empty[s], 1);
    }
    for (int x = 0; x < kDQT; ++x) {
      mbar_init(&sm.s_full[x], 1);
      mbar_init(&sm.p_full[x], kDQ);
      mbar_init(&sm.q_full[x], kDQ);
      mbar_init(&sm.pv_done[x], 1);
      mbar_init(&sm.o_full[x], 1);
    }
    fence_barrier_init();
  }
  if (warp == 9) tmem_alloc(&sm.tmem_base, kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sm.tmem_base;
  bool aborted = false;

  // Each warpgroup rebalances its registers (one setmaxnreg per warpgroup)
  // inside its own branch, so that the compiler budgets every role's code
  // for its own register count.
  if (warp >= 8) {
    setmaxnreg_dec<kRegOther>();
    if (warp == 8 && lane == 0) {
      // ------------------------------------------------------ TMA producer
      prefetch_tmap(&p.tmap_khi);
      prefetch_tmap(&p.tmap_klo);
      prefetch_tmap(&p.tmap_v);
      int kc = 0;
      for (int j = 0; j < T && !aborted; ++j) {
        const DenseTile tl = p.tiles[j];
        const int row = (int)((int64_t)bh * p.rows_per_bh + tl.row);
        for (int part = 0; part < (tl.lo_row >= 0 ? 2 : 1); ++part, ++kc) {
          const int s = kc % kDKSlots;
          if (kc >= kDKSlots && !dwait(&sm.k_empty[s], ((kc / kDKSlots) - 1) & 1, p.status, 30, aborted)) break;
          mbar_arrive_expect_tx(&sm.k_full[s], 32768u);
          const CUtensorMap* m = part == 0 ? &p.tmap_khi : &p.tmap_klo;
          const int rr = part == 0 ? row : (int)((int64_t)bh * p.lo_rows_per_bh + tl.lo_row);
          tma_load_2d(sm.k[s][0], m, 0, rr, &sm.k_full[s]);
          tma_load_2d(sm.k[s][1], m, 64, rr, &sm.k_full[s]);
        }
        const int s = j % kDVSlots;
        if (j >= kDVSlots && !dwait(&sm.v_empty[s], ((j / kDVSlots) - 1) & 1, p.status, 31, aborted)) break;
        mbar_arrive_expect_tx(&sm.v_full[s], 32768u);
        tma_load_2d(sm.v[s][0], &p.tmap_v, 0, row, &sm.v_full[s]);
        tma_load_2d(sm.v[s][1], &p.tmap_v, 64, row, &sm.v_full[s]);
      }
    }
    if (warp == 9 && lane == 0) {
      // ----------------------------------------------------- MMA issuer
      // One thread issues every MMA, alternating the Q tiles so that one
      // tile's softmax overlaps the other tile's MMAs:
      //   S_0(0), S_1(0); for each key tile j:
      //     O_0 += P_0(j) V(j), S_0(j+1);  O_1 += P_1(j) V(j), S_1(j+1).
      // This thread shares its SM sub-partition with busy softmax warps, so
      // it keeps its instructions per MMA to a minimum: descriptor low
      // words plus constants, slot counters without divisions, and barrier
      // checks issued as non-blocking tests between MMAs.
      constexpr uint32_t id_s = idesc_f16(kDQ, kDK, 0, 0);
      constexpr uint32_t id_o = idesc_f16(kDQ, kHeadDim, 0, 1);
      const uint32_t dhi = (uint32_t)(smem_desc_sw128(0, 16) >> 32);  // SBO, version, swizzle
      const uint32_t q_lo0 = (uint32_t)smem_desc_sw128(smem_u32(sm.q[0][0]), 16);
      const uint32_t q_lo1 = (uint32_t)smem_desc_sw128(smem_u32(sm.q[1][0]), 16);
      const uint32_t k_lo0 = (uint32_t)smem_desc_sw128(smem_u32(sm.k[0][0]), 16);
      const uint32_t v_lo0 = (uint32_t)smem_desc_sw128(smem_u32(sm.v[0][0]), 16384);
      constexpr uint32_t kSlotStep = sizeof(sm.k[0]) >> 4;   // descriptor units per K slot
      constexpr uint32_t kVSlotStep = sizeof(sm.v[0]) >> 4;  // per V slot
      // K ring position: slot and phase of the next K part to consume
      int ks = 0;
      uint32_t kph = 0;
      auto k_next = [&]() {
        if (++ks == kDKSlots) {
          ks = 0;
          kph ^= 1u;
        }
      };
      int hs = 0, ls = -1;  // slots of the tile whose S is issued next
      // issues S_x = Q_x K^T (+ Q_x K_lo^T) of the current (hs, ls)
      auto issue_s = [&](uint32_t q_lo, uint32_t d) {
        issue_qk<0>(d, q_lo, k_lo0 + (uint32_t)hs * kSlotStep, dhi, id_s);
        if (ls >= 0) issue_qk<1>(d, q_lo, k_lo0 + (uint32_t)ls * kSlotStep, dhi, id_s);
      };
      // O_x += P_x V(j), K steps 0-3 or 4-7: A = P in TMEM (columns of S_x)
      auto issue_pv_lo = [&](uint32_t d_s, uint32_t vb, uint32_t acc0) {
        umma_ts_off<0>(d_s + 128, d_s, vb, dhi, id_o, acc0);
        umma_ts_off<1>(d_s + 128, d_s, vb, dhi, id_o, 1u);
        umma_ts_off<2>(d_s + 128, d_s, vb, dhi, id_o, 1u);
        umma_ts_off<3>(d_s + 128, d_s, vb, dhi, id_o, 1u);
      };
      auto issue_pv_hi = [&](uint32_t d_s, uint32_t vb) {
        umma_ts_off<4>(d_s + 128, d_s, vb, dhi, id_o, 1u);
        umma_ts_off<5>(d_s + 128, d_s, vb, dhi, id_o, 1u);
        umma_ts_off<6>(d_s + 128, d_s, vb, dhi, id_o, 1u);
        umma_ts_off<7>(d_s + 128, d_s, vb, dhi, id_o, 1u);
      };
      // takes the K parts of tile j (waits unless a test already saw them)
      auto k_take = [&](bool lo, bool known_ready) -> bool {
        hs = ks;
        if (!known_ready && !dwait(&sm.k_full[ks], kph, p.status, 32, aborted)) return false;
        k_next();
        ls = -1;
        if (lo) {
          ls = ks;
          if (!known_ready && !dwait(&sm.k_full[ks], kph, p.status, 33, aborted)) return false;
          k_next();
        }
        return true;
      };
      auto k_test = [&](bool lo) -> bool {
        bool ok = mbar_test(&sm.k_full[ks], kph);
        if (lo) {
          const int s2 = ks + 1 == kDKSlots ? 0 : ks + 1;
          ok = mbar_test(&sm.k_full[s2], s2 == 0 ? kph ^ 1u : kph) && ok;
        }
        return ok;
      };
      const uint32_t d_s0 = tmem, d_s1 = tmem + 256;
      bool ok = dwait(&sm.q_full[0], 0, p.status, 34, aborted) && dwait(&sm.q_full[1], 0, p.status, 34, aborted);
      if (ok && T > 0 && k_take(sm.tlo[0] != 0, false)) {
        tc_fence_after();
        issue_s(q_lo0, d_s0);
        umma_commit(&sm.s_full[0]);
        issue_s(q_lo1, d_s1);
        umma_commit(&sm.s_full[1]);
        umma_commit(&sm.k_empty[hs]);
        if (ls >= 0) umma_commit(&sm.k_empty[ls]);
        bool v_ok = false;
        bool lo_next = T > 1 && sm.tlo[1] != 0;
        int vs = 0;
        uint32_t vph = 0;
        for (int j = 0; j < T; ++j) {
          const bool more = j + 1 < T;
          const uint32_t vb = v_lo0 + (uint32_t)vs * kVSlotStep;
          // ---- Q tile 0: O_0 += P_0(j) V(j), then S_0(j+1)
          if (!dwait(&sm.p_full[0], j & 1, p.status, 35, aborted)) break;
          if (!v_ok && !dwait(&sm.v_full[vs], vph, p.status, 36, aborted)) break;
          tc_fence_after();
          issue_pv_lo(d_s0, vb, j > 0);
          const bool k_ok = more && k_test(lo_next);
          issue_pv_hi(d_s0, vb);
          bool pb_ok = false;
          if (more) {
            if (p.serial_pv) {
              umma_commit(&sm.pv_done[0]);
              if (!dwait(&sm.pv_done[0], j & 1, p.status, 37, aborted)) break;
            }
            if (!k_take(lo_next, k_ok)) break;
            tc_fence_after();
            pb_ok = mbar_test(&sm.p_full[1], j & 1);
            issue_s(q_lo0, d_s0);
            umma_commit(&sm.s_full[0]);
          }
          // ---- Q tile 1: O_1 += P_1(j) V(j), then S_1(j+1)
          if (!pb_ok && !dwait(&sm.p_full[1], j & 1, p.status, 38, aborted)) break;
          tc_fence_after();
          issue_pv_lo(d_s1, vb, j > 0);
          const int vs_n = vs + 1 == kDVSlots ? 0 : vs + 1;
          const uint32_t vph_n = vs_n == 0 ? vph ^ 1u : vph;
          v_ok = more && mbar_test(&sm.v_full[vs_n], vph_n);
          issue_pv_hi(d_s1, vb);
          umma_commit(&sm.v_empty[vs]);
          vs = vs_n;
          vph = vph_n;
          if (more) {
            if (p.serial_pv) {
              umma_commit(&sm.pv_done[1]);
              if (!dwait(&sm.pv_done[1], j & 1, p.status, 39, aborted)) break;
              tc_fence_after();
            }
            issue_s(q_lo1, d_s1);
            umma_commit(&sm.s_full[1]);
            umma_commit(&sm.k_empty[hs]);
            if (ls >= 0) umma_commit(&sm.k_empty[ls]);
            lo_next = j + 2 < T && sm.tlo[j + 2] != 0;
          }
        }
        umma_commit(&sm.o_full[0]);
        umma_commit(&sm.o_full[1]);
      }
    }
  } else {
    setmaxnreg_inc<kRegSoftmax>();
    // ------------------------------------------------------------ softmax
    const int x = warp >> 2;          // Q tile of this warpgroup
    const int r = threadIdx.x & 127;  // query row within the tile = TMEM lane
    const int qi = (qp * kDQT + x) * kDQ + r;
    const bool row_ok = qi < p.n_qtok;
    {
      // Q row: bf16 -> fp16, swizzled K-major
      const __nv_bfloat16* qs = p.q + ((size_t)bhq * p.n_qtok + (row_ok ? qi : 0)) * kHeadDim;
#pragma unroll
      for (int c = 0; c < 16; ++c) {
        uint4 w = make_uint4(0, 0, 0, 0);
        if (row_ok) w = *reinterpret_cast<const uint4*>(qs + 8 * c);
        const uint4 o = make_uint4(pack_f16(bf16_lo(w.x), bf16_hi(w.x)), pack_f16(bf16_lo(w.y), bf16_hi(w.y)),
                                   pack_f16(bf16_lo(w.z), bf16_hi(w.z)), pack_f16(bf16_lo(w.w), bf16_hi(w.w)));
        *reinterpret_cast<uint4*>(sm.q[x][c >> 3] + r * 128 + (((c & 7) ^ (r & 7)) << 4)) = o;
      }
      // per-tile tables for this sequence (read by the MMA thread after q_full)
      for (int jj = threadIdx.x; jj < T; jj += kDQ * kDQT) {
        const DenseTile tl = p.tiles[jj];
        const int n = p.seg[tl.seg].n_kept[b];
        sm.valid[jj] = (uint8_t)min(kDK, max(0, n - tl.seg_tile * kDK));
        sm.tseg[jj] = (uint8_t)tl.seg;
        sm.tlo[jj] = (uint8_t)(tl.lo_row >= 0);
      }
      fence_proxy_async_smem();
      mbar_arrive(&sm.q_full[x]);
      softmax_bar();
    }
    const uint32_t lane_off = (uint32_t)(32 * (warp & 3)) << 16;
    const uint32_t s_col = x * 256, o_col = x * 256 + 128;
    const float sl2 = p.scale_log2;
    float m_ref = kDNegInf, l = 0.f;
    float ls[MAXSEG];
#pragma unroll
    for (int s = 0; s < MAXSEG; ++s) ls[s] = 0.f;
    const uint64_t sl2_2 = f2_pack(sl2, sl2);
    for (int j = 0; j < T; ++j) {
      if (!dwait_warp(&sm.s_full[x], j & 1, p.status, 40, aborted)) break;
      tc_fence_after();
      const int vld = sm.valid[j];
      uint32_t pk[2][32];
      float sum[4];
      // One pass: P = 2^(S sl2 - m_ref) with the current reference max while
      // the tile max is taken alongside (no max -> exp dependency). Redone,
      // from S reloaded out of TMEM (P is not stored yet), for the first
      // tile and whenever a row's max grows by more than 8 (P <= 2^8).
      bool redo = !__all_sync(0xffffffffu, m_ref != kDNegInf);
      if (!redo) {
        uint32_t sr[4][32];
#pragma unroll
        for (int c = 0; c < 4; ++c) tmem_ld32(tmem + lane_off + s_col + 32 * c, sr[c]);
        tmem_wait_ld();
        if (vld < kDK) {
#pragma unroll
          for (int c = 0; c < kDK; ++c)
            if (c >= vld) sr[c >> 5][c & 31] = __float_as_uint(kDNegInf);
        }
        const uint64_t nm2 = f2_pack(-m_ref, -m_ref);
        float mx[4] = {kDNegInf, kDNegInf, kDNegInf, kDNegInf};
        uint64_t acc[2] = {0ull, 0ull};
#pragma unroll
        for (int c2 = 0; c2 < kDK / 2; ++c2) {
          const float s0 = __uint_as_float(sr[(2 * c2) >> 5][(2 * c2) & 31]);
          const float s1 = __uint_as_float(sr[(2 * c2 + 1) >> 5][(2 * c2 + 1) & 31]);
          mx[c2 & 3] = fmax3(mx[c2 & 3], s0, s1);
          float e0, e1;
          f2_unpack(f2_fma(f2_pack(s0, s1), sl2_2, nm2), e0, e1);
          const float a = ex2_approx(e0), bb = ex2_approx(e1);
          acc[c2 & 1] = f2_add(acc[c2 & 1], f2_pack(a, bb));
          pk[c2 >> 5][c2 & 31] = pack_f16(a, bb);
        }
        const float tmax = fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])) * sl2;
        f2_unpack(acc[0], sum[0], sum[1]);
        f2_unpack(acc[1], sum[2], sum[3]);
        redo = __any_sync(0xffffffffu, tmax > m_ref + 8.f);
      }
      if (redo) {
        uint32_t sr[4][32];
#pragma unroll
        for (int c = 0; c < 4; ++c) tmem_ld32(tmem + lane_off + s_col + 32 * c, sr[c]);
        tmem_wait_ld();
        if (vld < kDK) {
#pragma unroll
          for (int c = 0; c < kDK; ++c)
            if (c >= vld) sr[c >> 5][c & 31] = __float_as_uint(kDNegInf);
        }
        float mx[4] = {kDNegInf, kDNegInf, kDNegInf, kDNegInf};
#pragma unroll
        for (int c2 = 0; c2 < kDK / 2; ++c2)
          mx[c2 & 3] = fmax3(mx[c2 & 3], __uint_as_float(sr[(2 * c2) >> 5][(2 * c2) & 31]),
                             __uint_as_float(sr[(2 * c2 + 1) >> 5][(2 * c2 + 1) & 31]));
        const float tmax = fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])) * sl2;
        // lazy rescale: the reference max moves only when the tile's max
        // exceeds it by more than 8; O in TMEM, final since the previous
        // P V completed before S of this tile, is rescaled warp-wide
        const bool grow = tmax > m_ref + 8.f;
        const float m_new = grow ? tmax : m_ref;
        const bool need_o = grow && m_ref != kDNegInf;
        const float mb = (m_new == kDNegInf) ? 0.f : m_new;
        const uint64_t nm2 = f2_pack(-mb, -mb);
        uint64_t acc[2] = {0ull, 0ull};
#pragma unroll
        for (int c2 = 0; c2 < kDK / 2; ++c2) {
          float e0, e1;
          f2_unpack(f2_fma(f2_pack(__uint_as_float(sr[(2 * c2) >> 5][(2 * c2) & 31]),
                                   __uint_as_float(sr[(2 * c2 + 1) >> 5][(2 * c2 + 1) & 31])),
                           sl2_2, nm2),
                    e0, e1);
          const float a = ex2_approx(e0), bb = ex2_approx(e1);
          acc[c2 & 1] = f2_add(acc[c2 & 1], f2_pack(a, bb));
          pk[c2 >> 5][c2 & 31] = pack_f16(a, bb);
        }
        f2_unpack(acc[0], sum[0], sum[1]);
        f2_unpack(acc[1], sum[2], sum[3]);
        if (__any_sync(0xffffffffu, need_o)) {
          const float alpha = need_o ? ex2_approx(m_ref - m_new) : 1.f;
#pragma unroll 1
          for (int cb = 0; cb < 4; ++cb) {
            uint32_t o[32];
            tmem_ld32(tmem + lane_off + o_col + cb * 32, o);
            tmem_wait_ld();
#pragma unroll
            for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * alpha);
            tmem_st32(tmem + lane_off + o_col + cb * 32, o);
          }
          l *= alpha;
#pragma unroll
          for (int s = 0; s < MAXSEG; ++s) ls[s] *= alpha;
        }
        m_ref = m_new;
      }
      tmem_st32(tmem + lane_off + s_col, pk[0]);
      tmem_st32(tmem + lane_off + s_col + 32, pk[1]);
      tmem_wait_st();
      tc_fence_before();
      mbar_arrive(&sm.p_full[x]);
      const float ts = (sum[0] + sum[1]) + (sum[2] + sum[3]);
      l += ts;
      const int sg = sm.tseg[j];
#pragma unroll
      for (int s = 0; s < MAXSEG; ++s)
        if (s == sg) ls[s] += ts;
    }
    // ------------------------------------------------------------ epilogue
    if (T > 0 && dwait_warp(&sm.o_full[x], 0, p.status, 41, aborted)) {
      tc_fence_after();
      const float inv = (l > 0.f) ? 1.f / l : 0.f;
      __nv_bfloat16* orow = p.out + ((size_t)bhq * p.n_qtok + (row_ok ? qi : 0)) * kHeadDim;
#pragma unroll 1
      for (int cb = 0; cb < 4; ++cb) {
        uint32_t o[32];
        tmem_ld32(tmem + lane_off + o_col + cb * 32, o);
        tmem_wait_ld();
        if (row_ok) {
#pragma unroll
          for (int e = 0; e < 32; e += 8) {
            uint4 w;
            w.x = pack_bf16(__uint_as_float(o[e]) * inv, __uint_as_float(o[e + 1]) * inv);
            w.y = pack_bf16(__uint_as_float(o[e + 2]) * inv, __uint_as_float(o[e + 3]) * inv);
            w.z = pack_bf16(__uint_as_float(o[e + 4]) * inv, __uint_as_float(o[e + 5]) * inv);
            w.w = pack_bf16(__uint_as_float(o[e + 6]) * inv, __uint_as_float(o[e + 7]) * inv);
            *reinterpret_cast<uint4*>(orow + cb * 32 + e) = w;
          }
        }
      }
      if (row_ok) {
        const size_t orx = (size_t)bhq * p.n_qtok + qi;
        if (p.lse) p.lse[orx] = (l > 0.f) ? (m_ref + log2f(l)) * 0.69314718055994530942f : kDNegInf;
        if (p.mass) {
#pragma unroll
          for (int s = 0; s < MAXSEG; ++s)
            if (s < p.nseg) p.mass[orx * p.nseg + s] = ls[s] * inv;
        }
      }
    }
    tc_fence_before();
  }
  __syncthreads();
  if (warp == 9) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// ---------------------------------------------------------------- launchers
size_t dense_smem_bytes() { return sizeof(DenseSmem) + 1024; }

void launch_dense(const DenseParams& p, cudaStream_t st) {
  static std::once_flag once;
  std::call_once(once, [] {
    cudaFuncSetAttribute(dense_kernel<4>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dense_smem_bytes());
    cudaFuncSetAttribute(dense_kernel<UC_MAX_SEGMENTS>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         (int)dense_smem_bytes());
    cudaFuncSetAttribute(materialize_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         (int)(kMatWarps * sizeof(MatStage)));
  });
  const int nbh = p.batch * p.n_kv_heads;
  const int warps = nbh * p.n_tiles * (kDK / kGroup);
  materialize_kernel<<<(warps + kMatWarps - 1) / kMatWarps, 32 * kMatWarps, kMatWarps * sizeof(MatStage), st>>>(p);
  count_launch();
  const int n_qp = (p.n_qtok + kDQ * kDQT - 1) / (kDQ * kDQT);
  const int grid = p.batch * p.n_q_heads * n_qp;
  if (p.nseg <= 4)
    dense_kernel<4><<<grid, kDThreads, dense_smem_bytes(), st>>>(p);
  else
    dense_kernel<UC_MAX_SEGMENTS><<<grid, kDThreads, dense_smem_bytes(), st>>>(p);
  count_launch();
}

}  // namespace uc
