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
// 2. dense_kernel: one CTA per 128 query rows of one head. Warp roles:
//      warps 0-3  softmax: one query row per thread (= one TMEM lane); online
//                 softmax in registers, P written to shared memory in fp16;
//      warp 4     TMA producer of 64-key tiles (K hi, K lo, V) into a 2-stage
//                 ring;
//      warp 5     allocates TMEM and issues tcgen05.mma from one thread:
//                 S = Q K^T (M=128, N=64, K=128) into a double-buffered TMEM
//                 S, then O += P V (M=128, N=128, K=64) into TMEM.
//    The running max is rescaled lazily: O in TMEM is only rescaled when a
//    row's max grows by more than 2^8 (P stays <= 256, exact enough in fp16).
#include <mutex>

#include "common.cuh"
#include "internal.h"

namespace uc {

// ------------------------------------------------------------ tcgen05 PTX
__device__ __forceinline__ void tmem_alloc(uint32_t* dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(dst_smem)),
               "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}

__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// D (TMEM) = A (smem) * B (smem) [+ D], kind::f16, one thread.
__device__ __forceinline__ void umma_f16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                         uint32_t accumulate) {
  asm volatile(
      "{\n"
      ".reg .pred p;\n"
      "setp.ne.b32 p, %4, 0;\n"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n"
      "}\n" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrive once on an mbarrier when every tcgen05.mma issued so far by this
// thread has completed.
__device__ __forceinline__ void umma_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                   smem_u32(bar))
               : "memory");
}

// 32 consecutive 32-bit TMEM columns of this thread's lane.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
        "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]),
        "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]),
        "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
}

__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
      "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
      "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]),
      "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(r[16]),
      "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]),
      "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
      : "memory");
}

__device__ __forceinline__ void tmem_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }
__device__ __forceinline__ void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

// Shared-memory matrix descriptor, 128-byte swizzle. K-major operands: rows
// of 128 B (64 fp16 along K), 8-row groups 1024 B apart (SBO). MN-major
// operands: 64 fp16 along MN per 128-B row, K rows 128 B apart, 8-row groups
// 1024 B apart (SBO), the next 64 MN elements `lbo` bytes further (LBO).
__device__ __forceinline__ uint64_t smem_desc_sw128(uint32_t saddr, uint32_t lbo_bytes) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)((lbo_bytes >> 4) & 0x3FFFu) << 16;
  d |= (uint64_t)(1024u >> 4) << 32;
  d |= (uint64_t)1 << 46;  // descriptor version
  d |= (uint64_t)2 << 61;  // 128-byte swizzle
  return d;
}

// Instruction descriptor, kind::f16: fp16 A and B, fp32 D, M x N, majors.
__host__ __device__ constexpr uint32_t idesc_f16(int m, int n, int a_mn_major, int b_mn_major) {
  return (1u << 4)                          // D = F32
         | (0u << 7) | (0u << 10)           // A, B = F16
         | ((uint32_t)a_mn_major << 15) | ((uint32_t)b_mn_major << 16) |
         ((uint32_t)(n >> 3) << 17) | ((uint32_t)(m >> 4) << 24);
}

// ------------------------------------------------------------ parameters
constexpr int kDQ = 128;       // query rows per CTA
constexpr int kDK = 64;        // keys per tile
constexpr int kDStages = 2;
constexpr int kDThreads = 192;
constexpr int kTmemCols = 256;  // S0 [0,64), S1 [64,128), O [128,256)
constexpr float kDNegInf = -INFINITY;

struct DenseSmem {
  uint8_t q[2][16384];                // Q fp16 [128 rows][2 x 64 cols], K-major, swizzled
  uint8_t khi[kDStages][2][8192];     // K hi [64 keys][2 x 64 cols]
  uint8_t klo[kDStages][2][8192];     // K lo
  uint8_t v[kDStages][2][8192];       // V [64 keys][2 x 64 cols] (MN-major B operand)
  uint8_t p[2][16384];                // P fp16 [128 rows][64 keys], K-major, swizzled
  uint64_t kv_full[kDStages], kv_empty[kDStages];
  uint64_t s_full[2], s_free[2], p_full[2], p_free[2], q_full;  // p_free[j & 1]: P V of tile j done
  uint32_t tmem_base;
};

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
// per (bh, tile of 64 rows); a tile never spans two segments.
__global__ void __launch_bounds__(256) materialize_kernel(const __grid_constant__ DenseParams p) {
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  const int nbh = p.batch * p.n_kv_heads;
  if (warp >= nbh * p.n_tiles) return;
  const int bh = warp / p.n_tiles, ti = warp % p.n_tiles;
  const int b = bh / p.n_kv_heads;
  const DenseTile tl = p.tiles[ti];
  const SegDev& sd = p.seg[tl.seg];
  const int n = sd.n_kept[b];
  const int t0 = tl.seg_tile * kDK;
  __half* khi = p.khi + ((size_t)bh * p.rows_per_bh + tl.row) * kHeadDim;
  __half* vv = p.v + ((size_t)bh * p.rows_per_bh + tl.row) * kHeadDim;
  __half* klo = tl.lo_row >= 0 ? p.klo + ((size_t)bh * p.lo_rows_per_bh + tl.lo_row) * kHeadDim : nullptr;
  const bool bf16_kind = sd.kind == UC_KIND_FULL || sd.kind == UC_KIND_EVICT;
  const int ng = bf16_kind ? 0 : n / kGroup;
  // lane handles channels 4*lane .. 4*lane+3 of each row
  for (int r = 0; r < kDK; ++r) {
    const int t = t0 + r;
    float kx[4] = {0.f, 0.f, 0.f, 0.f}, vx[4] = {0.f, 0.f, 0.f, 0.f};
    if (t < n) {
      const __nv_bfloat16* ks = nullptr;
      const __nv_bfloat16* vs = nullptr;
      if (bf16_kind) {
        const int64_t row = (int64_t)bh * sd.row_stride + sd.row_offset + t;
        ks = p.seg_k[tl.seg] + row * kHeadDim;
        vs = p.seg_v[tl.seg] + row * kHeadDim;
      } else if (t >= ng * kGroup) {
        const int64_t row = (int64_t)bh * kGroup + (t - ng * kGroup);
        ks = p.seg_k[tl.seg] + row * kHeadDim;
        vs = p.seg_v[tl.seg] + row * kHeadDim;
      }
      if (ks != nullptr) {
        const uint2 a = *reinterpret_cast<const uint2*>(ks + 4 * lane);
        const uint2 c = *reinterpret_cast<const uint2*>(vs + 4 * lane);
        kx[0] = bf16_lo(a.x); kx[1] = bf16_hi(a.x); kx[2] = bf16_lo(a.y); kx[3] = bf16_hi(a.y);
        vx[0] = bf16_lo(c.x); vx[1] = bf16_hi(c.x); vx[2] = bf16_lo(c.y); vx[3] = bf16_hi(c.y);
      } else {
        // packed token: K per channel (group t / 32), V per token
        const int bits = sd.bits, g = t / kGroup, tg = t % kGroup;
        const size_t blk_codes = (size_t)bh * sd.cap * kHeadDim * bits / 8;
        const uint8_t* kc = sd.k_codes + blk_codes;
        const uint8_t* vc = sd.v_codes + blk_codes;
        const uint8_t* kp = sd.k_params + (size_t)bh * (sd.cap / kGroup) * 512 + (size_t)g * 512;
        const uint8_t* vp = sd.v_params + (size_t)bh * sd.cap * 16;
        const int mask = (1 << bits) - 1;
        for (int e = 0; e < 4; ++e) {
          const int c = 4 * lane + e;
          // K code of (token tg of group g, channel c) in the fragment layout
          const int nt = tg >> 3, nn = tg & 7, i = c >> 4, cc = c & 15;
          const int j = (cc & 7) >> 1, sub = cc >> 3, ee = cc & 1;
          const int kl = nn * 4 + j;
          const int pr = (bits == 4) ? (2 * (i & 1) + sub) : (2 * (i & 3) + sub);
          const int wq = (bits == 4) ? (i >> 1) : (i >> 2);
          const uint32_t w = *reinterpret_cast<const uint32_t*>(kc + ((size_t)(g * 4 + nt) * 32 + kl) * (bits * 4) + 4 * wq);
          const int code = (w >> (bits * pr + 16 * ee)) & mask;
          const __half* kpar = reinterpret_cast<const __half*>(kp + (i * 4 + j) * 16);
          const float s = __half2float(kpar[sub * 2 + ee]), z = __half2float(kpar[4 + sub * 2 + ee]);
          kx[e] = __fmaf_rn((float)code, s, z);
          // V code of (token t, channel c): 16-token tile, lane (c % 8, token pair)
          const int t16 = t >> 4, tt = t & 15, m = c >> 3, gq = c & 7;
          const int vsub = tt >> 3, vj = (tt & 7) >> 1, ve = tt & 1;
          const int vl = gq * 4 + vj;
          const int vpr = (bits == 4) ? (2 * (m & 1) + vsub) : (2 * (m & 3) + vsub);
          const int vwq = (bits == 4) ? (m >> 1) : (m >> 2);
          const uint32_t vw = *reinterpret_cast<const uint32_t*>(vc + ((size_t)t16 * 32 + vl) * (bits * 8) + 4 * vwq);
          const int vcode = (vw >> (bits * vpr + 16 * ve)) & mask;
          const int grp = c >> 5;
          const __half* vpar = reinterpret_cast<const __half*>(vp + (size_t)t16 * 256 + (grp * 4 + vj) * 16);
          const float vs_ = __half2float(vpar[vsub * 2 + ve]), vz = __half2float(vpar[4 + vsub * 2 + ve]);
          vx[e] = __fmaf_rn((float)vcode, vs_, vz);
        }
      }
    }
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

// ---------------------------------------------------------------- dense
__global__ void __launch_bounds__(kDThreads, 1) dense_kernel(const __grid_constant__ DenseParams p) {
  extern __shared__ uint8_t dyn_smem[];
  DenseSmem& sm = *reinterpret_cast<DenseSmem*>(
      (reinterpret_cast<uintptr_t>(dyn_smem) + 1023) & ~static_cast<uintptr_t>(1023));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n_qt = (p.n_qtok + kDQ - 1) / kDQ;
  const int qt = blockIdx.x % n_qt;
  const int bhq = blockIdx.x / n_qt;  // b * Hq + h
  const int b = bhq / p.n_q_heads, h = bhq % p.n_q_heads;
  const int kvh = h / p.group;
  const int bh = b * p.n_kv_heads + kvh;
  const int T = p.n_tiles;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kDStages; ++s) {
      mbar_init(&sm.kv_full[s], 1);
      mbar_init(&sm.kv_empty[s], 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(&sm.s_full[s], 1);
      mbar_init(&sm.s_free[s], 128);
      mbar_init(&sm.p_full[s], 128);
      mbar_init(&sm.p_free[s], 1);
    }
    mbar_init(&sm.q_full, 128);
    fence_barrier_init();
  }
  if (warp == 5) tmem_alloc(&sm.tmem_base, kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sm.tmem_base;
  bool aborted = false;

  if (warp == 4) {
    // -------------------------------------------------------- TMA producer
    if (lane == 0) {
      prefetch_tmap(&p.tmap_khi);
      prefetch_tmap(&p.tmap_klo);
      prefetch_tmap(&p.tmap_v);
      for (int j = 0; j < T; ++j) {
        const int st = j % kDStages;
        if (j >= kDStages && !dwait(&sm.kv_empty[st], ((j / kDStages) - 1) & 1, p.status, 30, aborted)) break;
        const DenseTile tl = p.tiles[j];
        const int row = (int)((int64_t)bh * p.rows_per_bh + tl.row);
        const uint32_t bytes = (tl.lo_row >= 0 ? 3u : 2u) * 16384u;
        mbar_arrive_expect_tx(&sm.kv_full[st], bytes);
        tma_load_2d(sm.khi[st][0], &p.tmap_khi, 0, row, &sm.kv_full[st]);
        tma_load_2d(sm.khi[st][1], &p.tmap_khi, 64, row, &sm.kv_full[st]);
        tma_load_2d(sm.v[st][0], &p.tmap_v, 0, row, &sm.kv_full[st]);
        tma_load_2d(sm.v[st][1], &p.tmap_v, 64, row, &sm.kv_full[st]);
        if (tl.lo_row >= 0) {
          const int lrow = (int)((int64_t)bh * p.lo_rows_per_bh + tl.lo_row);
          tma_load_2d(sm.klo[st][0], &p.tmap_klo, 0, lrow, &sm.kv_full[st]);
          tma_load_2d(sm.klo[st][1], &p.tmap_klo, 64, lrow, &sm.kv_full[st]);
        }
      }
    }
  } else if (warp == 5) {
    // --------------------------------------------------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t id_s = idesc_f16(128, 64, 0, 0);
      constexpr uint32_t id_o = idesc_f16(128, 128, 0, 1);
      const uint32_t q0 = smem_u32(sm.q[0]);
      dwait(&sm.q_full, 0, p.status, 31, aborted);
      tc_fence_after();
      // S_j for j = 0, 1, ... and O += P_{j-1} V_{j-1}, software pipelined
      for (int j = 0; j <= T && !aborted; ++j) {
        if (j < T) {
          const int st = j % kDStages, sb = j & 1;
          if (!dwait(&sm.kv_full[st], (j / kDStages) & 1, p.status, 32, aborted)) break;
          if (j >= 2 && !dwait(&sm.s_free[sb], ((j >> 1) - 1) & 1, p.status, 33, aborted)) break;
          tc_fence_after();
          const uint32_t d = tmem + sb * 64;
          const bool lo = p.tiles[j].lo_row >= 0;
          const uint32_t kh0 = smem_u32(sm.khi[st][0]), kl0 = smem_u32(sm.klo[st][0]);
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const uint32_t aoff = (k >> 2) * 16384 + (k & 3) * 32;
            const uint32_t boff = (k >> 2) * 8192 + (k & 3) * 32;
            umma_f16(d, smem_desc_sw128(q0 + aoff, 16), smem_desc_sw128(kh0 + boff, 16), id_s, k > 0);
          }
          if (lo) {
#pragma unroll
            for (int k = 0; k < 8; ++k) {
              const uint32_t aoff = (k >> 2) * 16384 + (k & 3) * 32;
              const uint32_t boff = (k >> 2) * 8192 + (k & 3) * 32;
              umma_f16(d, smem_desc_sw128(q0 + aoff, 16), smem_desc_sw128(kl0 + boff, 16), id_s, 1);
            }
          }
          umma_commit(&sm.s_full[sb]);
        }
        if (j >= 1) {
          const int jj = j - 1, st = jj % kDStages, pb = jj & 1;
          if (!dwait(&sm.p_full[pb], (jj >> 1) & 1, p.status, 34, aborted)) break;
          tc_fence_after();
          const uint32_t p0 = smem_u32(sm.p[pb]), v0 = smem_u32(sm.v[st][0]);
#pragma unroll
          for (int k = 0; k < 4; ++k)
            umma_f16(tmem + 128, smem_desc_sw128(p0 + k * 32, 16), smem_desc_sw128(v0 + k * 2048, 8192), id_o,
                     (jj > 0 || k > 0) ? 1u : 0u);
          umma_commit(&sm.p_free[pb]);
          umma_commit(&sm.kv_empty[st]);
        }
      }
    }
  } else {
    // ------------------------------------------------------------ softmax
    const int r = threadIdx.x;  // query row within the tile = TMEM lane
    const int qi = qt * kDQ + r;
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
        *reinterpret_cast<uint4*>(sm.q[c >> 3] + r * 128 + (((c & 7) ^ (r & 7)) << 4)) = o;
      }
      fence_proxy_async_smem();
      mbar_arrive(&sm.q_full);
    }
    const uint32_t lane_off = (uint32_t)(32 * warp) << 16;
    float m_ref = kDNegInf, l = 0.f;
    float ls[UC_MAX_SEGMENTS];
#pragma unroll
    for (int s = 0; s < UC_MAX_SEGMENTS; ++s) ls[s] = 0.f;
    for (int j = 0; j < T; ++j) {
      const int sb = j & 1;
      if (!dwait_warp(&sm.s_full[sb], (j >> 1) & 1, p.status, 35, aborted)) break;
      tc_fence_after();
      uint32_t sr[2][32];
      tmem_ld32(tmem + lane_off + sb * 64, sr[0]);
      tmem_ld32(tmem + lane_off + sb * 64 + 32, sr[1]);
      tmem_wait_ld();
      tc_fence_before();
      mbar_arrive(&sm.s_free[sb]);
      const DenseTile tl = p.tiles[j];
      const int valid = min(kDK, max(0, p.seg[tl.seg].n_kept[b] - tl.seg_tile * kDK));
      float x[64];
      float tmax = kDNegInf;
#pragma unroll
      for (int c = 0; c < 64; ++c) {
        const float v = __uint_as_float(sr[c >> 5][c & 31]) * p.scale_log2;
        x[c] = (c < valid) ? v : kDNegInf;
        tmax = fmaxf(tmax, x[c]);
      }
      // lazy rescale: a row moves its reference max only when the tile's max
      // exceeds it by more than 8 (P <= 2^8); O in TMEM is rescaled by the
      // whole warp (collective TMEM access) once the previous P V completed
      const bool grow = tmax > m_ref + 8.f;
      const float m_new = grow ? tmax : m_ref;
      const bool need_o = grow && m_ref != kDNegInf && j >= 1;
      if (__any_sync(0xffffffffu, need_o)) {
        if (!dwait_warp(&sm.p_free[(j - 1) & 1], ((j - 1) >> 1) & 1, p.status, 36, aborted)) break;
        tc_fence_after();
        const float alpha = need_o ? exp2f(m_ref - m_new) : 1.f;
#pragma unroll 1
        for (int cb = 0; cb < 4; ++cb) {
          uint32_t o[32];
          tmem_ld32(tmem + lane_off + 128 + cb * 32, o);
          tmem_wait_ld();
#pragma unroll
          for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * alpha);
          tmem_st32(tmem + lane_off + 128 + cb * 32, o);
        }
        tmem_wait_st();
        tc_fence_before();
        l *= alpha;
#pragma unroll
        for (int s = 0; s < UC_MAX_SEGMENTS; ++s) ls[s] *= alpha;
      }
      m_ref = m_new;
      if (j >= 2 && !dwait_warp(&sm.p_free[sb], ((j >> 1) - 1) & 1, p.status, 37, aborted)) break;
      float sum = 0.f;
      uint8_t* prow = sm.p[sb] + r * 128;
#pragma unroll
      for (int c8 = 0; c8 < 8; ++c8) {
        uint32_t w[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float a = (m_ref == kDNegInf) ? 0.f : exp2f(x[8 * c8 + 2 * e] - m_ref);
          const float bb = (m_ref == kDNegInf) ? 0.f : exp2f(x[8 * c8 + 2 * e + 1] - m_ref);
          sum += a + bb;
          w[e] = pack_f16(a, bb);
        }
        *reinterpret_cast<uint4*>(prow + ((c8 ^ (r & 7)) << 4)) = make_uint4(w[0], w[1], w[2], w[3]);
      }
      l += sum;
#pragma unroll
      for (int s = 0; s < UC_MAX_SEGMENTS; ++s)
        if (s == tl.seg) ls[s] += sum;
      fence_proxy_async_smem();
      mbar_arrive(&sm.p_full[sb]);
    }
    // ------------------------------------------------------------ epilogue
    if (T > 0 && dwait_warp(&sm.p_free[(T - 1) & 1], ((T - 1) >> 1) & 1, p.status, 38, aborted)) {
      tc_fence_after();
      const float inv = (l > 0.f) ? 1.f / l : 0.f;
      __nv_bfloat16* orow = p.out + ((size_t)bhq * p.n_qtok + (row_ok ? qi : 0)) * kHeadDim;
#pragma unroll 1
      for (int cb = 0; cb < 4; ++cb) {
        uint32_t o[32];
        tmem_ld32(tmem + lane_off + 128 + cb * 32, o);
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
        if (p.mass)
          for (int s = 0; s < p.nseg; ++s) p.mass[orx * p.nseg + s] = ls[s] * inv;
      }
    }
    tc_fence_before();
  }
  __syncthreads();
  if (warp == 5) {
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
    cudaFuncSetAttribute(dense_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dense_smem_bytes());
  });
  const int nbh = p.batch * p.n_kv_heads;
  const int warps = nbh * p.n_tiles;
  materialize_kernel<<<(warps + 7) / 8, 256, 0, st>>>(p);
  count_launch();
  const int n_qt = (p.n_qtok + kDQ - 1) / kDQ;
  dense_kernel<<<p.batch * p.n_q_heads * n_qt, kDThreads, dense_smem_bytes(), st>>>(p);
  count_launch();
}

}  // namespace uc
