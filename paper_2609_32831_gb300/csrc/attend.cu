// Fused dequant-and-gather decode attention over heterogeneous segments
// (App. E "Attention over heterogeneous cache segments": one shared softmax
// across segments, chunks merged by log-sum-exp; Eq. 1's per-segment mass as
// a by-product).
//
// Design (GB300, HBM-bound): persistent CTAs walk a static list of work
// items; an item is one chunk of 64-token tiles of one segment of one
// (sequence, KV head). Per CTA one producer warp streams tiles into a
// 3-stage shared-memory ring (TMA 2D loads with 128-byte swizzle for bf16
// rows, 1D bulk copies for packed codes and parameters) and four consumer
// warps compute with mma.sync m16n8k16:
//   bf16 rows:  S = Q K^T in bf16 (exact products), P split into bf16 hi + lo
//               parts so P V keeps ~16 mantissa bits;
//   packed:     codes -> fp16 exactly (magic-number trick), x = code*s + z in
//               one fp16 FMA, S and P V in fp16 with fp32 accumulation.
// Each item leaves an unnormalised partial (O, m, l); the last CTA to finish
// a (sequence, KV head) merges its items by log-sum-exp, writes O, lse and
// the per-segment probability mass, and re-arms the counter.
#include "common.cuh"
#include "internal.h"

namespace uc {

constexpr int kTileTok = 64;
constexpr int kStages = 3;
constexpr int kConsumers = 4;
constexpr int kAttnThreads = 32 * (kConsumers + 1);
constexpr int kSlotBytes = 32768;
constexpr float kNegInf = -INFINITY;
constexpr float kLn2 = 0.69314718055994530942f;

// slot layout of a packed tile (two quantization groups)
constexpr int kSlotKParams = 4096;
constexpr int kSlotVCodes = 8192;
constexpr int kSlotVParams = 16384;

struct AttnSmem {
  uint8_t slot[kStages][kSlotBytes];
  uint64_t full[kStages];
  uint64_t empty[kStages];
  int last_flag;
};

__host__ __device__ size_t attend_part_floats(int mtiles) { return (size_t)mtiles * 16 * (kHeadDim + 2); }

__device__ __forceinline__ bool seg_is_bf16(int kind) {
  return kind == UC_KIND_FULL || kind == UC_KIND_EVICT;
}

// Tiles of a segment holding n tokens; *qtiles = packed tiles before the tail.
__device__ __forceinline__ int seg_tiles(const SegDev& sd, int n, int* qtiles) {
  if (seg_is_bf16(sd.kind)) {
    *qtiles = 0;
    return (n + kTileTok - 1) / kTileTok;
  }
  const int ng = n / kGroup;
  *qtiles = (ng + 1) / 2;
  return *qtiles + ((n % kGroup) ? 1 : 0);
}

struct ItemInfo {
  int bh, b, s, tb, te, qtiles, n;
};

__device__ __forceinline__ ItemInfo decode_item(const AttnParams& p, int it) {
  ItemInfo r;
  r.bh = it / p.items_per_bh;
  const int local = it % p.items_per_bh;
  r.b = r.bh / p.n_kv_heads;
  r.s = 0;
  for (int s = 0; s < p.nseg; ++s)
    if (local >= p.seg[s].chunk_begin) r.s = s;
  const SegDev& sd = p.seg[r.s];
  const int c = local - sd.chunk_begin;
  r.n = sd.n_kept[r.b];
  const int nt = seg_tiles(sd, r.n, &r.qtiles);
  r.tb = (int)(((int64_t)c * nt) / sd.n_chunks);
  r.te = (int)(((int64_t)(c + 1) * nt) / sd.n_chunks);
  return r;
}

__device__ __forceinline__ void consumer_sync() { asm volatile("bar.sync 1, 128;" ::: "memory"); }

__device__ __forceinline__ void fence_proxy_async() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ uint4 lds128(uint32_t a) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "r"(a));
  return v;
}

__device__ __forceinline__ uint2 lds64(uint32_t a) {
  uint2 v;
  asm volatile("ld.shared.v2.u32 {%0,%1}, [%2];" : "=r"(v.x), "=r"(v.y) : "r"(a));
  return v;
}

// ------------------------------------------------------------- producer
__device__ void produce(const AttnParams& p, AttnSmem& sm) {
  uint32_t seq = 0;
  for (int it = blockIdx.x; it < p.n_items; it += gridDim.x) {
    const ItemInfo ii = decode_item(p, it);
    const SegDev& sd = p.seg[ii.s];
    for (int t = ii.tb; t < ii.te; ++t, ++seq) {
      const int slot = seq % kStages;
      if (seq >= kStages && !mbar_wait(&sm.empty[slot], ((seq / kStages) - 1) & 1, p.status, 10))
        return;
      uint8_t* dst = sm.slot[slot];
      const bool tail = !seg_is_bf16(sd.kind) && t >= ii.qtiles;
      if (seg_is_bf16(sd.kind) || tail) {
        int64_t row;
        if (tail)
          row = (int64_t)ii.bh * kGroup;
        else
          row = (int64_t)ii.bh * sd.row_stride + sd.row_offset + (int64_t)t * kTileTok;
        mbar_arrive_expect_tx(&sm.full[slot], kSlotBytes);
        const CUtensorMap* mk = &p.tmap[2 * ii.s];
        const CUtensorMap* mv = &p.tmap[2 * ii.s + 1];
        tma_load_2d(dst, mk, 0, (int)row, &sm.full[slot]);
        tma_load_2d(dst + 8192, mk, 64, (int)row, &sm.full[slot]);
        tma_load_2d(dst + 16384, mv, 0, (int)row, &sm.full[slot]);
        tma_load_2d(dst + 24576, mv, 64, (int)row, &sm.full[slot]);
      } else {
        const int ng = ii.n / kGroup;
        const int g0 = 2 * t;
        const int ngt = min(2, ng - g0);
        const uint32_t kc = 32 * kHeadDim * sd.bits / 8;  // code bytes per group (K or V)
        const uint32_t bytes = (uint32_t)ngt * (2 * kc + 1024);
        mbar_arrive_expect_tx(&sm.full[slot], bytes);
        const size_t blk_codes = (size_t)ii.bh * sd.cap * kHeadDim * sd.bits / 8;
        const size_t blk_kpar = (size_t)ii.bh * (sd.cap / kGroup) * 512;
        const size_t blk_vpar = (size_t)ii.bh * sd.cap * 16;
        bulk_load(dst, sd.k_codes + blk_codes + (size_t)g0 * kc, ngt * kc, &sm.full[slot]);
        bulk_load(dst + kSlotKParams, sd.k_params + blk_kpar + (size_t)g0 * 512, ngt * 512,
                  &sm.full[slot]);
        bulk_load(dst + kSlotVCodes, sd.v_codes + blk_codes + (size_t)g0 * kc, ngt * kc,
                  &sm.full[slot]);
        bulk_load(dst + kSlotVParams, sd.v_params + blk_vpar + (size_t)g0 * 512, ngt * 512,
                  &sm.full[slot]);
      }
    }
  }
}

// ------------------------------------------------------------- consumer
struct WarpState {
  float o[16][4];
  float m0, m1, l0, l1;
};

__device__ __forceinline__ void online_softmax(WarpState& st, float (&x)[2][4], float (&pr)[2][4]) {
  float r0 = fmaxf(fmaxf(x[0][0], x[0][1]), fmaxf(x[1][0], x[1][1]));
  float r1 = fmaxf(fmaxf(x[0][2], x[0][3]), fmaxf(x[1][2], x[1][3]));
  r0 = fmaxf(r0, __shfl_xor_sync(0xffffffffu, r0, 1));
  r0 = fmaxf(r0, __shfl_xor_sync(0xffffffffu, r0, 2));
  r1 = fmaxf(r1, __shfl_xor_sync(0xffffffffu, r1, 1));
  r1 = fmaxf(r1, __shfl_xor_sync(0xffffffffu, r1, 2));
  const float n0 = fmaxf(st.m0, r0), n1 = fmaxf(st.m1, r1);
  const float u0 = (n0 == kNegInf) ? 0.f : n0;
  const float u1 = (n1 == kNegInf) ? 0.f : n1;
  const float a0 = exp2f(st.m0 - u0), a1 = exp2f(st.m1 - u1);
#pragma unroll
  for (int nt = 0; nt < 2; ++nt) {
    pr[nt][0] = exp2f(x[nt][0] - u0);
    pr[nt][1] = exp2f(x[nt][1] - u0);
    pr[nt][2] = exp2f(x[nt][2] - u1);
    pr[nt][3] = exp2f(x[nt][3] - u1);
  }
  st.l0 = st.l0 * a0 + (pr[0][0] + pr[0][1] + pr[1][0] + pr[1][1]);
  st.l1 = st.l1 * a1 + (pr[0][2] + pr[0][3] + pr[1][2] + pr[1][3]);
  if (__any_sync(0xffffffffu, a0 != 1.f || a1 != 1.f)) {
#pragma unroll
    for (int n = 0; n < 16; ++n) {
      st.o[n][0] *= a0;
      st.o[n][1] *= a0;
      st.o[n][2] *= a1;
      st.o[n][3] *= a1;
    }
  }
  st.m0 = n0;
  st.m1 = n1;
}

__device__ __forceinline__ uint32_t swz(uint32_t base, int key, int chunk) {
  return base + (chunk >> 3) * 8192 + key * 128 + ((((chunk & 7) ^ (key & 7))) << 4);
}

// One 16-key subunit of a bf16 tile.
__device__ __forceinline__ void sub_bf16(WarpState& st, const uint32_t (&qb)[8][4], uint32_t kbase,
                                         int u, int valid, float scale) {
  const int lane = threadIdx.x & 31;
  const int mi = lane >> 3, rr = lane & 7, j = lane & 3;
  float s[2][4] = {};
  const int kk = 16 * u + 8 * (mi >> 1) + rr;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    uint32_t b0, b1, b2, b3;
    ldsm_x4(swz(kbase, kk, 2 * i + (mi & 1)), b0, b1, b2, b3);
    mma_bf16(s[0], qb[i], b0, b1);
    mma_bf16(s[1], qb[i], b2, b3);
  }
  float x[2][4], pr[2][4];
  const int key0 = 16 * u + 2 * j;
#pragma unroll
  for (int nt = 0; nt < 2; ++nt)
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      const bool ok = key0 + 8 * nt + e < valid;
      x[nt][e] = ok ? s[nt][e] * scale : kNegInf;
      x[nt][2 + e] = ok ? s[nt][2 + e] * scale : kNegInf;
    }
  online_softmax(st, x, pr);
  uint32_t ah[4], al[4];
  ah[0] = pack_bf16(pr[0][0], pr[0][1]);
  ah[1] = pack_bf16(pr[0][2], pr[0][3]);
  ah[2] = pack_bf16(pr[1][0], pr[1][1]);
  ah[3] = pack_bf16(pr[1][2], pr[1][3]);
  al[0] = pack_bf16(pr[0][0] - bf16_lo(ah[0]), pr[0][1] - bf16_hi(ah[0]));
  al[1] = pack_bf16(pr[0][2] - bf16_lo(ah[1]), pr[0][3] - bf16_hi(ah[1]));
  al[2] = pack_bf16(pr[1][0] - bf16_lo(ah[2]), pr[1][1] - bf16_hi(ah[2]));
  al[3] = pack_bf16(pr[1][2] - bf16_lo(ah[3]), pr[1][3] - bf16_hi(ah[3]));
  const uint32_t vbase = kbase + 16384;
  const int vk = 16 * u + 8 * (mi & 1) + rr;
#pragma unroll
  for (int m2 = 0; m2 < 8; ++m2) {
    uint32_t r0, r1, r2, r3;
    ldsm_x4_t(swz(vbase, vk, 2 * m2 + (mi >> 1)), r0, r1, r2, r3);
    mma_bf16(st.o[2 * m2], ah, r0, r1);
    mma_bf16(st.o[2 * m2], al, r0, r1);
    mma_bf16(st.o[2 * m2 + 1], ah, r2, r3);
    mma_bf16(st.o[2 * m2 + 1], al, r2, r3);
  }
}

// One 16-key subunit of a packed tile (both groups complete).
template <int BITS>
__device__ __forceinline__ void sub_quant(WarpState& st, const uint32_t (&qh)[8][4], uint32_t base,
                                          int u, float scale) {
  constexpr int MASK = (1 << BITS) - 1;
  const int lane = threadIdx.x & 31;
  const int j = lane & 3;
  float s[2][4] = {};
  uint32_t kw[2][4];
#pragma unroll
  for (int nt = 0; nt < 2; ++nt) {
    const uint32_t a = base + ((2 * u + nt) * 32 + lane) * (BITS * 4);
    if (BITS == 4) {
      const uint4 v = lds128(a);
      kw[nt][0] = v.x;
      kw[nt][1] = v.y;
      kw[nt][2] = v.z;
      kw[nt][3] = v.w;
    } else {
      const uint2 v = lds64(a);
      kw[nt][0] = v.x;
      kw[nt][1] = v.y;
      kw[nt][2] = 0;
      kw[nt][3] = 0;
    }
  }
  const uint32_t kp = base + kSlotKParams + (u >> 1) * 512 + j * 16;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const uint4 P = lds128(kp + i * 64);
#pragma unroll
    for (int nt = 0; nt < 2; ++nt) {
      uint32_t w;
      int sh0, sh1;
      if (BITS == 4) {
        w = kw[nt][i >> 1];
        sh0 = 4 * (2 * (i & 1));
        sh1 = sh0 + 4;
      } else {
        w = kw[nt][i >> 2];
        sh0 = 2 * (2 * (i & 3));
        sh1 = sh0 + 2;
      }
      const uint32_t b0 = hfma2_u32(codes_to_h2<MASK>(w, sh0), P.x, P.z);
      const uint32_t b1 = hfma2_u32(codes_to_h2<MASK>(w, sh1), P.y, P.w);
      mma_f16(s[nt], qh[i], b0, b1);
    }
  }
  float x[2][4], pr[2][4];
#pragma unroll
  for (int nt = 0; nt < 2; ++nt)
#pragma unroll
    for (int e = 0; e < 4; ++e) x[nt][e] = s[nt][e] * scale;
  online_softmax(st, x, pr);
  uint32_t a[4];
  a[0] = pack_f16(pr[0][0], pr[0][1]);
  a[1] = pack_f16(pr[0][2], pr[0][3]);
  a[2] = pack_f16(pr[1][0], pr[1][1]);
  a[3] = pack_f16(pr[1][2], pr[1][3]);
  uint32_t vw[8];
  {
    const uint32_t va = base + kSlotVCodes + (u * 32 + lane) * (BITS * 8);
    const uint4 v0 = lds128(va);
    vw[0] = v0.x;
    vw[1] = v0.y;
    vw[2] = v0.z;
    vw[3] = v0.w;
    if (BITS == 4) {
      const uint4 v1 = lds128(va + 16);
      vw[4] = v1.x;
      vw[5] = v1.y;
      vw[6] = v1.z;
      vw[7] = v1.w;
    } else {
      vw[4] = vw[5] = vw[6] = vw[7] = 0;
    }
  }
  uint4 vp[4];
#pragma unroll
  for (int g = 0; g < 4; ++g) vp[g] = lds128(base + kSlotVParams + u * 256 + (g * 4 + j) * 16);
#pragma unroll
  for (int m = 0; m < 16; ++m) {
    const uint4& P = vp[m >> 2];
    uint32_t w;
    int sh0, sh1;
    if (BITS == 4) {
      w = vw[m >> 1];
      sh0 = 4 * (2 * (m & 1));
      sh1 = sh0 + 4;
    } else {
      w = vw[m >> 2];
      sh0 = 2 * (2 * (m & 3));
      sh1 = sh0 + 2;
    }
    const uint32_t b0 = hfma2_u32(codes_to_h2<MASK>(w, sh0), P.x, P.z);
    const uint32_t b1 = hfma2_u32(codes_to_h2<MASK>(w, sh1), P.y, P.w);
    mma_f16(st.o[m], a, b0, b1);
  }
}

// Zero the V rows [valid, 64) of a bf16 tile that lie in subunit u.
__device__ __forceinline__ void zero_v_rows(uint8_t* slot, int u, int valid) {
  const int lane = threadIdx.x & 31;
  const int lo = max(valid, 16 * u), hi = 16 * u + 16;
  for (int r = lo; r < hi; ++r) {
    uint8_t* row0 = slot + 16384 + r * 128;
    if (lane < 8)
      *reinterpret_cast<uint4*>(row0 + lane * 16) = make_uint4(0, 0, 0, 0);
    else if (lane < 16)
      *reinterpret_cast<uint4*>(row0 + 8192 + (lane - 8) * 16) = make_uint4(0, 0, 0, 0);
  }
  __syncwarp();
}

__device__ void final_merge(const AttnParams& p, int bh) {
  const int tid = threadIdx.x;  // 0..127 = channel
  const int b = bh / p.n_kv_heads, kvh = bh % p.n_kv_heads;
  const size_t pf = attend_part_floats(p.mtiles);
  const int rows_pad = 16 * p.mtiles;
  const float* base = p.part + (size_t)bh * p.items_per_bh * pf;
  for (int r = 0; r < p.rows; ++r) {
    float M = kNegInf;
    for (int i = 0; i < p.items_per_bh; ++i)
      M = fmaxf(M, __ldcg(base + i * pf + rows_pad * kHeadDim + r));
    const float Mu = (M == kNegInf) ? 0.f : M;
    float L = 0.f, acc = 0.f;
    float Ls[UC_MAX_SEGMENTS];
#pragma unroll
    for (int s = 0; s < UC_MAX_SEGMENTS; ++s) Ls[s] = 0.f;
    for (int i = 0; i < p.items_per_bh; ++i) {
      const float* pi = base + i * pf;
      const float mi = __ldcg(pi + rows_pad * kHeadDim + r);
      const float li = __ldcg(pi + rows_pad * kHeadDim + rows_pad + r);
      const float w = (mi == kNegInf) ? 0.f : exp2f(mi - Mu);
      L += li * w;
      acc += w * __ldcg(pi + r * kHeadDim + tid);
      int s = 0;
      for (int q = 0; q < p.nseg; ++q)
        if (i >= p.seg[q].chunk_begin) s = q;
#pragma unroll
      for (int q = 0; q < UC_MAX_SEGMENTS; ++q)
        if (q == s) Ls[q] += li * w;
    }
    const int hl = r / p.n_qtok, t = r % p.n_qtok;
    const int h = kvh * p.group + hl;
    const size_t orow = ((size_t)(b * p.n_q_heads + h) * p.n_qtok + t);
    const float inv = (L > 0.f) ? 1.f / L : 0.f;
    p.out[orow * kHeadDim + tid] = __float2bfloat16_rn(acc * inv);
    if (tid == 0) {
      if (p.lse) p.lse[orow] = (L > 0.f) ? (M + log2f(L)) * kLn2 : kNegInf;
      if (p.mass)
        for (int q = 0; q < p.nseg; ++q) p.mass[orow * p.nseg + q] = Ls[q] * inv;
    }
  }
}

__global__ void __launch_bounds__(kAttnThreads, 2) attend_kernel(const __grid_constant__ AttnParams p) {
  extern __shared__ uint8_t dyn_smem[];
  AttnSmem& sm = *reinterpret_cast<AttnSmem*>(
      (reinterpret_cast<uintptr_t>(dyn_smem) + 1023) & ~static_cast<uintptr_t>(1023));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&sm.full[s], 1);
      mbar_init(&sm.empty[s], kConsumers);
    }
    fence_barrier_init();
  }
  __syncthreads();

  if (warp == kConsumers) {
    if (lane == 0) {
      for (int s = 0; s < p.nseg; ++s) {
        prefetch_tmap(&p.tmap[2 * s]);
        prefetch_tmap(&p.tmap[2 * s + 1]);
      }
      produce(p, sm);
    }
    return;
  }

  // ---------------------------------------------------------- consumers
  const int MT = p.mtiles, KS = kConsumers / MT;
  const int mt = warp % MT, ks = warp / MT;
  const int g = lane >> 2, j = lane & 3;
  const size_t pf = attend_part_floats(MT);
  const int rows_pad = 16 * MT;
  uint32_t seq = 0;
  bool aborted = false;

  for (int it = blockIdx.x; it < p.n_items; it += gridDim.x) {
    const ItemInfo ii = decode_item(p, it);
    const SegDev& sd = p.seg[ii.s];
    const int kvh = ii.bh % p.n_kv_heads;

    // query fragments of this warp's m-tile (bf16 and an fp16 copy)
    uint32_t qb[8][4], qh[8][4];
    {
      const int r0 = mt * 16 + g, r1 = r0 + 8;
      const __nv_bfloat16* q0 = nullptr;
      const __nv_bfloat16* q1 = nullptr;
      if (r0 < p.rows)
        q0 = p.q + ((size_t)(ii.b * p.n_q_heads + kvh * p.group + r0 / p.n_qtok) * p.n_qtok +
                    r0 % p.n_qtok) * kHeadDim;
      if (r1 < p.rows)
        q1 = p.q + ((size_t)(ii.b * p.n_q_heads + kvh * p.group + r1 / p.n_qtok) * p.n_qtok +
                    r1 % p.n_qtok) * kHeadDim;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int c = 16 * i + 2 * j;
        qb[i][0] = q0 ? *reinterpret_cast<const uint32_t*>(q0 + c) : 0u;
        qb[i][1] = q1 ? *reinterpret_cast<const uint32_t*>(q1 + c) : 0u;
        qb[i][2] = q0 ? *reinterpret_cast<const uint32_t*>(q0 + c + 8) : 0u;
        qb[i][3] = q1 ? *reinterpret_cast<const uint32_t*>(q1 + c + 8) : 0u;
#pragma unroll
        for (int e = 0; e < 4; ++e) qh[i][e] = pack_f16(bf16_lo(qb[i][e]), bf16_hi(qb[i][e]));
      }
    }

    WarpState st;
#pragma unroll
    for (int n = 0; n < 16; ++n) st.o[n][0] = st.o[n][1] = st.o[n][2] = st.o[n][3] = 0.f;
    st.m0 = st.m1 = kNegInf;
    st.l0 = st.l1 = 0.f;

    int last_slot = -1;
    for (int t = ii.tb; t < ii.te; ++t, ++seq) {
      const int slot = seq % kStages;
      if (!aborted && !mbar_wait(&sm.full[slot], (seq / kStages) & 1, p.status, 11)) aborted = true;
      const uint32_t sbase = smem_u32(sm.slot[slot]);
      if (!aborted) {
        const bool tail = !seg_is_bf16(sd.kind) && t >= ii.qtiles;
        if (seg_is_bf16(sd.kind) || tail) {
          const int valid = tail ? (ii.n % kGroup) : min(kTileTok, ii.n - t * kTileTok);
          for (int x = 0; x < MT; ++x) {
            const int u = ks + KS * x;
            if (16 * u >= valid) continue;
            if (valid < 16 * u + 16) zero_v_rows(sm.slot[slot], u, valid);
            sub_bf16(st, qb, sbase, u, valid, p.scale_log2);
          }
        } else {
          const int ng = ii.n / kGroup;
          const int valid = 32 * min(2, ng - 2 * t);
          for (int x = 0; x < MT; ++x) {
            const int u = ks + KS * x;
            if (16 * u >= valid) continue;
            if (sd.bits == 4)
              sub_quant<4>(st, qh, sbase, u, p.scale_log2);
            else
              sub_quant<2>(st, qh, sbase, u, p.scale_log2);
          }
        }
      }
      if (t + 1 < ii.te || KS == 1) {
        fence_proxy_async();
        __syncwarp();
        if (lane == 0) mbar_arrive(&sm.empty[slot]);
      } else {
        last_slot = slot;
      }
    }

    // full row sums
    st.l0 += __shfl_xor_sync(0xffffffffu, st.l0, 1);
    st.l0 += __shfl_xor_sync(0xffffffffu, st.l0, 2);
    st.l1 += __shfl_xor_sync(0xffffffffu, st.l1, 1);
    st.l1 += __shfl_xor_sync(0xffffffffu, st.l1, 2);

    // merge the warps that share an m-tile, through the last slot
    if (KS > 1 && last_slot >= 0) {
      float* buf = reinterpret_cast<float*>(sm.slot[last_slot]);
      consumer_sync();
      for (int step = 1; step < KS; step *= 2) {
        const bool writer = (ks % (2 * step)) == step;
        const bool reader = (ks % (2 * step)) == 0;
        const int region = (ks / (2 * step)) * MT + mt;
        float* rb = buf + region * (68 * 32);
        if (writer) {
#pragma unroll
          for (int n = 0; n < 16; ++n)
#pragma unroll
            for (int e = 0; e < 4; ++e) rb[(n * 4 + e) * 32 + lane] = st.o[n][e];
          rb[64 * 32 + lane] = st.m0;
          rb[65 * 32 + lane] = st.m1;
          rb[66 * 32 + lane] = st.l0;
          rb[67 * 32 + lane] = st.l1;
        }
        consumer_sync();
        if (reader) {
          const float om0 = rb[64 * 32 + lane], om1 = rb[65 * 32 + lane];
          const float ol0 = rb[66 * 32 + lane], ol1 = rb[67 * 32 + lane];
          const float n0 = fmaxf(st.m0, om0), n1 = fmaxf(st.m1, om1);
          const float u0 = (n0 == kNegInf) ? 0.f : n0, u1 = (n1 == kNegInf) ? 0.f : n1;
          const float a0 = exp2f(st.m0 - u0), b0 = exp2f(om0 - u0);
          const float a1 = exp2f(st.m1 - u1), b1 = exp2f(om1 - u1);
#pragma unroll
          for (int n = 0; n < 16; ++n) {
            st.o[n][0] = st.o[n][0] * a0 + rb[(n * 4 + 0) * 32 + lane] * b0;
            st.o[n][1] = st.o[n][1] * a0 + rb[(n * 4 + 1) * 32 + lane] * b0;
            st.o[n][2] = st.o[n][2] * a1 + rb[(n * 4 + 2) * 32 + lane] * b1;
            st.o[n][3] = st.o[n][3] * a1 + rb[(n * 4 + 3) * 32 + lane] * b1;
          }
          st.l0 = st.l0 * a0 + ol0 * b0;
          st.l1 = st.l1 * a1 + ol1 * b1;
          st.m0 = n0;
          st.m1 = n1;
        }
        consumer_sync();
      }
      fence_proxy_async();
      __syncwarp();
      if (lane == 0) mbar_arrive(&sm.empty[last_slot]);
    }

    // this item's partial
    if (ks == 0) {
      float* pi = p.part + (size_t)it * pf;
      const int r0 = mt * 16 + g, r1 = r0 + 8;
#pragma unroll
      for (int n = 0; n < 16; ++n) {
        const int c = 8 * n + 2 * j;
        *reinterpret_cast<float2*>(pi + r0 * kHeadDim + c) = make_float2(st.o[n][0], st.o[n][1]);
        *reinterpret_cast<float2*>(pi + r1 * kHeadDim + c) = make_float2(st.o[n][2], st.o[n][3]);
      }
      if (j == 0) {
        pi[rows_pad * kHeadDim + r0] = st.m0;
        pi[rows_pad * kHeadDim + r1] = st.m1;
        pi[rows_pad * kHeadDim + rows_pad + r0] = st.l0;
        pi[rows_pad * kHeadDim + rows_pad + r1] = st.l1;
      }
    }
    __threadfence();
    consumer_sync();
    if (threadIdx.x == 0) {
      const int prev = atomicAdd(&p.counters[ii.bh], 1);
      sm.last_flag = (prev == p.items_per_bh - 1);
    }
    consumer_sync();
    if (sm.last_flag) {
      __threadfence();
      final_merge(p, ii.bh);
      consumer_sync();
      if (threadIdx.x == 0) p.counters[ii.bh] = 0;
    }
    consumer_sync();
  }
}

int attend_ctas_per_sm() {
  int n = 0;
  const size_t smem = sizeof(AttnSmem) + 1024;
  cudaFuncSetAttribute(attend_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, attend_kernel, kAttnThreads, smem);
  return n > 0 ? n : 1;
}

void launch_attend(const AttnParams& p, int grid, cudaStream_t st) {
  const size_t smem = sizeof(AttnSmem) + 1024;
  cudaFuncSetAttribute(attend_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  attend_kernel<<<grid, kAttnThreads, smem, st>>>(p);
  count_launch();
}

}  // namespace uc
