// Group quantization of one run of 32 kept tokens, by one warp, into the
// fragment-ordered packed layout declared in unicache.h.
//
// Keys are quantized per channel over the 32 tokens, values per token over
// each run of 32 channels (App. E storage; constants from the measured
// workloads). Every step is IEEE fp32 round-to-nearest-even:
//   s = fp16((max - min) / qmax), z = fp16(min + 0) (a zero minimum is
//   stored as +0, whichever signed zero the minimum search returns),
//   code = clamp(rint((x - z) / s), 0, qmax), code = 0 if s == 0.
// The explicit __fsub_rn / __fdiv_rn calls keep the compiler from contracting
// or approximating these operations.
#pragma once

#include "common.cuh"

namespace uc {

struct QuantOut {
  uint8_t* k_codes;   // block base (b, kvh)
  uint8_t* k_params;
  uint8_t* v_codes;
  uint8_t* v_params;
};

// Per-warp shared scratch: codes [32 tokens][128 channels] (rows padded to
// 132 bytes so that rows 128 B apart do not share banks) and params.
constexpr int kCodeRow = 132;
struct QuantSmem {
  uint8_t code[32][kCodeRow];
  __half s[128];
  __half z[128];
  __half vs[32][4];
  __half vz[32][4];
};

// code = clamp(rint(fl(t / s)), 0, qmax) with t = fl(x - z) and fl() IEEE
// round-to-nearest. The quotient is first formed as t * fl(1 / s), which is
// within 1.5 * 2^-23 |t / s| of fl(t / s); its rounding to an integer can
// only differ from that of fl(t / s) when it lies within that distance of a
// half-integer, and only then is the correctly rounded division taken.
// Quotients clamp outside [0, qmax], so only |q| <= qmax + 1 needs care.
//
// Split in two so that the common path has no branch: q_code_fast returns
// the code from t * fl(1 / s) and raises `near` when the quotient lies that
// close to a half-integer; the caller then redoes its elements with
// q_code_exact (rare: about one element in 10^5). The test uses one bound for
// the whole clamp range, 4e-6 (qmax + 2) >= 4e-6 max(1, |q|) for
// |q| <= qmax + 2 (quotients beyond clamp to qmax whichever way they round,
// and a spurious `near` only costs the exact recomputation).
__device__ __forceinline__ uint32_t q_code_fast(float x, float z, float inv_s, uint32_t qmax, bool& near) {
  const float t = __fsub_rn(x, z);
  const float q = __fmul_rn(t, inv_s);
  const float r = rintf(q);  // round half to even
  near |= fabsf(fabsf(__fsub_rn(q, r)) - 0.5f) <= 4e-6f * (float)(qmax + 2u);
  // r is integral: negative -> 0 (saturating conversion), then clamp to qmax
  return min(__float2uint_rz(r), qmax);
}

__device__ __forceinline__ uint32_t q_code_exact(float x, float z, float s, uint32_t qmax) {
  if (s == 0.0f) return 0u;
  return min(__float2uint_rn(__fdiv_rn(__fsub_rn(x, z), s)), qmax);
}

__device__ __forceinline__ bool half_finite(__half h) {
  return (__half_as_ushort(h) & 0x7c00u) != 0x7c00u;
}

// Quantize group `g` (tokens 32g .. 32g+31 of the kept sequence). Row t of
// the group is read from krow(t) / vrow(t) (bf16, 128 channels). Returns
// false (in every lane) if a value was not finite or a scale / zero-point
// overflowed fp16; nothing is written in that case.
template <int BITS, typename RowK, typename RowV>
__device__ bool quantize_group_warp(RowK krow, RowV vrow, int g, QuantOut out, QuantSmem& sm) {
  constexpr float qmax = (float)((1 << BITS) - 1);
  constexpr uint32_t qmax_u = (1u << BITS) - 1u;
  const int lane = threadIdx.x & 31;
  bool ok = true;

  // ---- keys: lane owns channels 4*lane .. 4*lane+3 over the 32 tokens
  {
    uint2 raw[32];
#pragma unroll
    for (int t = 0; t < 32; ++t) raw[t] = *reinterpret_cast<const uint2*>(krow(t) + 4 * lane);
    float mn[4], mx[4];
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      mn[c] = INFINITY;
      mx[c] = -INFINITY;
    }
#pragma unroll
    for (int t = 0; t < 32; ++t) {
      const float x[4] = {bf16_lo(raw[t].x), bf16_hi(raw[t].x), bf16_lo(raw[t].y), bf16_hi(raw[t].y)};
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        ok = ok && isfinite(x[c]);
        mn[c] = fminf(mn[c], x[c]);
        mx[c] = fmaxf(mx[c], x[c]);
      }
    }
    float sf[4], zf[4], rf[4];
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const __half s = __float2half_rn(__fdiv_rn(__fsub_rn(mx[c], mn[c]), qmax));
      const __half z = __float2half_rn(__fadd_rn(mn[c], 0.0f));
      ok = ok && half_finite(s) && half_finite(z);
      sm.s[4 * lane + c] = s;
      sm.z[4 * lane + c] = z;
      sf[c] = __half2float(s);
      zf[c] = __half2float(z);
      rf[c] = sf[c] != 0.0f ? __frcp_rn(sf[c]) : 0.0f;  // s == 0: every code is 0
    }
    bool near = false;
#pragma unroll
    for (int t = 0; t < 32; ++t) {
      const float x[4] = {bf16_lo(raw[t].x), bf16_hi(raw[t].x), bf16_lo(raw[t].y), bf16_hi(raw[t].y)};
      uint32_t packed = 0;
#pragma unroll
      for (int c = 0; c < 4; ++c) packed |= q_code_fast(x[c], zf[c], rf[c], qmax_u, near) << (8 * c);
      *reinterpret_cast<uint32_t*>(&sm.code[t][4 * lane]) = packed;
    }
    if (near) {
#pragma unroll 1
      for (int t = 0; t < 32; ++t) {
        const float x[4] = {bf16_lo(raw[t].x), bf16_hi(raw[t].x), bf16_lo(raw[t].y), bf16_hi(raw[t].y)};
        uint32_t packed = 0;
        for (int c = 0; c < 4; ++c) packed |= q_code_exact(x[c], zf[c], sf[c], qmax_u) << (8 * c);
        *reinterpret_cast<uint32_t*>(&sm.code[t][4 * lane]) = packed;
      }
    }
  }
  ok = __all_sync(0xffffffffu, ok);
  __syncwarp();
  if (ok) {
    // K codes: 4 tiles of 8 tokens; lane L = (n, j) gets token 8*nt + n,
    // channels {16i + 2j + 8*sub + e}.
    const int n = lane >> 2, j = lane & 3;
#pragma unroll
    for (int nt = 0; nt < 4; ++nt) {
      const uint8_t* row = sm.code[nt * 8 + n];
      constexpr int kWords = BITS;  // int4: 4 words (16 B), int2: 2 words (8 B)
      uint32_t w[kWords];
#pragma unroll
      for (int q = 0; q < kWords; ++q) {
        uint32_t word = 0;
        constexpr int kPairs = 16 / BITS / 2 * 2;  // pairs per word: 4 (int4) or 8 (int2)
#pragma unroll
        for (int p = 0; p < kPairs; ++p) {
          const int i = q * (kPairs / 2) + p / 2;
          const int sub = p & 1;
          const int ca = 16 * i + 2 * j + 8 * sub;
          // codes of channels ca, ca + 1 -> bits BITS p and 16 + BITS p
          const uint32_t h = *reinterpret_cast<const uint16_t*>(row + ca);
          word |= __byte_perm(h, 0u, 0x4140) << (BITS * p);
        }
        w[q] = word;
      }
      uint8_t* dst = out.k_codes + ((size_t)(g * 4 + nt) * 32 + lane) * (BITS * 4);
      if (BITS == 4)
        *reinterpret_cast<uint4*>(dst) = make_uint4(w[0], w[1], w[BITS > 2 ? 2 : 0], w[BITS > 2 ? 3 : 0]);
      else
        *reinterpret_cast<uint2*>(dst) = make_uint2(w[0], w[1]);
    }
    // K params: lane -> entry (j = lane / 8, i = lane % 8)
    {
      const int jj = lane >> 3, i = lane & 7;
      const int c0 = 16 * i + 2 * jj;
      __half2 s01 = __halves2half2(sm.s[c0], sm.s[c0 + 1]);
      __half2 s89 = __halves2half2(sm.s[c0 + 8], sm.s[c0 + 9]);
      __half2 z01 = __halves2half2(sm.z[c0], sm.z[c0 + 1]);
      __half2 z89 = __halves2half2(sm.z[c0 + 8], sm.z[c0 + 9]);
      uint4 e = make_uint4(*reinterpret_cast<uint32_t*>(&s01), *reinterpret_cast<uint32_t*>(&s89),
                           *reinterpret_cast<uint32_t*>(&z01), *reinterpret_cast<uint32_t*>(&z89));
      *reinterpret_cast<uint4*>(out.k_params + (size_t)g * 512 + (i * 4 + jj) * 16) = e;
    }
  }
  __syncwarp();

  // ---- values: per token, channel group = lane / 8 (all 32 rows are loaded
  // first, so their latencies overlap)
  bool okv = true;
  {
    const float inf = INFINITY;
    uint2 raw[32];
#pragma unroll
    for (int t = 0; t < 32; ++t) raw[t] = *reinterpret_cast<const uint2*>(vrow(t) + 4 * lane);
#pragma unroll 4
    for (int t = 0; t < 32; ++t) {
      const uint2 r = raw[t];
      const float x[4] = {bf16_lo(r.x), bf16_hi(r.x), bf16_lo(r.y), bf16_hi(r.y)};
      float mn = inf, mx = -inf;
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        okv = okv && isfinite(x[c]);
        mn = fminf(mn, x[c]);
        mx = fmaxf(mx, x[c]);
      }
#pragma unroll
      for (int o = 1; o < 8; o <<= 1) {
        mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, o));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
      }
      const __half s = __float2half_rn(__fdiv_rn(__fsub_rn(mx, mn), qmax));
      const __half z = __float2half_rn(__fadd_rn(mn, 0.0f));
      okv = okv && half_finite(s) && half_finite(z);
      const float sf = __half2float(s), zf = __half2float(z);
      const float rf = sf != 0.0f ? __frcp_rn(sf) : 0.0f;  // s == 0: every code is 0
      bool near = false;
      uint32_t packed = 0;
#pragma unroll
      for (int c = 0; c < 4; ++c) packed |= q_code_fast(x[c], zf, rf, qmax_u, near) << (8 * c);
      if (near) {
        packed = 0;
        for (int c = 0; c < 4; ++c) packed |= q_code_exact(x[c], zf, sf, qmax_u) << (8 * c);
      }
      *reinterpret_cast<uint32_t*>(&sm.code[t][4 * lane]) = packed;
      if ((lane & 7) == 0) {
        sm.vs[t][lane >> 3] = s;
        sm.vz[t][lane >> 3] = z;
      }
    }
  }
  okv = __all_sync(0xffffffffu, okv) && ok;
  __syncwarp();
  if (okv) {
    // V codes: 2 tiles of 16 tokens; lane L = (gq, j): tokens {2j, 2j+1,
    // 2j+8, 2j+9} of the tile, channels {8m + gq}.
    const int gq = lane >> 2, j = lane & 3;
#pragma unroll
    for (int kt = 0; kt < 2; ++kt) {
      constexpr int kWords = 2 * BITS;  // int4: 8 words (32 B), int2: 4 words (16 B)
      constexpr int kPairs = 16 / BITS;  // pairs per word: 4 (int4) or 8 (int2)
      uint32_t w[kWords];
#pragma unroll
      for (int q = 0; q < kWords; ++q) {
        uint32_t word = 0;
#pragma unroll
        for (int p = 0; p < kPairs; ++p) {
          const int m = q * (kPairs / 2) + p / 2;
          const int sub = p & 1;
          const int ta = kt * 16 + 2 * j + 8 * sub;
          const int c = 8 * m + gq;
          word |= (uint32_t)sm.code[ta][c] << (BITS * p);
          word |= (uint32_t)sm.code[ta + 1][c] << (16 + BITS * p);
        }
        w[q] = word;
      }
      uint8_t* dst = out.v_codes + ((size_t)(g * 2 + kt) * 32 + lane) * (BITS * 8);
#pragma unroll
      for (int q = 0; q < kWords; q += 4)
        *reinterpret_cast<uint4*>(dst + 4 * q) = make_uint4(w[q], w[q + 1], w[q + 2], w[q + 3]);
    }
    // V params: lanes 0..15 tile 0, 16..31 tile 1; entry (j, group)
    {
      const int kt = lane >> 4, jj = (lane >> 2) & 3, grp = lane & 3;
      const int t0 = kt * 16 + 2 * jj;
      __half2 s01 = __halves2half2(sm.vs[t0][grp], sm.vs[t0 + 1][grp]);
      __half2 s89 = __halves2half2(sm.vs[t0 + 8][grp], sm.vs[t0 + 9][grp]);
      __half2 z01 = __halves2half2(sm.vz[t0][grp], sm.vz[t0 + 1][grp]);
      __half2 z89 = __halves2half2(sm.vz[t0 + 8][grp], sm.vz[t0 + 9][grp]);
      uint4 e = make_uint4(*reinterpret_cast<uint32_t*>(&s01), *reinterpret_cast<uint32_t*>(&s89),
                           *reinterpret_cast<uint32_t*>(&z01), *reinterpret_cast<uint32_t*>(&z89));
      *reinterpret_cast<uint4*>(out.v_params + (size_t)(g * 2 + kt) * 256 + (grp * 4 + jj) * 16) = e;
    }
  }
  __syncwarp();
  return okv;
}

}  // namespace uc
