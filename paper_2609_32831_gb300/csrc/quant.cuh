// Group quantization of one run of 32 kept tokens, by one warp, into the
// fragment-ordered packed layout declared in unicache.h.
//
// Keys are quantized per channel over the 32 tokens, values per token over
// each run of 32 channels (App. E storage; constants from the measured
// workloads). Every step is IEEE fp32 round-to-nearest-even:
//   s = fp16((max - min) / qmax + 0), z = fp16(min + 0) (a zero scale or
//   minimum is stored as +0, whichever signed zeros the searches return),
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

// Per-warp shared scratch: for keys per channel, for values per (token,
// channel group), the zero-point and reciprocal scale in fp32 (fast path)
// and the fp16 scale (exact path and parameter stores).
struct __align__(16) QuantStats {
  float2 zr[128];
  __half s[128];
};

// code = clamp(rint(fl(t / s)), 0, qmax) with t = fl(x - z) and fl() IEEE
// round-to-nearest. The quotient is first formed as t * fl(1 / s), which is
// within 1.5 * 2^-23 |t / s| of fl(t / s); its rounding to an integer can
// only differ from that of fl(t / s) when it lies within that distance of a
// half-integer, and only then is the correctly rounded division taken.
// Quotients clamp outside [0, qmax], so only |q| <= qmax + 1 needs care.
//
// q_code_fast returns the code from t * fl(1 / s) and sets `bit` in `near`
// when the quotient lies within 4e-6 (qmax + 2) >= 4e-6 max(1, |q|) of a
// half-integer (one bound for the whole clamp range: quotients beyond it
// clamp to qmax whichever way they round, and a spurious hit only costs one
// exact recomputation). Such elements are redone one at a time with
// q_code_exact. On bf16 inputs they are not rare (about 7 in 10^4: the
// quotient of two short bf16 differences often lands on a half-integer), so
// the redo is per element, never per lane or warp.
//
// Rounding adds 1.5 * 2^23: for |q| < 2^22 the sum is 1.5 * 2^23 + rint(q)
// (round half to even), its bits kQBase + rint(q); beyond, the bits still
// order like q, so clamping them as signed integers to [kQBase, kQBase +
// qmax] gives kQBase + code for every finite or infinite q. The fast path
// returns that biased code; a word of biased fields is corrected once by
// subtracting kQBase times the sum of its fields' place values (mod 2^32).
constexpr float kQMagic = 12582912.0f;  // 1.5 * 2^23
constexpr int kQBase = 0x4B400000;      // bits of kQMagic

// kQBase * (sum of 2^(BITS f) over the 32 / BITS fields of a word), mod 2^32
template <int BITS>
__host__ __device__ constexpr uint32_t word_bias() {
  return (uint32_t)(((uint64_t)(uint32_t)kQBase * (0xffffffffull / ((1ull << BITS) - 1ull))) & 0xffffffffull);
}

//
// The quotient is monotone in x (each step rounds a monotone function), so a
// group whose minimum and maximum round into [0, qmax] (group_params checks
// them) needs no clamp at all: CLAMP = false skips it for a warp whose
// groups all pass, the common case.
template <int BITS, bool CLAMP = true>
__device__ __forceinline__ uint32_t q_code_fast(float x, float z, float inv_s, uint32_t& near, uint32_t bit) {
  constexpr int qmax = (1 << BITS) - 1;
  constexpr float kEdge = 0.5f - 4e-6f * (float)((1u << BITS) + 1u);
  const float t = __fsub_rn(x, z);
  const float q = __fmul_rn(t, inv_s);
  const float y = __fadd_rn(q, kQMagic);
  const float r = __fsub_rn(y, kQMagic);  // rint(q) for |q| < 2^22; |q - r| <= 1/2 is exact
  if (fabsf(__fsub_rn(q, r)) >= kEdge) near |= bit;
  if constexpr (CLAMP) return (uint32_t)min(max(__float_as_int(y), kQBase), kQBase + qmax);
  return (uint32_t)__float_as_int(y);
}

template <int BITS>
__device__ __forceinline__ uint32_t q_code_exact(float x, float z, float s) {
  constexpr uint32_t qmax = (1u << BITS) - 1u;
  if (s == 0.0f) return 0u;
  return min(__float2uint_rn(__fdiv_rn(__fsub_rn(x, z), s)), qmax);
}

// The correction of one element the fast path coded: its field of word q
// (runtime) of w, at `shift`, moves from the fast code to the exact one.
template <int BITS, int N>
__device__ __forceinline__ void fix_code(uint32_t (&w)[N], int q, int shift, float x, float z, float inv_s,
                                         float s) {
  uint32_t unused = 0;
  const uint32_t fast = q_code_fast<BITS>(x, z, inv_s, unused, 0u) - (uint32_t)kQBase;
  const uint32_t delta = (q_code_exact<BITS>(x, z, s) - fast) << shift;  // mod 2^32
#pragma unroll
  for (int k = 0; k < N; ++k)
    if (k == q) w[k] += delta;
}

__device__ __forceinline__ bool half_finite(__half h) {
  return (__half_as_ushort(h) & 0x7c00u) != 0x7c00u;
}

__device__ __forceinline__ __nv_bfloat162 as_bf2(uint32_t w) { return *reinterpret_cast<__nv_bfloat162*>(&w); }

// Scale and zero-point of one group from its minimum and maximum (a NaN in
// either, an infinite input or an fp16 overflow clears ok). Zeros are stored
// as +0 whichever signed zero the searches returned.
template <int BITS>
__device__ __forceinline__ void group_params(float mn, float mx, int e, QuantStats& st, bool& ok, bool& inrange) {
  constexpr float qmax = (float)((1 << BITS) - 1);
  const __half s16 = __float2half_rn(__fadd_rn(__fdiv_rn(__fsub_rn(mx, mn), qmax), 0.0f));
  const __half z16 = __float2half_rn(__fadd_rn(mn, 0.0f));
  ok = ok && half_finite(s16) && half_finite(z16);
  const float sf = __half2float(s16), zf = __half2float(z16);
  const float rf = sf != 0.0f ? __frcp_rn(sf) : 0.0f;  // s == 0: codes 0
  st.zr[e] = make_float2(zf, rf);
  st.s[e] = s16;
  // the fast codes of the group's extremes, unclamped, inside [0, qmax]?
  uint32_t unused = 0;
  const int lo = (int)q_code_fast<BITS, false>(mn, zf, rf, unused, 0u) - kQBase;
  const int hi = (int)q_code_fast<BITS, false>(mx, zf, rf, unused, 0u) - kQBase;
  inrange = inrange && lo >= 0 && hi <= (1 << BITS) - 1;
}

// One parameter entry of the fragment-ordered layout: scales of elements
// (e0, e1) and (e8, e9), zero-points of the same.
__device__ __forceinline__ uint4 param_entry(const QuantStats& st, int e0, int e1, int e8, int e9) {
  const __half2 s01 = __halves2half2(st.s[e0], st.s[e1]);
  const __half2 s89 = __halves2half2(st.s[e8], st.s[e9]);
  const __half2 z01 = __floats2half2_rn(st.zr[e0].x, st.zr[e1].x);  // exact: the zr were fp16
  const __half2 z89 = __floats2half2_rn(st.zr[e8].x, st.zr[e9].x);
  return make_uint4(*reinterpret_cast<const uint32_t*>(&s01), *reinterpret_cast<const uint32_t*>(&s89),
                    *reinterpret_cast<const uint32_t*>(&z01), *reinterpret_cast<const uint32_t*>(&z89));
}

// Codes of tile nt (tokens 8 nt .. 8 nt + 7) of one lane's key elements in
// fragment order: token 8 nt + n, channels 16 i + 2 j + 8 sub + {0, 1}; word
// q holds channels 16 i + 2 j + 8 sub, +1 of blocks i = q * 8 / BITS .. at
// bits BITS p and 16 + BITS p, p = 2 (i mod (8 / BITS)) + sub.
template <int BITS, bool CLAMP, typename RowK>
__device__ __forceinline__ void key_tile_codes(RowK krow, const QuantStats& st, int nt, uint32_t (&w)[BITS]) {
  const int lane = threadIdx.x & 31;
  const int n = lane >> 2, j = lane & 3;
  constexpr int kb = 8 / BITS;  // 16-channel blocks per word
  const __nv_bfloat16* row = krow(8 * nt + n);
  uint32_t near = 0;  // bit 4 i + e: element e (c, c + 1, c + 8, c + 9) of block i
#pragma unroll
  for (int q = 0; q < BITS; ++q) w[q] = 0u;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int c = 16 * i + 2 * j;
    const float4 a = *reinterpret_cast<const float4*>(&st.zr[c]);      // z, 1/s of c, c + 1
    const float4 b = *reinterpret_cast<const float4*>(&st.zr[c + 8]);  // of c + 8, c + 9
    const uint32_t x01 = *reinterpret_cast<const uint32_t*>(row + c);
    const uint32_t x89 = *reinterpret_cast<const uint32_t*>(row + c + 8);
    const int q = i / kb, p = 2 * (i % kb);
    w[q] += (q_code_fast<BITS, CLAMP>(bf16_lo(x01), a.x, a.y, near, 1u << (4 * i)) << (BITS * p)) +
            (q_code_fast<BITS, CLAMP>(bf16_hi(x01), a.z, a.w, near, 1u << (4 * i + 1)) << (16 + BITS * p)) +
            (q_code_fast<BITS, CLAMP>(bf16_lo(x89), b.x, b.y, near, 1u << (4 * i + 2)) << (BITS * (p + 1))) +
            (q_code_fast<BITS, CLAMP>(bf16_hi(x89), b.z, b.w, near, 1u << (4 * i + 3)) << (16 + BITS * (p + 1)));
  }
#pragma unroll
  for (int q = 0; q < BITS; ++q) w[q] -= word_bias<BITS>();
  while (__any_sync(0xffffffffu, near != 0)) {
    if (near != 0) {
      const int bit = __ffs(near) - 1;
      near &= near - 1u;
      const int i = bit >> 2, e = bit & 3;
      const int c = 16 * i + 2 * j + (e & 1) + 8 * (e >> 1);
      fix_code<BITS>(w, i / kb, BITS * (2 * (i % kb) + (e >> 1)) + 16 * (e & 1), __bfloat162float(row[c]),
                     st.zr[c].x, st.zr[c].y, __half2float(st.s[c]));
    }
  }
}

// Keys of group g (tokens 32 g .. 32 g + 31): per channel over the 32 tokens.
// Row t is read from krow(t) (bf16, 128 channels). Returns false in every
// lane (nothing written) if a value is not finite or a parameter overflows
// fp16.
template <int BITS, typename RowK>
__device__ bool quantize_keys(RowK krow, int g, const QuantOut& out, QuantStats& st) {
  const int lane = threadIdx.x & 31;
  // ---- parameters: lane owns channels 4 lane .. 4 lane + 3
  bool ok = true, inrange = true;
  {
    const uint2 v0 = *reinterpret_cast<const uint2*>(krow(0) + 4 * lane);
    __nv_bfloat162 mn0 = as_bf2(v0.x), mn1 = as_bf2(v0.y), mx0 = mn0, mx1 = mn1;
#pragma unroll 8
    for (int t = 1; t < 32; ++t) {
      const uint2 v = *reinterpret_cast<const uint2*>(krow(t) + 4 * lane);
      mn0 = __hmin2_nan(mn0, as_bf2(v.x));
      mx0 = __hmax2_nan(mx0, as_bf2(v.x));
      mn1 = __hmin2_nan(mn1, as_bf2(v.y));
      mx1 = __hmax2_nan(mx1, as_bf2(v.y));
    }
    group_params<BITS>(__low2float(mn0), __low2float(mx0), 4 * lane + 0, st, ok, inrange);
    group_params<BITS>(__high2float(mn0), __high2float(mx0), 4 * lane + 1, st, ok, inrange);
    group_params<BITS>(__low2float(mn1), __low2float(mx1), 4 * lane + 2, st, ok, inrange);
    group_params<BITS>(__high2float(mn1), __high2float(mx1), 4 * lane + 3, st, ok, inrange);
  }
  ok = __all_sync(0xffffffffu, ok);
  const bool clamp = !__all_sync(0xffffffffu, inrange);
  __syncwarp();
  if (!ok) return false;
  // ---- codes in fragment order, one 8-token tile at a time
#pragma unroll 1
  for (int nt = 0; nt < 4; ++nt) {
    uint32_t w[BITS];
    if (clamp)
      key_tile_codes<BITS, true>(krow, st, nt, w);
    else
      key_tile_codes<BITS, false>(krow, st, nt, w);
    uint8_t* dst = out.k_codes + ((size_t)(g * 4 + nt) * 32 + lane) * (BITS * 4);
    if constexpr (BITS == 4)
      *reinterpret_cast<uint4*>(dst) = make_uint4(w[0], w[1], w[BITS > 2 ? 2 : 0], w[BITS > 3 ? 3 : 0]);
    else
      *reinterpret_cast<uint2*>(dst) = make_uint2(w[0], w[1]);
  }
  // ---- parameters: lane -> entry (jj = lane / 8, i = lane % 8) of channels
  // c0 = 16 i + 2 jj, c0 + 1, c0 + 8, c0 + 9
  {
    const int jj = lane >> 3, i = lane & 7;
    const int c0 = 16 * i + 2 * jj;
    *reinterpret_cast<uint4*>(out.k_params + (size_t)g * 512 + (i * 4 + jj) * 16) =
        param_entry(st, c0, c0 + 1, c0 + 8, c0 + 9);
  }
  __syncwarp();
  return true;
}

// Codes of one lane's value elements in fragment order: tile kt of 16
// tokens, tokens 16 kt + 2 j + 8 sub + {0, 1}, channels 8 m + gq; word q of
// tile kt holds channels of blocks m = q * 8 / BITS .. at bits BITS p
// (token 2 j + 8 sub) and 16 + BITS p (the next token), p = 2 (m mod
// (8 / BITS)) + sub.
template <int BITS, bool CLAMP, typename RowV>
__device__ __forceinline__ void value_codes(RowV vrow, const QuantStats& st, uint32_t (&w)[2][2 * BITS]) {
  const int lane = threadIdx.x & 31;
  const int gq = lane >> 2, j = lane & 3;
  constexpr int kb = 8 / BITS;  // 8-channel blocks per word
#pragma unroll
  for (int kt = 0; kt < 2; ++kt)
#pragma unroll
    for (int q = 0; q < 2 * BITS; ++q) w[kt][q] = 0u;
#pragma unroll 1
  for (int sh = 0; sh < 4; ++sh) {  // sh = 2 sub + h: token 2 j + 8 sub + h of each tile
    const int sub = sh >> 1, h = sh & 1;
    const int shift0 = 16 * h + BITS * sub;
    uint32_t near = 0;  // bit 16 kt + m
#pragma unroll
    for (int kt = 0; kt < 2; ++kt) {
      const int t = 16 * kt + 2 * j + 8 * sub + h;
      const __nv_bfloat16* row = vrow(t);
#pragma unroll
      for (int gi = 0; gi < 4; ++gi) {
        const float2 zr = st.zr[4 * t + gi];
#pragma unroll
        for (int mm = 0; mm < 4; ++mm) {
          const int m = 4 * gi + mm;
          const float x = __uint_as_float((uint32_t)(*reinterpret_cast<const uint16_t*>(row + 8 * m + gq)) << 16);
          const uint32_t code = q_code_fast<BITS, CLAMP>(x, zr.x, zr.y, near, 1u << (16 * kt + m));
          w[kt][m / kb] += code << (shift0 + 2 * BITS * (m % kb));
        }
      }
    }
    while (__any_sync(0xffffffffu, near != 0)) {
      if (near != 0) {
        const int bit = __ffs(near) - 1;
        near &= near - 1u;
        const int kt = bit >> 4, m = bit & 15;
        const int t = 16 * kt + 2 * j + 8 * sub + h, e = 4 * t + (m >> 2);
        const float x = __bfloat162float(vrow(t)[8 * m + gq]);
        const float sf = __half2float(st.s[e]);
        const int shift = shift0 + 2 * BITS * (m % kb);
        if (kt == 0)
          fix_code<BITS>(w[0], m / kb, shift, x, st.zr[e].x, st.zr[e].y, sf);
        else
          fix_code<BITS>(w[1], m / kb, shift, x, st.zr[e].x, st.zr[e].y, sf);
      }
    }
  }
#pragma unroll
  for (int kt = 0; kt < 2; ++kt)
#pragma unroll
    for (int q = 0; q < 2 * BITS; ++q) w[kt][q] -= word_bias<BITS>();
}

// Values of group g: per token over each run of 32 channels. Row t is read
// from vrow(t). Returns false in every lane (nothing written) if a value is
// not finite or a parameter overflows fp16.
template <int BITS, typename RowV>
__device__ bool quantize_values(RowV vrow, int g, const QuantOut& out, QuantStats& st) {
  const int lane = threadIdx.x & 31;
  // ---- parameters: lane owns token `lane`, all four channel groups
  bool ok = true, inrange = true;
  {
    const __nv_bfloat16* row = vrow(lane);
#pragma unroll
    for (int gi = 0; gi < 4; ++gi) {
      uint4 c[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) c[k] = *reinterpret_cast<const uint4*>(row + 32 * gi + 8 * k);
      __nv_bfloat162 mn[4], mx[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        mn[k] = __hmin2_nan(__hmin2_nan(as_bf2(c[k].x), as_bf2(c[k].y)), __hmin2_nan(as_bf2(c[k].z), as_bf2(c[k].w)));
        mx[k] = __hmax2_nan(__hmax2_nan(as_bf2(c[k].x), as_bf2(c[k].y)), __hmax2_nan(as_bf2(c[k].z), as_bf2(c[k].w)));
      }
      const __nv_bfloat162 mn2 = __hmin2_nan(__hmin2_nan(mn[0], mn[1]), __hmin2_nan(mn[2], mn[3]));
      const __nv_bfloat162 mx2 = __hmax2_nan(__hmax2_nan(mx[0], mx[1]), __hmax2_nan(mx[2], mx[3]));
      const float mnf = __bfloat162float(__hmin_nan(__low2bfloat16(mn2), __high2bfloat16(mn2)));
      const float mxf = __bfloat162float(__hmax_nan(__low2bfloat16(mx2), __high2bfloat16(mx2)));
      group_params<BITS>(mnf, mxf, 4 * lane + gi, st, ok, inrange);
    }
  }
  ok = __all_sync(0xffffffffu, ok);
  const bool clamp = !__all_sync(0xffffffffu, inrange);
  __syncwarp();
  if (!ok) return false;
  uint32_t w[2][2 * BITS];
  if (clamp)
    value_codes<BITS, true>(vrow, st, w);
  else
    value_codes<BITS, false>(vrow, st, w);
#pragma unroll
  for (int kt = 0; kt < 2; ++kt) {
    uint8_t* dst = out.v_codes + ((size_t)(g * 2 + kt) * 32 + lane) * (BITS * 8);
#pragma unroll
    for (int q = 0; q < 2 * BITS; q += 4)
      *reinterpret_cast<uint4*>(dst + 4 * q) = make_uint4(w[kt][q], w[kt][q + 1], w[kt][q + 2], w[kt][q + 3]);
  }
  // ---- parameters: lanes 0..15 tile 0, 16..31 tile 1; entry (jj, group):
  // tokens t0 = 16 kt + 2 jj, t0 + 1, t0 + 8, t0 + 9 of channel group grp
  {
    const int kt = lane >> 4, jj = (lane >> 2) & 3, grp = lane & 3;
    const int t0 = kt * 16 + 2 * jj;
    *reinterpret_cast<uint4*>(out.v_params + (size_t)(g * 2 + kt) * 256 + (grp * 4 + jj) * 16) =
        param_entry(st, 4 * t0 + grp, 4 * (t0 + 1) + grp, 4 * (t0 + 8) + grp, 4 * (t0 + 9) + grp);
  }
  __syncwarp();
  return true;
}

// Keys then values of group g (the scratch is reused between them).
template <int BITS, typename RowK, typename RowV>
__device__ bool quantize_group_warp(RowK krow, RowV vrow, int g, const QuantOut& out, QuantStats& st) {
  if (!quantize_keys<BITS>(krow, g, out, st)) return false;
  return quantize_values<BITS>(vrow, g, out, st);
}

}  // namespace uc
