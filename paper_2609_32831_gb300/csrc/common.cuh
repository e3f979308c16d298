// Device helpers shared by the UniCache kernels: status word, bounded
// mbarrier waits, TMA / bulk-copy issue, ldmatrix and mma.sync wrappers.
// Everything here is inline PTX written for sm_103a.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <stdint.h>

#include "../../include/unicache.h"

namespace uc {

constexpr int kHeadDim = UC_HEAD_DIM;
constexpr int kGroup = UC_GROUP;

// ----------------------------------------------------------------- status
// The first 16 bytes of every workspace: {code, detail, spare, spare}.
struct DevStatus {
  int32_t code;
  int32_t detail;
  int32_t spare[2];
};

__device__ __forceinline__ void set_status(DevStatus* st, int code, int detail) {
  if (st == nullptr) return;
  if (atomicCAS(&st->code, 0, code) == 0) atomicExch(&st->detail, detail);
}

__device__ __forceinline__ uint64_t global_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Bounded waits give up after this many nanoseconds and report
// UC_ERR_TIMEOUT; a healthy wait in these kernels lasts microseconds.
constexpr uint64_t kWaitLimitNs = 2000000000ull;

// ---------------------------------------------------------------- mbarrier
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count));
}

__device__ __forceinline__ void fence_barrier_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n"
      ".reg .pred p;\n"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      "selp.u32 %0, 1, 0, p;\n"
      "}\n"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Waits for the phase with `parity` to complete. Returns false (and records
// UC_ERR_TIMEOUT with `where`) if it did not complete within `limit_ns`.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, DevStatus* st, int where,
                                          uint64_t limit_ns = kWaitLimitNs) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_ns();
  for (uint32_t it = 0;; ++it) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((it & 15u) == 15u && global_ns() - t0 > limit_ns) {
      set_status(st, UC_ERR_TIMEOUT, where);
      return false;
    }
  }
}

// ------------------------------------------- programmatic dependent launch
// Launched with programmatic stream serialisation, a kernel may start while
// the kernel before it in the stream is still finishing. griddep_wait blocks
// until that kernel has completed and its writes are visible (a no-op for an
// ordinary launch); griddep_launch_dependents lets the next kernel start.
__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void griddep_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// ------------------------------------------------------------ TMA / bulk
__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, int c0, int c1,
                                            uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(smem_u32(bar))
      : "memory");
}

// Contiguous copy: dst, src 16-byte aligned, bytes a multiple of 16.
__device__ __forceinline__ void bulk_load(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}

// Order this thread's earlier generic-proxy global accesses (an acquire of
// data other CTAs wrote) before its later bulk copies from global memory.
__device__ __forceinline__ void fence_proxy_async_global() {
  asm volatile("fence.proxy.async.global;" ::: "memory");
}

// Make generic-proxy shared-memory writes visible to the async proxy (TMA,
// tensor cores) before the barrier that hands the data over.
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void prefetch_tmap(const CUtensorMap* map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}

// ------------------------------------------------------- ldmatrix / mma
__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                        uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                          uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

// Transpose of an 8x8 b16 matrix held one 32-bit pair per lane.
__device__ __forceinline__ uint32_t movmatrix_t(uint32_t a) {
  uint32_t d;
  asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(d) : "r"(a));
  return d;
}

// D += A * B, m16n8k16, bf16 inputs, fp32 accumulate.
__device__ __forceinline__ void mma_bf16(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                         uint32_t b1) {
  asm(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// D += A * B, m16n8k16, fp16 inputs, fp32 accumulate.
__device__ __forceinline__ void mma_f16(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                        uint32_t b1) {
  asm(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

__device__ __forceinline__ uint32_t pack_h2(__half lo, __half hi) {
  __half2 v = __halves2half2(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

__device__ __forceinline__ uint32_t pack_f16(float lo, float hi) {
  __half2 v = __floats2half2_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

// Extract two codes (bit offsets `shift` and 16 + `shift`) as the fp16 pair
// (1024 + a, 1024 + b), then subtract 1024 exactly: returns half2(a, b).
template <int MASK>
__device__ __forceinline__ uint32_t codes_to_h2(uint32_t w, int shift) {
  uint32_t x;
  const uint32_t m = (uint32_t)MASK | ((uint32_t)MASK << 16);
  asm("lop3.b32 %0, %1, %2, %3, 0xea;" : "=r"(x) : "r"(w >> shift), "r"(m), "r"(0x64006400u));
  __half2 h = *reinterpret_cast<__half2*>(&x);
  const __half2 magic = __halves2half2(__ushort_as_half(0x6400), __ushort_as_half(0x6400));
  h = __hsub2(h, magic);
  return *reinterpret_cast<uint32_t*>(&h);
}

// Codes of width W at bit offset B (1 <= B, B + W <= 10) of both 16-bit
// halves of w, as exact fp16 values code - C with C = (2^W - 1) / 2 (codes
// centred on their range): OR-ing the exponent 25 - B gives 2^(10-B) + code
// (the code lands in the mantissa with unit weight), and 2^(10-B) + C is
// itself exact because C is a multiple of 2^-1 >= 2^-B. Two instructions per
// pair of codes.
template <int W, int B>
__device__ __forceinline__ uint32_t codes_centred_h2(uint32_t w) {
  static_assert(B >= 1 && B + W <= 10, "code must sit in the fp16 mantissa above bit 0");
  constexpr uint32_t mask = ((1u << W) - 1u) << B;
  constexpr uint32_t expo = (uint32_t)(25 - B) << 10;
  // 2^(10-B) + C in fp16: exponent 25 - B, mantissa C * 2^B
  constexpr uint32_t sub = expo | (uint32_t)(((1u << W) - 1u) << (B - 1));
  uint32_t x;
  asm("lop3.b32 %0, %1, %2, %3, 0xea;" : "=r"(x) : "r"(w), "r"(mask | (mask << 16)), "r"(expo | (expo << 16)));
  const __half m = __ushort_as_half((unsigned short)sub);
  __half2 h = __hsub2(*reinterpret_cast<__half2*>(&x), __halves2half2(m, m));
  return *reinterpret_cast<uint32_t*>(&h);
}

// Shifted copies of a packed code word so that every pair of codes sits at
// a bit offset between 1 and 10 - BITS.
struct CodeWord {
  uint32_t lo;  // word << 1
  uint32_t mid; // word
  uint32_t hi;  // word >> 9 (int2) or >> 7 (int4)
};

template <int BITS>
__device__ __forceinline__ CodeWord code_word(uint32_t w) {
  return CodeWord{w << 1, w, BITS == 2 ? (w >> 9) : (w >> 7)};
}

// Pair p of a packed code word (codes at bit offsets p*BITS and 16 + p*BITS)
// as exact centred fp16 values.
template <int BITS, int P>
__device__ __forceinline__ uint32_t code_pair(const CodeWord& c) {
  if constexpr (BITS == 2) {
    if constexpr (P == 0)
      return codes_centred_h2<2, 1>(c.lo);
    else if constexpr (P < 5)
      return codes_centred_h2<2, 2 * P>(c.mid);
    else
      return codes_centred_h2<2, 2 * (P - 5) + 1>(c.hi);
  } else {
    if constexpr (P == 0)
      return codes_centred_h2<4, 1>(c.lo);
    else if constexpr (P == 1)
      return codes_centred_h2<4, 4>(c.mid);
    else
      return codes_centred_h2<4, 4 * (P - 2) + 1>(c.hi);
  }
}

// 2^x with the hardware approximation (flushes subnormal results to 0).
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint32_t hmul2_u32(uint32_t a, uint32_t b) {
  __half2 r = __hmul2(*reinterpret_cast<__half2*>(&a), *reinterpret_cast<__half2*>(&b));
  return *reinterpret_cast<uint32_t*>(&r);
}

__device__ __forceinline__ uint32_t hfma2_u32(uint32_t a, uint32_t b, uint32_t c) {
  __half2 r = __hfma2(*reinterpret_cast<__half2*>(&a), *reinterpret_cast<__half2*>(&b),
                      *reinterpret_cast<__half2*>(&c));
  return *reinterpret_cast<uint32_t*>(&r);
}

// a * b - c (the negation is an operand modifier of the fused multiply-add)
__device__ __forceinline__ uint32_t hfms2_u32(uint32_t a, uint32_t b, uint32_t c) {
  __half2 r = __hfma2(*reinterpret_cast<__half2*>(&a), *reinterpret_cast<__half2*>(&b),
                      __hneg2(*reinterpret_cast<__half2*>(&c)));
  return *reinterpret_cast<uint32_t*>(&r);
}

}  // namespace uc
