// Fused dequant-and-gather decode attention over heterogeneous segments
// (App. E "Attention over heterogeneous cache segments": one shared softmax
// across segments, chunks merged by log-sum-exp; Eq. 1's per-segment mass as
// a by-product).
//
// Design (GB300, HBM-bound): persistent CTAs walk a static list of work
// items; an item is one chunk of 64-token tiles of one segment of one
// (sequence, KV head). Per CTA one producer warp streams tiles into a
// 2- or 3-stage shared-memory ring (TMA 2D loads with 128-byte swizzle for bf16
// rows, 1D bulk copies for packed codes and parameters) and four consumer
// warps compute with mma.sync m16n8k16:
//   bf16 rows:  S = Q K^T in bf16 (exact products), P split into bf16 hi + lo
//               parts so P V keeps ~16 mantissa bits;
//   packed:     each pair of codes -> an exact fp16 pair 2^(10-B) + code with
//               one LOP3 (magic-number trick; the offset is removed exactly
//               by small extra MMAs), scales folded into the queries (keys)
//               and the probabilities (values), S and P V in fp16 with fp32
//               accumulation.
// Each item leaves an unnormalised partial (O, m, l); the last CTA to finish
// a (sequence, KV head) merges its items by log-sum-exp, writes O, lse and
// the per-segment probability mass, and re-arms the counter.
#include <mutex>

#include "common.cuh"
#include "internal.h"

namespace uc {

constexpr int kTileTok = 64;
constexpr int kMaxStages = 3;
// Ring stages: one query n-tile runs 3 CTAs per SM with 2 stages each (the
// register budget is 128), larger calls 1 CTA per SM with 3.
template <int NTW>
__host__ __device__ constexpr int stages_for() { return NTW == 1 ? 2 : 3; }
template <int NTW>
__host__ __device__ constexpr int ctas_for() { return NTW == 1 ? 3 : 1; }
constexpr int kConsumers = 4;
constexpr int kAttnThreads = 32 * (kConsumers + 1);
constexpr int kSlotBytes = 32768;
constexpr float kNegInf = -INFINITY;
constexpr float kLn2 = 0.69314718055994530942f;

// slot layout of a packed tile: up to 8 int2 or 4 int4 quantization groups
// (codes 1 KB / 2 KB per group for K and for V, parameters 512 B per group)
constexpr int kSlotKParams = 8192;
constexpr int kSlotVCodes = 12288;
constexpr int kSlotVParams = 20480;

__host__ __device__ constexpr int quant_groups_per_tile(int bits) { return bits == 2 ? 8 : 4; }

constexpr int kMaxItemsPerBh = 64;
constexpr int kMaxPendingMerges = 64;
constexpr int kItemQ = 2;  // items handed from the producer to the consumers ahead

struct AttnSmem {
  float merge_w[kMaxItemsPerBh * 8];  // per (item, row of an 8-row block): m, then weight
  float merge_l[kMaxItemsPerBh * 8];
  uint64_t full[kMaxStages];
  uint64_t empty[kMaxStages];
  uint64_t item_full[kItemQ];   // producer -> consumers: item position and its query rows
  uint64_t item_empty[kItemQ];  // consumers -> producer: the entry is free again
  int item_pos[kItemQ];         // processing position, -1: no more work
  int n_pending;                    // (sequence, KV head) merges this CTA owes
  int pending[kMaxPendingMerges];
  alignas(1024) uint8_t slot[kMaxStages][kSlotBytes];  // only stages_for<NTW>() are allocated
};

// Query fragments of the current item live in shared memory (2 KB per
// n-tile of 8 query rows): for one n-tile in the merge staging arrays, which
// are idle while an item runs (merges happen between items), keeping three
// CTAs per SM; for up to eight n-tiles after the ring.
template <int NTW>
__host__ __device__ constexpr int qfrag_tiles() { return NTW == 1 ? 0 : 8; }

// bf16 query rows of one item as copied by the producer (g * T rows)
template <int NTW>
__host__ __device__ constexpr int qrow_bytes() { return NTW == 1 ? 8 * 256 : 64 * 256; }

template <int NTW>
__host__ __device__ constexpr size_t attend_smem_bytes() {
  return offsetof(AttnSmem, slot) + (size_t)stages_for<NTW>() * kSlotBytes + (size_t)qfrag_tiles<NTW>() * 2048 +
         (size_t)kItemQ * qrow_bytes<NTW>() + 1024;
}

// Shared-memory regions after the ring: query fragments (NTW > 1), then the
// producer's query-row buffers.
template <int NTW>
__device__ __forceinline__ uint8_t* after_ring(AttnSmem& sm) {
  return reinterpret_cast<uint8_t*>(sm.slot) + stages_for<NTW>() * kSlotBytes;
}
template <int NTW>
__device__ __forceinline__ uint8_t* qrows_buf(AttnSmem& sm, int k) {
  return after_ring<NTW>(sm) + qfrag_tiles<NTW>() * 2048 + k * qrow_bytes<NTW>();
}

__host__ __device__ size_t attend_part_floats(int ntiles) { return (size_t)ntiles * 8 * (kHeadDim + 2); }

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
  const int tg = quant_groups_per_tile(sd.bits);
  *qtiles = (ng + tg - 1) / tg;
  return *qtiles + ((n % kGroup) ? 1 : 0);
}

struct ItemInfo {
  int bh, b, s, tb, te, qtiles, n;
  bool tail;  // the bf16 residual tail of a packed segment
};

// Item at processing position pos; *it receives its partial-output index.
__device__ __forceinline__ ItemInfo decode_item(const AttnParams& p, int pos, int* it) {
  ItemInfo r;
  const int nbh = p.batch * p.n_kv_heads;
  int local;
  if (pos < p.n_heavy * nbh) {
    r.bh = pos / p.n_heavy;
    local = p.heavy_local[pos % p.n_heavy];
  } else {
    const int q = pos - p.n_heavy * nbh;
    r.bh = q / p.n_light;
    local = p.light_local[q % p.n_light];
  }
  *it = r.bh * p.items_per_bh + local;
  r.b = r.bh / p.n_kv_heads;
  r.s = 0;
  for (int s = 0; s < p.nseg; ++s)
    if (local >= p.seg[s].chunk_begin) r.s = s;
  const SegDev& sd = p.seg[r.s];
  const int c = local - sd.chunk_begin;
  r.n = sd.n_kept[r.b];
  const int nt = seg_tiles(sd, r.n, &r.qtiles);
  r.tail = false;
  if (seg_is_bf16(sd.kind)) {
    r.tb = (int)(((int64_t)c * nt) / sd.n_chunks);
    r.te = (int)(((int64_t)(c + 1) * nt) / sd.n_chunks);
  } else if (c == sd.n_chunks - 1) {  // last chunk: the tail tile (empty if no tail)
    r.tail = true;
    r.tb = r.qtiles;
    r.te = nt;
  } else {
    const int cq = sd.n_chunks - 1;
    r.tb = (int)(((int64_t)c * r.qtiles) / cq);
    r.te = (int)(((int64_t)(c + 1) * r.qtiles) / cq);
  }
  return r;
}

// Work lists. OneCall walks the items of one call; ManyCalls walks several
// calls' items in one launch, the heavy items of every call first, then the
// light tail items. locate() maps a processing position to its call's
// parameters and to the position inside that call's own order.
struct OneCall {
  const AttnParams& p;
  __device__ int n_items() const { return p.n_items; }
  __device__ int n_calls() const { return 1; }
  __device__ const AttnParams& call(int) const { return p; }
  __device__ int items_per_bh(int) const { return p.items_per_bh; }
  __device__ const AttnParams& locate(int pos, int* local, int* c) const {
    *local = pos;
    *c = 0;
    return p;
  }
};

struct ManyCalls {
  const MultiAttnParams& m;
  __device__ int n_items() const { return m.n_items; }
  __device__ int n_calls() const { return m.n_calls; }
  __device__ const AttnParams& call(int c) const { return m.call[c]; }
  __device__ int items_per_bh(int c) const { return m.call[c].items_per_bh; }
  __device__ const AttnParams& locate(int pos, int* local, int* c) const {
    const int nh = m.heavy_begin[m.n_calls];
    int k = 0;
    if (pos < nh) {
      while (k + 1 < m.n_calls && pos >= m.heavy_begin[k + 1]) ++k;
      *local = pos - m.heavy_begin[k];
    } else {
      const int q = pos - nh;
      while (k + 1 < m.n_calls && q >= m.light_begin[k + 1]) ++k;
      const AttnParams& p = m.call[k];
      *local = p.n_heavy * p.batch * p.n_kv_heads + (q - m.light_begin[k]);
    }
    *c = k;
    return m.call[k];
  }
};

template <class P>
struct WorkOf;
template <>
struct WorkOf<AttnParams> {
  using type = OneCall;
};
template <>
struct WorkOf<MultiAttnParams> {
  using type = ManyCalls;
};

__device__ __forceinline__ void consumer_sync() { asm volatile("bar.sync 1, 128;" ::: "memory"); }

// Arrival on a (sequence, KV head) counter, acquire-release at GPU scope:
// after a CTA barrier, the partial outputs every consumer thread wrote are
// ordered before the increment (release is cumulative over the barrier), and
// the arrival that completes the count has acquired every earlier one, so
// the CTA that merges needs no further fence (a later CTA barrier carries the
// acquire to its other threads).
__device__ __forceinline__ int counter_arrive_acq_rel(int* c) {
  int prev;
  asm volatile("atom.add.acq_rel.gpu.global.s32 %0, [%1], 1;" : "=r"(prev) : "l"(c) : "memory");
  return prev;
}

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
// Items come from a launch-wide counter (the next position to process, in
// the plan's order: heavy items first), so a CTA that finishes early takes
// more. The producer claims its next position once it has issued every tile
// of the current item (the ring still holds work for the consumers, which
// hides the atomic's latency, and no CTA claims work long before it can
// start it), hands each position to the consumers through a two-entry queue
// and copies the item's query rows (the g * T rows of one KV head are
// contiguous) along with it.
template <int NTW, class W>
__device__ void produce(const W& w, AttnSmem& sm) {
  constexpr int ST = stages_for<NTW>();
  const AttnParams& p0 = w.call(0);
  int* sched = p0.sched;
  uint32_t seq = 0;
  bool stop = false;
  // the first item of every CTA is its own index (the grid never exceeds
  // the item count); later items come from the launch-wide counter, so the
  // first copies are issued without waiting for an atomic's round trip
  int pos = blockIdx.x;
  for (uint32_t iseq = 0;; ++iseq) {
    const int k = iseq % kItemQ;
    if (iseq >= kItemQ && !mbar_wait(&sm.item_empty[k], ((iseq / kItemQ) - 1) & 1, p0.status, 12, p0.wait_ns))
      break;
    if (pos >= w.n_items()) {
      sm.item_pos[k] = -1;
      mbar_arrive(&sm.item_full[k]);
      break;
    }
    int it, local, c;
    const AttnParams& p = w.locate(pos, &local, &c);
    const ItemInfo ii = decode_item(p, local, &it);
    const SegDev& sd = p.seg[ii.s];
    sm.item_pos[k] = pos;
    const uint32_t qbytes = (uint32_t)p.rows * kHeadDim * 2;
    const __nv_bfloat16* qsrc =
        p.q + (size_t)(ii.b * p.n_q_heads + (ii.bh % p.n_kv_heads) * p.group) * p.n_qtok * kHeadDim;
    mbar_arrive_expect_tx(&sm.item_full[k], qbytes);
    bulk_load(qrows_buf<NTW>(sm, k), qsrc, qbytes, &sm.item_full[k]);
    for (int t = ii.tb; t < ii.te; ++t, ++seq) {
      const int slot = seq % ST;
      if (seq >= ST && !mbar_wait(&sm.empty[slot], ((seq / ST) - 1) & 1, p.status, 10, p.wait_ns)) {
        stop = true;
        break;
      }
      if (pos == p.withhold_pos && t == ii.tb) continue;  // test hook: this tile is never copied
      uint8_t* dst = sm.slot[slot];
      const bool tail = ii.tail;
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
        const int tg = quant_groups_per_tile(sd.bits);
        const int g0 = tg * t;
        const int ngt = min(tg, ng - g0);
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
    if (stop) break;
    pos = (int)gridDim.x + atomicAdd(sched, 1);
  }
  // This producer claims nothing more: the last producer of the launch to
  // get here re-arms the work queue for the next launch. Done here rather
  // than at the CTA's exit, so that the fence and the atomic stay off the
  // path of the consumers' final merges.
  __threadfence();
  if (atomicAdd(sched + 1, 1) == (int)gridDim.x - 1) {
    sched[0] = 0;
    sched[1] = 0;
  }
  // A consumer that gave up on a bounded wait (the status word is set) no
  // longer waits for the copies this producer issued: they land before the
  // CTA leaves. (Otherwise the consumers have waited for every one.)
  const bool failed = stop || (p0.status != nullptr && *reinterpret_cast<volatile int32_t*>(&p0.status->code) != 0);
  for (int s = 0; failed && s < ST; ++s) {
    if (seq < (uint32_t)s + 1u) break;
    const uint32_t sq = seq - 1u - (uint32_t)s;
    if (!mbar_wait(&sm.full[sq % ST], (sq / ST) & 1, p0.status, 15, p0.wait_ns)) break;
  }
}

// ------------------------------------------------------------- consumer
//
// Transposed formulation: with T query tokens the g = Hq / Hkv heads of one
// KV head give 7T query rows, far fewer than the 16 rows of an m16n8k16 A
// operand. Keys therefore take the M role and query rows the N role:
//   S^T [keys x rows]    = K [keys x d] . Q^T [d x rows]
//   O^T [d x rows]      += V^T [d x keys] . P^T [keys x rows]
// An n8 tile of query rows per MMA wastes at most one row for T = 1. P^T
// moves from the accumulator layout into the B-operand layout with one
// movmatrix.trans per 8 x 8 block.
//
// Per thread (g = lane / 4, j = lane % 4), n-tile nt of query rows:
//   Q^T  B fragment: rows nt*8 + g, channels {16i + 2j, +1} and {+8, +9}
//   S^T  accumulator: keys {g, g + 8} x rows nt*8 + {2j, 2j + 1}
//   O^T  accumulator: channels {16mt + g, 16mt + 8 + g} x rows nt*8 + {2j, 2j + 1}

template <int NTW>
struct WarpState {
  float o[NTW][8][4];
  float z[NTW][4];  // packed values: zero-point term per channel group (rows = groups 0..3)
  float m[NTW][2];  // running max per query row (rows 2j, 2j + 1 of each n-tile), log2 units
  float l[NTW][2];  // this thread's share of the row sums
};

template <int NTW>
__device__ __forceinline__ void state_init(WarpState<NTW>& st) {
#pragma unroll
  for (int nt = 0; nt < NTW; ++nt) {
#pragma unroll
    for (int mt = 0; mt < 8; ++mt) st.o[nt][mt][0] = st.o[nt][mt][1] = st.o[nt][mt][2] = st.o[nt][mt][3] = 0.f;
    st.z[nt][0] = st.z[nt][1] = st.z[nt][2] = st.z[nt][3] = 0.f;
    st.m[nt][0] = st.m[nt][1] = kNegInf;
    st.l[nt][0] = st.l[nt][1] = 0.f;
  }
}

// Online softmax over NB 16-key blocks: x[blk][nt][e] (e: 0/1 key g, 2/3 key
// g+8; e & 1 selects the row), in log2 units. Writes probabilities into pr.
// The reference max m moves only when a row's max exceeds it by more than
// 8, so P = 2^(x - m) <= 2^8 (exact enough in fp16 / bf16 pairs) and o, z, l
// are rescaled only on those (rare) moves. Each lane first tests its own
// logits against m + 8; the row maxima (shuffle reductions) are formed only
// when some lane's test fires.
template <int NTW, int NB>
__device__ __forceinline__ void softmax_rows(WarpState<NTW>& st, const float (&x)[NB][NTW][4],
                                             float (&pr)[NB][NTW][4]) {
#pragma unroll
  for (int nt = 0; nt < NTW; ++nt) {
    bool over = false;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const float lim = st.m[nt][h] + 8.f;
#pragma unroll
      for (int k = 0; k < NB; ++k) over |= (x[k][nt][h] > lim) | (x[k][nt][2 + h] > lim);
    }
    if (__any_sync(0xffffffffu, over)) {
      float mx[2];
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        float v = fmaxf(x[0][nt][h], x[0][nt][2 + h]);
#pragma unroll
        for (int k = 1; k < NB; ++k) v = fmaxf(v, fmaxf(x[k][nt][h], x[k][nt][2 + h]));
        v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, 4));
        v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, 8));
        v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, 16));
        mx[h] = v;
      }
      const bool g0 = mx[0] > st.m[nt][0] + 8.f, g1 = mx[1] > st.m[nt][1] + 8.f;
      float alpha[2];
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const bool gh = h ? g1 : g0;
        const float nm = gh ? mx[h] : st.m[nt][h];
        alpha[h] = (st.m[nt][h] == kNegInf) ? 0.f : ex2_approx(st.m[nt][h] - nm);
        st.m[nt][h] = nm;
        st.l[nt][h] *= alpha[h];
      }
#pragma unroll
      for (int mt = 0; mt < 8; ++mt) {
        st.o[nt][mt][0] *= alpha[0];
        st.o[nt][mt][1] *= alpha[1];
        st.o[nt][mt][2] *= alpha[0];
        st.o[nt][mt][3] *= alpha[1];
      }
      st.z[nt][0] *= alpha[0];
      st.z[nt][1] *= alpha[1];
      st.z[nt][2] *= alpha[0];
      st.z[nt][3] *= alpha[1];
    }
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const float um = (st.m[nt][h] == kNegInf) ? 0.f : st.m[nt][h];
      float sum = 0.f;
#pragma unroll
      for (int k = 0; k < NB; ++k) {
        pr[k][nt][h] = ex2_approx(x[k][nt][h] - um);
        pr[k][nt][2 + h] = ex2_approx(x[k][nt][2 + h] - um);
        sum += pr[k][nt][h] + pr[k][nt][2 + h];
      }
      st.l[nt][h] += sum;
    }
  }
}

__device__ __forceinline__ uint32_t swz(uint32_t base, int key, int chunk) {
  return base + (chunk >> 3) * 8192 + key * 128 + ((((chunk & 7) ^ (key & 7))) << 4);
}

// One 16-key block (keys 16u .. 16u + 15 of a bf16 tile).
template <int NTW>
__device__ __forceinline__ void block_bf16(WarpState<NTW>& st, uint32_t qs,
                                           uint32_t kbase, int u, int valid, float scale) {
  const int lane = threadIdx.x & 31;
  const int mi = lane >> 3, rr = lane & 7, g = lane >> 2;
  float s[NTW][4];
#pragma unroll
  for (int nt = 0; nt < NTW; ++nt) s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.f;
  {
    const int kk = 16 * u + 8 * (mi & 1) + rr;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      uint32_t a[4];
      ldsm_x4(swz(kbase, kk, 2 * i + (mi >> 1)), a[0], a[1], a[2], a[3]);
#pragma unroll
      for (int nt = 0; nt < NTW; ++nt) {
        const uint2 qv = lds64(qs + ((nt * 8 + i) * 32 + lane) * 8);
        mma_bf16(s[nt], a, qv.x, qv.y);
      }
    }
  }
  float x[1][NTW][4], pr[1][NTW][4];
  const bool ok0 = 16 * u + g < valid, ok1 = 16 * u + 8 + g < valid;
#pragma unroll
  for (int nt = 0; nt < NTW; ++nt) {
    x[0][nt][0] = ok0 ? s[nt][0] * scale : kNegInf;
    x[0][nt][1] = ok0 ? s[nt][1] * scale : kNegInf;
    x[0][nt][2] = ok1 ? s[nt][2] * scale : kNegInf;
    x[0][nt][3] = ok1 ? s[nt][3] * scale : kNegInf;
  }
  softmax_rows<NTW, 1>(st, x, pr);
  // P^T as B fragments (bf16 hi + lo parts)
  uint32_t bh[NTW][2], bl[NTW][2];
#pragma unroll
  for (int nt = 0; nt < NTW; ++nt) {
#pragma unroll
    for (int half = 0; half < 2; ++half) {
      const float p0 = pr[0][nt][2 * half], p1 = pr[0][nt][2 * half + 1];
      const uint32_t hi = pack_bf16(p0, p1);
      const uint32_t lo = pack_bf16(p0 - bf16_lo(hi), p1 - bf16_hi(hi));
      bh[nt][half] = movmatrix_t(hi);
      bl[nt][half] = movmatrix_t(lo);
    }
  }
  const uint32_t vbase = kbase + 16384;
  const int vk = 16 * u + 8 * (mi >> 1) + rr;
#pragma unroll
  for (int mt = 0; mt < 8; ++mt) {
    uint32_t a[4];
    ldsm_x4_t(swz(vbase, vk, 2 * mt + (mi & 1)), a[0], a[1], a[2], a[3]);
#pragma unroll
    for (int nt = 0; nt < NTW; ++nt) {
      mma_bf16(st.o[nt][mt], a, bh[nt][0], bh[nt][1]);
      mma_bf16(st.o[nt][mt], a, bl[nt][0], bl[nt][1]);
    }
  }
}

// ---- packed codes
//
// A code word holds 16 int2 or 8 int4 codes as pairs: pair p is the code at
// bit p * BITS of the low half and the one at the same bit of the high half.
// One LOP3 turns a pair into the exact fp16 pair (2^(10-B) + a, 2^(10-B) + b)
// when both codes sit at mantissa bit B (OR-ing exponent 25 - B). Shifted
// copies of the word bring every pair to such a bit:
//   int2  L = w << 6, M = w, R = w >> 6:  p0 L@6, p1 L@8, p2 M@4, p3 M@6,
//                                         p4 M@8, p5 R@4, p6 R@6, p7 R@8
//   int4  L = w << 4, M = w, R = w >> 4, R2 = w >> 8: p0..p3 at bit 4
// (bits that a shift moves across the half boundary fall outside the masks).
// The offset 2^(10-B) (64, 16 or 4) is removed exactly by extra MMAs with
// fp16 powers of two, so no rounded zero-point absorbs it.
template <int BITS>
struct Words {
  uint32_t l, m, r, r2;
};

template <int BITS>
__device__ __forceinline__ Words<BITS> words(uint32_t w) {
  if constexpr (BITS == 2)
    return Words<BITS>{w << 6, w, w >> 6, 0u};
  else
    return Words<BITS>{w << 4, w, w >> 4, w >> 8};
}

template <int BITS, int P>
struct PairAt {
  // bit of the pair in its source copy and the offset 2^(10 - bit)
  static constexpr int kBit = BITS == 4 ? 4 : (P % 3 == 2 ? 4 : (P % 3 == 0 ? 6 : 8));
  static constexpr int kOff = 1 << (10 - kBit);
};

template <int BITS, int P>
__device__ __forceinline__ uint32_t pair_h2(const Words<BITS>& c) {
  constexpr int B = PairAt<BITS, P>::kBit;
  constexpr uint32_t qmax = (1u << BITS) - 1u;
  constexpr uint32_t mask = (qmax << B) | (qmax << (B + 16));
  constexpr uint32_t expo = ((uint32_t)(25 - B) << 10) | ((uint32_t)(25 - B) << 26);
  uint32_t src;
  if constexpr (BITS == 2)
    src = P < 2 ? c.l : (P < 5 ? c.m : c.r);
  else
    src = P == 0 ? c.l : (P == 1 ? c.m : (P == 2 ? c.r : c.r2));
  uint32_t x;
  asm("lop3.b32 %0, %1, %2, %3, 0xea;" : "=r"(x) : "r"(src), "n"(mask), "n"(expo));
  return x;
}

// The same pair centred: (a - C, b - C) with C = qmax / 2, exact (one more
// HSUB2 of 2^(10-B) + C). Used for values, whose accumulator sums thousands
// of tokens: uncentred values would carry off * sum(s p) next to the signal.
template <int BITS, int P>
__device__ __forceinline__ uint32_t pair_centred_h2(const Words<BITS>& c) {
  constexpr int B = PairAt<BITS, P>::kBit;
  // 2^(10-B) + C in fp16: exponent 25 - B, mantissa C * 2^B (C = qmax / 2)
  constexpr uint32_t sub = ((uint32_t)(25 - B) << 10) | (((1u << BITS) - 1u) << (B - 1));
  const uint32_t x = pair_h2<BITS, P>(c);
  const __half m = __ushort_as_half((unsigned short)sub);
  __half2 h = __hsub2(*reinterpret_cast<const __half2*>(&x), __halves2half2(m, m));
  return *reinterpret_cast<uint32_t*>(&h);
}

// -offset of pair P as an fp16 pair (a power of two, exact)
template <int BITS, int P>
__device__ __forceinline__ constexpr uint32_t neg_off_h2() {
  constexpr int off = PairAt<BITS, P>::kOff;
  // -2^k in fp16: sign 1, exponent k + 15, mantissa 0
  constexpr uint32_t h = 0x8000u | ((uint32_t)((off == 64 ? 6 : (off == 16 ? 4 : 2)) + 15) << 10);
  return h | (h << 16);
}

// Row of the beta MMA that collects s . q for the channels of pair P:
// offset 64 -> row 1, 16 -> row 2, 4 -> row 3.
template <int BITS>
__host__ __device__ constexpr int off_row(int p) {
  return BITS == 4 ? 1 : (p % 3 == 2 ? 1 : (p % 3 == 0 ? 2 : 3));
}
template <int BITS>
__host__ __device__ constexpr int off_of_row(int r) {
  return BITS == 4 ? (r == 1 ? 64 : 0) : (r == 1 ? 64 : (r == 2 ? 16 : 4));
}

// One quantization group (32 keys = two 16-key blocks) of a packed tile.
// With codes entering as c + off (off per pair position, see above) and
// x_hat = c * s + z:
//   S^T  = (c + off)_K . (s_K (.) Q)^T + beta,
//          beta = z_K . Q^T - sum_off off * (s_K . Q^T over that offset's channels)
//          (one MMA per 16 channels: A rows z, s|off=64, s|off=16, s|off=4, all
//          against the unscaled query: exact fp16 products, fp32 sums)
//   O^T += (c - C)_V^T . (s_V (.) P^T) + z'_V^T . P^T,  C = qmax / 2,
//          z' = fp16(z + C s)  (centred values: their accumulator sums
//          thousands of tokens, so no offset may ride along)
// The per-channel key scales fold into the queries as fp16 hi + lo parts (the
// scaled query keeps ~22 bits) and the per-token value scales into the
// probabilities.
// beta of two groups of one tile with one set of MMAs: A rows 0..3 hold
// group a's (z, s over the channels of the offsets 64, 16, 4), rows 4..7
// group b's, against the unscaled query. bt[h][nt] = beta of group h for
// query rows 2j, 2j + 1 of n-tile nt.
template <int NTW, int BITS>
__device__ __forceinline__ void group_beta_pair(uint32_t qsm, uint32_t base, int ga, int gb,
                                                float (&bt)[2][NTW][2]) {
  const int lane = threadIdx.x & 31;
  const int g = lane >> 2, j = lane & 3, gg = g & 3;
  float bq[NTW][4];
#pragma unroll
  for (int nt = 0; nt < NTW; ++nt) bq[nt][0] = bq[nt][1] = bq[nt][2] = bq[nt][3] = 0.f;
  const uint32_t kp = base + kSlotKParams + (g < 4 ? ga : gb) * 512 + j * 16;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const uint4 P = lds128(kp + i * 64);  // s(c0 c1), s(c8 c9), z(c0 c1), z(c8 c9)
    const int p0 = BITS == 4 ? 2 * (i & 1) : 2 * (i & 3);
    const int r0 = off_row<BITS>(p0), r1 = off_row<BITS>(p0 + 1);
    const uint32_t az[4] = {gg == 0 ? P.z : (gg == r0 ? P.x : 0u), 0u, gg == 0 ? P.w : (gg == r1 ? P.y : 0u), 0u};
#pragma unroll
    for (int nt = 0; nt < NTW; ++nt) {
      const uint2 qv = lds64(qsm + ((nt * 8 + i) * 32 + lane) * 8);
      mma_f16(bq[nt], az, qv.x, qv.y);
    }
  }
#pragma unroll
  for (int nt = 0; nt < NTW; ++nt)
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      // row r of group h sits in lanes 4 (4h + r) + j
      float b0 = __shfl_sync(0xffffffffu, bq[nt][0], 16 * h + j);
      float b1 = __shfl_sync(0xffffffffu, bq[nt][1], 16 * h + j);
#pragma unroll
      for (int r = 1; r < 4; ++r) {
        const float w = -(float)off_of_row<BITS>(r);
        if (w != 0.f) {
          b0 = fmaf(w, __shfl_sync(0xffffffffu, bq[nt][0], 16 * h + 4 * r + j), b0);
          b1 = fmaf(w, __shfl_sync(0xffffffffu, bq[nt][1], 16 * h + 4 * r + j), b1);
        }
      }
      bt[h][nt][0] = b0;
      bt[h][nt][1] = b1;
    }
}

// kBeta = false: the group's beta comes in bt_in (from group_beta_pair)
// instead of its own MMAs.
template <int NTW, int BITS, bool kBeta = true>
__device__ __forceinline__ void group_quant(WarpState<NTW>& st, uint32_t qsm,
                                            uint32_t base, int gl, float scale,
                                            const float (&bt_in)[NTW][2]) {
  const int lane = threadIdx.x & 31;
  const int g = lane >> 2, j = lane & 3;
  constexpr int KW = BITS == 4 ? 4 : 2;  // code words per lane per 8-token tile
  const __half hc = __float2half_rn(0.5f * (float)((1 << BITS) - 1));
  const uint32_t vc_c = pack_h2(hc, hc);  // C = qmax / 2

  // ---- per 16 channels: scaled queries (fp16 hi + lo), beta, and S of both
  // 16-key blocks (four independent MMA chains; beta is added at the end)
  // beta rows: 0: z . q, 1..3: s . q over the channels whose pairs carry the
  // offset 64, 16, 4 (exact fp16 products, fp32 sums); beta = row 0 - 64 row 1
  // - 16 row 2 - 4 row 3 is formed in fp32 afterwards.
  float bq[NTW][4];
  float sa[2][NTW][4], sl[2][NTW][4];
#pragma unroll
  for (int nt = 0; nt < NTW; ++nt)
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      bq[nt][e] = 0.f;
      sa[0][nt][e] = sa[1][nt][e] = sl[0][nt][e] = sl[1][nt][e] = 0.f;
    }
  // key code words of the 8-token tiles 4 gl + t (t = 0..3: keys g, g + 8 of
  // block 0, then of block 1)
  uint32_t kw[4][KW];
#pragma unroll
  for (int t = 0; t < 4; ++t) {
    const uint32_t a = base + ((4 * gl + t) * 32 + lane) * (BITS * 4);
    if constexpr (BITS == 4) {
      const uint4 v = lds128(a);
      kw[t][0] = v.x;
      kw[t][1] = v.y;
      kw[t][KW > 2 ? 2 : 0] = v.z;
      kw[t][KW > 3 ? 3 : 1] = v.w;
    } else {
      const uint2 v = lds64(a);
      kw[t][0] = v.x;
      kw[t][1] = v.y;
    }
  }
  const uint32_t kp = base + kSlotKParams + gl * 512 + j * 16;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const uint4 P = lds128(kp + i * 64);  // s(c0 c1), s(c8 c9), z(c0 c1), z(c8 c9)
    // offset rows of the pairs of channels (16i + 2j, +1) and (16i + 2j + 8, +9)
    const int p0 = BITS == 4 ? 2 * (i & 1) : 2 * (i & 3);
    const int r0 = off_row<BITS>(p0), r1 = off_row<BITS>(p0 + 1);
    const uint32_t az[4] = {kBeta ? (g == 0 ? P.z : (g == r0 ? P.x : 0u)) : 0u, 0u,
                            kBeta ? (g == 0 ? P.w : (g == r1 ? P.y : 0u)) : 0u, 0u};
    // A fragments of both blocks for channels 16 i .. 16 i + 15
    uint32_t af[2][4];
    const int q = BITS == 4 ? (i >> 1) : (i >> 2);
#pragma unroll
    for (int blk = 0; blk < 2; ++blk) {
      const Words<BITS> w0 = words<BITS>(kw[2 * blk][q]), w1 = words<BITS>(kw[2 * blk + 1][q]);
      if constexpr (BITS == 4) {
        if ((i & 1) == 0) {
          af[blk][0] = pair_h2<4, 0>(w0); af[blk][1] = pair_h2<4, 0>(w1);
          af[blk][2] = pair_h2<4, 1>(w0); af[blk][3] = pair_h2<4, 1>(w1);
        } else {
          af[blk][0] = pair_h2<4, 2>(w0); af[blk][1] = pair_h2<4, 2>(w1);
          af[blk][2] = pair_h2<4, 3>(w0); af[blk][3] = pair_h2<4, 3>(w1);
        }
      } else {
        switch (i & 3) {
          case 0:
            af[blk][0] = pair_h2<2, 0>(w0); af[blk][1] = pair_h2<2, 0>(w1);
            af[blk][2] = pair_h2<2, 1>(w0); af[blk][3] = pair_h2<2, 1>(w1);
            break;
          case 1:
            af[blk][0] = pair_h2<2, 2>(w0); af[blk][1] = pair_h2<2, 2>(w1);
            af[blk][2] = pair_h2<2, 3>(w0); af[blk][3] = pair_h2<2, 3>(w1);
            break;
          case 2:
            af[blk][0] = pair_h2<2, 4>(w0); af[blk][1] = pair_h2<2, 4>(w1);
            af[blk][2] = pair_h2<2, 5>(w0); af[blk][3] = pair_h2<2, 5>(w1);
            break;
          default:
            af[blk][0] = pair_h2<2, 6>(w0); af[blk][1] = pair_h2<2, 6>(w1);
            af[blk][2] = pair_h2<2, 7>(w0); af[blk][3] = pair_h2<2, 7>(w1);
            break;
        }
      }
    }
#pragma unroll
    for (int nt = 0; nt < NTW; ++nt) {
      const uint2 qv = lds64(qsm + ((nt * 8 + i) * 32 + lane) * 8);
      const uint32_t qs0 = hmul2_u32(qv.x, P.x);
      const uint32_t qs1 = hmul2_u32(qv.y, P.y);
      const uint32_t ql0 = hfms2_u32(qv.x, P.x, qs0);
      const uint32_t ql1 = hfms2_u32(qv.y, P.y, qs1);
      if constexpr (kBeta) mma_f16(bq[nt], az, qv.x, qv.y);
#pragma unroll
      for (int blk = 0; blk < 2; ++blk) {
        mma_f16(sa[blk][nt], af[blk], qs0, qs1);
        mma_f16(sl[blk][nt], af[blk], ql0, ql1);
      }
    }
  }
  float x[2][NTW][4];
#pragma unroll
  for (int nt = 0; nt < NTW; ++nt) {
    float bt0 = bt_in[nt][0], bt1 = bt_in[nt][1];
    if constexpr (kBeta) {
      // rows 0..3 of bq sit in lanes (0..3, j)
      bt0 = __shfl_sync(0xffffffffu, bq[nt][0], j);
      bt1 = __shfl_sync(0xffffffffu, bq[nt][1], j);
#pragma unroll
      for (int r = 1; r < 4; ++r) {
        const float w = -(float)off_of_row<BITS>(r);
        if (w != 0.f) {
          bt0 = fmaf(w, __shfl_sync(0xffffffffu, bq[nt][0], 4 * r + j), bt0);
          bt1 = fmaf(w, __shfl_sync(0xffffffffu, bq[nt][1], 4 * r + j), bt1);
        }
      }
    }
#pragma unroll
    for (int blk = 0; blk < 2; ++blk) {
      x[blk][nt][0] = ((sa[blk][nt][0] + sl[blk][nt][0]) + bt0) * scale;
      x[blk][nt][1] = ((sa[blk][nt][1] + sl[blk][nt][1]) + bt1) * scale;
      x[blk][nt][2] = ((sa[blk][nt][2] + sl[blk][nt][2]) + bt0) * scale;
      x[blk][nt][3] = ((sa[blk][nt][3] + sl[blk][nt][3]) + bt1) * scale;
    }
  }

  // ---- softmax over the group's 32 keys
  float pr[2][NTW][4];
  softmax_rows<NTW, 2>(st, x, pr);

  // ---- P V for both blocks
#pragma unroll
  for (int blk = 0; blk < 2; ++blk) {
    const int u = 2 * gl + blk;
    uint32_t b[NTW][2];
#pragma unroll
    for (int nt = 0; nt < NTW; ++nt) {
      b[nt][0] = movmatrix_t(pack_f16(pr[blk][nt][0], pr[blk][nt][1]));
      b[nt][1] = movmatrix_t(pack_f16(pr[blk][nt][2], pr[blk][nt][3]));
    }
    // value parameters of this block's 16 tokens: scales of the 4 channel
    // groups, zero points of groups g / 4 and g / 4 + 2 (rows g and g + 8 of Z)
    const uint32_t vpa = base + kSlotVParams + u * 256 + j * 16;
    uint2 vs[4];
#pragma unroll
    for (int gi = 0; gi < 4; ++gi) vs[gi] = lds64(vpa + gi * 64);  // s(t0 t1), s(t8 t9)
    {
      // Z row gi (lanes g = gi < 4): z' = z + C s of group gi, one MMA
      const uint4 vg = lds128(vpa + (g & 3) * 64);                   // s(t0 t1), s(t8 t9), z(t0 t1), z(t8 t9)
      const uint32_t z0 = g < 4 ? hfma2_u32(vg.x, vc_c, vg.z) : 0u;
      const uint32_t z1 = g < 4 ? hfma2_u32(vg.y, vc_c, vg.w) : 0u;
      const uint32_t az[4] = {z0, 0u, z1, 0u};
#pragma unroll
      for (int nt = 0; nt < NTW; ++nt) mma_f16(st.z[nt], az, b[nt][0], b[nt][1]);
    }
    Words<BITS> vc[2 * KW];
    {
      const uint32_t va = base + kSlotVCodes + (u * 32 + lane) * (BITS * 8);
      const uint4 v0 = lds128(va);
      vc[0] = words<BITS>(v0.x);
      vc[1] = words<BITS>(v0.y);
      vc[2] = words<BITS>(v0.z);
      vc[3] = words<BITS>(v0.w);
      if constexpr (BITS == 4) {
        const uint4 v1 = lds128(va + 16);
        vc[2 * KW > 4 ? 4 : 0] = words<BITS>(v1.x);
        vc[2 * KW > 5 ? 5 : 1] = words<BITS>(v1.y);
        vc[2 * KW > 6 ? 6 : 2] = words<BITS>(v1.z);
        vc[2 * KW > 7 ? 7 : 3] = words<BITS>(v1.w);
      }
    }
#pragma unroll
    for (int gi = 0; gi < 4; ++gi) {
      uint32_t bs[NTW][2];
#pragma unroll
      for (int nt = 0; nt < NTW; ++nt) {
        bs[nt][0] = hmul2_u32(b[nt][0], vs[gi].x);
        bs[nt][1] = hmul2_u32(b[nt][1], vs[gi].y);
      }
#pragma unroll
      for (int mh = 0; mh < 2; ++mh) {
        const int mt = 2 * gi + mh;
        uint32_t a[4];
        // rows: channels 8m + g with m = 2 mt (a0, a2) and 2 mt + 1 (a1, a3);
        // a0 / a1 tokens 2j, 2j + 1 (pair p0), a2 / a3 tokens 2j + 8, 2j + 9 (p0 + 1)
        if constexpr (BITS == 4) {
          // m = 2mt + h: word m >> 1 = mt, p0 = 2 (m & 1) = 2h
          a[0] = pair_centred_h2<4, 0>(vc[mt]);
          a[2] = pair_centred_h2<4, 1>(vc[mt]);
          a[1] = pair_centred_h2<4, 2>(vc[mt]);
          a[3] = pair_centred_h2<4, 3>(vc[mt]);
        } else {
          // word m >> 2 = mt >> 1, p0 = 2 (m & 3) = 4 (mt & 1) + 2h
          const int q = mt >> 1;
          if ((mt & 1) == 0) {
            a[0] = pair_centred_h2<2, 0>(vc[q]);
            a[2] = pair_centred_h2<2, 1>(vc[q]);
            a[1] = pair_centred_h2<2, 2>(vc[q]);
            a[3] = pair_centred_h2<2, 3>(vc[q]);
          } else {
            a[0] = pair_centred_h2<2, 4>(vc[q]);
            a[2] = pair_centred_h2<2, 5>(vc[q]);
            a[1] = pair_centred_h2<2, 6>(vc[q]);
            a[3] = pair_centred_h2<2, 7>(vc[q]);
          }
        }
#pragma unroll
        for (int nt = 0; nt < NTW; ++nt) mma_f16(st.o[nt][mt], a, bs[nt][0], bs[nt][1]);
      }
    }
  }
}

// Zero the V rows [valid, 64) of a bf16 tile that lie in block u.
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

// Partial layout per item: [rows_pad][128] O (unnormalised), [rows_pad] m,
// [rows_pad] l, rows_pad = 8 * (number of n-tiles).
//
// The merge runs on the 128 consumer threads of the CTA that finished the
// last item of a (sequence, KV head), per block of 8 query rows: the
// log-sum-exp weights of every item (16 threads per row), then each thread
// (one output channel) sums the weighted partial outputs. After the CTA's
// last item the ring is idle (`seq` given) and the partials come through it
// by bulk copies continuing the consumers' tile sequence: for one n-tile and
// at most seven items per stage, the whole partials (O, m, l) in one round
// trip; otherwise (m, l) by loads and the 4 KB row blocks of O eight items
// per slot, copies issued ahead. Without `seq` (a merge between items) each
// thread loads the partial outputs, eight items at a time.
//
// Weights of the 8-row block r0: m_of(i, rr), l_of(i, rr) read item i's
// values; the normalised weights go to merge_l[i * 8 + rr]; lse and the
// per-segment mass are written for the block's nr valid rows.
template <class MOf, class LOf>
__device__ __forceinline__ void merge_weights(const AttnParams& p, float* wts, int b, int kvh, int r0,
                                              int nr, MOf m_of, LOf l_of, bool outputs = true) {
  const int tid = threadIdx.x;
  const int I = p.items_per_bh;
  const int rr = tid >> 4, part = tid & 15;
  float M = kNegInf;
  for (int i = part; i < I; i += 16) M = fmaxf(M, m_of(i, rr));
#pragma unroll
  for (int o = 8; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
  const float Mu = (M == kNegInf) ? 0.f : M;
  float L = 0.f;
  float Ls[UC_MAX_SEGMENTS];
#pragma unroll
  for (int q = 0; q < UC_MAX_SEGMENTS; ++q) Ls[q] = 0.f;
  for (int i = part; i < I; i += 16) {
    int sg = 0;
#pragma unroll
    for (int q = 1; q < UC_MAX_SEGMENTS; ++q) sg += (q < p.nseg && i >= p.seg[q].chunk_begin) ? 1 : 0;
    const float mi = m_of(i, rr);
    const float w = (mi == kNegInf) ? 0.f : exp2f(mi - Mu);
    const float lw = l_of(i, rr) * w;
    L += lw;
#pragma unroll
    for (int q = 0; q < UC_MAX_SEGMENTS; ++q)
      if (q == sg) Ls[q] += lw;
    wts[i * 8 + rr] = w;  // unnormalised weight
  }
#pragma unroll
  for (int o = 8; o > 0; o >>= 1) {
    L += __shfl_xor_sync(0xffffffffu, L, o);
#pragma unroll
    for (int q = 0; q < UC_MAX_SEGMENTS; ++q)
      if (q < p.nseg) Ls[q] += __shfl_xor_sync(0xffffffffu, Ls[q], o);
  }
  const float inv = (L > 0.f) ? 1.f / L : 0.f;
  for (int i = part; i < I; i += 16) wts[i * 8 + rr] *= inv;
  if (outputs && part == 0 && rr < nr) {
    const int r = r0 + rr;
    const int hl = r / p.n_qtok, t = r % p.n_qtok;
    const size_t orow = ((size_t)(b * p.n_q_heads + kvh * p.group + hl) * p.n_qtok + t);
    if (p.lse) p.lse[orow] = (L > 0.f) ? (M + log2f(L)) * kLn2 : kNegInf;
    if (p.mass)
      for (int q = 0; q < p.nseg; ++q) p.mass[orow * p.nseg + q] = Ls[q] * inv;
  }
}

__device__ __forceinline__ void merge_store(const AttnParams& p, int b, int kvh, int r0, int nr,
                                            const float (&acc)[8]) {
#pragma unroll
  for (int rr = 0; rr < 8; ++rr) {
    if (rr >= nr) continue;
    const int r = r0 + rr;
    const int hl = r / p.n_qtok, t = r % p.n_qtok;
    const size_t orow = ((size_t)(b * p.n_q_heads + kvh * p.group + hl) * p.n_qtok + t);
    p.out[orow * kHeadDim + threadIdx.x] = __float2bfloat16_rn(acc[rr]);
  }
}

template <int NTW>
__device__ void final_merge(const AttnParams& p, AttnSmem& sm, int bh, uint32_t* seq) {
  const int tid = threadIdx.x;  // 0..127 = channel
  const int b = bh / p.n_kv_heads, kvh = bh % p.n_kv_heads;
  const size_t pf = attend_part_floats(p.mtiles);
  const int rows_pad = 8 * p.mtiles;
  const int I = p.items_per_bh;
  const float* base = p.part + (size_t)bh * I * pf;
  constexpr int ST = stages_for<NTW>();

  // ---- one n-tile, few items: whole partials through the ring at once
  constexpr int kWholeFloats = 8 * (kHeadDim + 2);              // O, m, l of one n-tile
  constexpr int kWhole = kSlotBytes / (kWholeFloats * 4);       // items per slot (7)
  static_assert(NTW != 1 || kWhole * ST == kWholeMergeItems, "planner's whole-merge item limit");
  if (seq != nullptr && p.mtiles == 1 && I <= kWhole * ST) {
    const int nbw = (I + kWhole - 1) / kWhole;
    if (tid == 0) {
      // the partials were written by other CTAs (generic proxy) and acquired
      // at GPU scope; order that acquire before the copy engine's reads
      fence_proxy_async_global();
      for (int j = 0; j < nbw; ++j) {
        const uint32_t sq = *seq + j;
        uint64_t* bar = &sm.full[sq % ST];
        const int i0 = j * kWhole, cnt = min(kWhole, I - i0);
        mbar_arrive_expect_tx(bar, (uint32_t)(cnt * kWholeFloats * 4));
        for (int k = 0; k < cnt; ++k)
          bulk_load(sm.slot[sq % ST] + k * kWholeFloats * 4, base + (i0 + k) * pf, kWholeFloats * 4, bar);
      }
    }
    for (int j = 0; j < nbw; ++j) {
      const uint32_t sq = *seq + j;
      mbar_wait(&sm.full[sq % ST], (sq / ST) & 1, p.status, 14, p.wait_ns);
    }
    auto item = [&](int i) {
      return reinterpret_cast<const float*>(sm.slot[(*seq + i / kWhole) % ST]) + (i % kWhole) * kWholeFloats;
    };
    merge_weights(p, sm.merge_l, b, kvh, 0, p.rows, [&](int i, int rr) { return item(i)[8 * kHeadDim + rr]; },
                  [&](int i, int rr) { return item(i)[8 * kHeadDim + 8 + rr]; });
    consumer_sync();
    float acc[8];
#pragma unroll
    for (int rr = 0; rr < 8; ++rr) acc[rr] = 0.f;
    for (int i = 0; i < I; ++i) {
      const float* o = item(i);
#pragma unroll
      for (int rr = 0; rr < 8; ++rr) acc[rr] += sm.merge_l[i * 8 + rr] * o[rr * kHeadDim + tid];
    }
    merge_store(p, b, kvh, 0, p.rows, acc);
    consumer_sync();  // the slots are read before any later copy into them
    *seq += nbw;
    return;
  }

  constexpr int kPerSlot = kSlotBytes / (8 * kHeadDim * 4);  // 8-row blocks of O per ring slot
  const int nb = (I + kPerSlot - 1) / kPerSlot;
  auto issue = [&](int r0, int j) {  // batch j of the 8-row block r0 (thread 0)
    const uint32_t sq = *seq + j;
    uint64_t* bar = &sm.full[sq % ST];
    const int i0 = j * kPerSlot, cnt = min(kPerSlot, I - i0);
    mbar_arrive_expect_tx(bar, (uint32_t)cnt * 8 * kHeadDim * 4);
    for (int k = 0; k < cnt; ++k)
      bulk_load(sm.slot[sq % ST] + k * 8 * kHeadDim * 4, base + (i0 + k) * pf + (size_t)r0 * kHeadDim,
                8 * kHeadDim * 4, bar);
  };
  for (int r0 = 0; r0 < p.rows; r0 += 8) {
    const int nr = min(8, p.rows - r0);
    if (seq != nullptr && tid == 0) {
      fence_proxy_async_global();
      for (int j = 0; j < min(ST, nb); ++j) issue(r0, j);
    }
    for (int x = tid; x < I * 8; x += 128) {
      const int i = x >> 3, rr = x & 7;
      float m = kNegInf, l = 0.f;
      if (rr < nr) {
        m = __ldcg(base + i * pf + rows_pad * kHeadDim + r0 + rr);
        l = __ldcg(base + i * pf + rows_pad * kHeadDim + rows_pad + r0 + rr);
      }
      sm.merge_w[x] = m;
      sm.merge_l[x] = l;
    }
    consumer_sync();
    merge_weights(p, sm.merge_l, b, kvh, r0, nr, [&](int i, int rr) { return sm.merge_w[i * 8 + rr]; },
                  [&](int i, int rr) { return sm.merge_l[i * 8 + rr]; });
    consumer_sync();
    float acc[8];
#pragma unroll
    for (int rr = 0; rr < 8; ++rr) acc[rr] = 0.f;
    int i = 0;
    if (seq != nullptr) {
      for (int j = 0; j < nb; ++j) {
        const uint32_t sq = *seq + j;
        const bool ok = mbar_wait(&sm.full[sq % ST], (sq / ST) & 1, p.status, 14, p.wait_ns);
        const float* buf = reinterpret_cast<const float*>(sm.slot[sq % ST]);
        const int i0 = j * kPerSlot, cnt = min(kPerSlot, I - i0);
        if (ok) {
          for (int k = 0; k < cnt; ++k)
#pragma unroll
            for (int rr = 0; rr < 8; ++rr)
              acc[rr] += sm.merge_l[(i0 + k) * 8 + rr] * buf[(k * 8 + rr) * kHeadDim + tid];
        }
        consumer_sync();  // the slot is read: refill it
        if (tid == 0 && j + ST < nb) issue(r0, j + ST);
      }
      *seq += nb;
      i = I;
    }
    for (; i + 8 <= I; i += 8) {
      // eight items' loads in flight at once
      float v[8][8];
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const float* pi = base + (i + k) * pf + (size_t)r0 * kHeadDim + tid;
#pragma unroll
        for (int rr = 0; rr < 8; ++rr) v[k][rr] = (rr < nr) ? __ldcg(pi + rr * kHeadDim) : 0.f;
      }
#pragma unroll
      for (int k = 0; k < 8; ++k)
#pragma unroll
        for (int rr = 0; rr < 8; ++rr) acc[rr] += sm.merge_l[(i + k) * 8 + rr] * v[k][rr];
    }
    for (; i < I; ++i) {
      const float* pi = base + i * pf + (size_t)r0 * kHeadDim + tid;
      float v[8];
#pragma unroll
      for (int rr = 0; rr < 8; ++rr) v[rr] = (rr < nr) ? __ldcg(pi + rr * kHeadDim) : 0.f;
#pragma unroll
      for (int rr = 0; rr < 8; ++rr) acc[rr] += sm.merge_l[i * 8 + rr] * v[rr];
    }
    merge_store(p, b, kvh, r0, nr, acc);
    consumer_sync();
  }
}

// Split-K merge as a kernel of its own, for calls with many items per
// (sequence, KV head) (few long sequences): one CTA per (sequence, KV head,
// 8-row block, 32 output channels), so the partials of one (b, kvh) are read
// by several SMs at once instead of streaming through one. Eight warps take
// every eighth item each, all their loads in flight together; the warps'
// sums meet in shared memory. The attend launch before it leaves the
// partials and skips its own merges (`defer_merge`).
constexpr int kMergeChunks = kHeadDim / 32;
__global__ void __launch_bounds__(256) merge_partials_kernel(const __grid_constant__ AttnParams p) {
  __shared__ float s_m[kMaxItemsPerBh * 8], s_w[kMaxItemsPerBh * 8];
  __shared__ float s_red[8][8][33];
  griddep_wait();  // the attention launch whose partials this merges has completed
  griddep_launch_dependents();
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int rblocks = p.mtiles;
  const int ch = blockIdx.x % kMergeChunks;
  const int r0 = ((blockIdx.x / kMergeChunks) % rblocks) * 8;
  const int bh = blockIdx.x / (kMergeChunks * rblocks);
  const int b = bh / p.n_kv_heads, kvh = bh % p.n_kv_heads;
  const int nr = min(8, p.rows - r0);
  const size_t pf = attend_part_floats(p.mtiles);
  const int rows_pad = 8 * p.mtiles;
  const int I = p.items_per_bh;
  const float* base = p.part + (size_t)bh * I * pf;
  // every (item, row) pair's m and l: at most two pairs per thread
  for (int x = tid; x < I * 8; x += 256) {
    const int i = x >> 3, rr = x & 7;
    float m = kNegInf, l = 0.f;
    if (rr < nr) {
      m = __ldg(base + i * pf + rows_pad * kHeadDim + r0 + rr);
      l = __ldg(base + i * pf + rows_pad * kHeadDim + rows_pad + r0 + rr);
    }
    s_m[x] = m;
    s_w[x] = l;
  }
  __syncthreads();
  if (tid < 128)
    merge_weights(p, s_w, b, kvh, r0, nr, [&](int i, int rr) { return s_m[i * 8 + rr]; },
                  [&](int i, int rr) { return s_w[i * 8 + rr]; }, ch == 0);
  __syncthreads();
  const int c = ch * 32 + lane;
  float v[kMaxItemsPerBh / 8][8];
#pragma unroll
  for (int k = 0; k < kMaxItemsPerBh / 8; ++k) {
    const int i = warp + 8 * k;
#pragma unroll
    for (int rr = 0; rr < 8; ++rr)
      v[k][rr] = (i < I && rr < nr) ? __ldg(base + i * pf + (size_t)(r0 + rr) * kHeadDim + c) : 0.f;
  }
  float acc[8];
#pragma unroll
  for (int rr = 0; rr < 8; ++rr) acc[rr] = 0.f;
#pragma unroll
  for (int k = 0; k < kMaxItemsPerBh / 8; ++k) {
    const int i = warp + 8 * k;
    if (i < I)
#pragma unroll
      for (int rr = 0; rr < 8; ++rr) acc[rr] += s_w[i * 8 + rr] * v[k][rr];
  }
#pragma unroll
  for (int rr = 0; rr < 8; ++rr) s_red[warp][rr][lane] = acc[rr];
  __syncthreads();
  {
    const int rr = warp;  // 8 warps: one row each
    float sum = 0.f;
#pragma unroll
    for (int w = 0; w < 8; ++w) sum += s_red[w][rr][lane];
    if (rr < nr) {
      const int r = r0 + rr;
      const int hl = r / p.n_qtok, t = r % p.n_qtok;
      const size_t orow = ((size_t)(b * p.n_q_heads + kvh * p.group + hl) * p.n_qtok + t);
      p.out[orow * kHeadDim + c] = __float2bfloat16_rn(sum);
    }
  }
}

// Query rows of every n-tile as Q^T B fragments (bf16 for BF16, else fp16)
// in shared memory: word w of lane (g, j) for channels 16i + 2j (+8) of row
// 8 nt + g at [((nt * 8 + i) * 32 + lane) * 2 + w], from the bf16 rows the
// producer copied (row r = head * T + token). All consumer threads.
template <bool BF16>
__device__ __forceinline__ void store_q(const AttnParams& p, uint32_t* qf, const uint8_t* rows) {
  for (int x = threadIdx.x; x < p.mtiles * 512; x += 128) {
    const int nt = x >> 9, i = (x >> 6) & 7, ln = (x >> 1) & 31, w = x & 1;
    const int r = nt * 8 + (ln >> 2);
    const int c = 16 * i + 2 * (ln & 3) + 8 * w;
    uint32_t word = 0u;
    if (r < p.rows) {
      const uint32_t w0 = *reinterpret_cast<const uint32_t*>(rows + (r * kHeadDim + c) * 2);
      word = BF16 ? w0 : pack_f16(bf16_lo(w0), bf16_hi(w0));
    }
    qf[x] = word;
  }
}

// Merge the warps that share n-tiles (through the item's last slot), then
// write this item's partial.
template <int NTW>
__device__ __forceinline__ void finish_item(const AttnParams& p, AttnSmem& sm, WarpState<NTW>& st,
                                            int it, int last_slot, int NG, int KS, int grp, int ks) {
  const int lane = threadIdx.x & 31;
  const int g = lane >> 2, j = lane & 3;
  // zero-point term of packed values: channel group gi of query rows 2j,
  // 2j + 1 sits in lane (gi, j)
#pragma unroll
  for (int nt = 0; nt < NTW; ++nt)
#pragma unroll
    for (int gi = 0; gi < 4; ++gi) {
      const float z0 = __shfl_sync(0xffffffffu, st.z[nt][0], 4 * gi + j);
      const float z1 = __shfl_sync(0xffffffffu, st.z[nt][1], 4 * gi + j);
#pragma unroll
      for (int mh = 0; mh < 2; ++mh) {
        st.o[nt][2 * gi + mh][0] += z0;
        st.o[nt][2 * gi + mh][1] += z1;
        st.o[nt][2 * gi + mh][2] += z0;
        st.o[nt][2 * gi + mh][3] += z1;
      }
    }
  // full row sums: add the shares of the 8 key lanes (g)
#pragma unroll
  for (int nt = 0; nt < NTW; ++nt)
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      float v = st.l[nt][h];
      v += __shfl_xor_sync(0xffffffffu, v, 4);
      v += __shfl_xor_sync(0xffffffffu, v, 8);
      v += __shfl_xor_sync(0xffffffffu, v, 16);
      st.l[nt][h] = v;
    }
  constexpr int kVals = NTW * 36;
  if (KS > 1 && last_slot >= 0) {
    float* buf = reinterpret_cast<float*>(sm.slot[last_slot]);
    consumer_sync();
    for (int step = 1; step < KS; step *= 2) {
      const bool writer = (ks % (2 * step)) == step;
      const bool reader = (ks % (2 * step)) == 0;
      const int region = (ks / (2 * step)) * NG + grp;
      float* rb = buf + region * (kVals * 32);
      if (writer) {
#pragma unroll
        for (int nt = 0; nt < NTW; ++nt) {
#pragma unroll
          for (int mt = 0; mt < 8; ++mt)
#pragma unroll
            for (int e = 0; e < 4; ++e) rb[((nt * 36) + mt * 4 + e) * 32 + lane] = st.o[nt][mt][e];
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            rb[(nt * 36 + 32 + h) * 32 + lane] = st.m[nt][h];
            rb[(nt * 36 + 34 + h) * 32 + lane] = st.l[nt][h];
          }
        }
      }
      consumer_sync();
      if (reader) {
#pragma unroll
        for (int nt = 0; nt < NTW; ++nt) {
          float a[2], bb[2];
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            const float om = rb[(nt * 36 + 32 + h) * 32 + lane];
            const float ol = rb[(nt * 36 + 34 + h) * 32 + lane];
            const float nm = fmaxf(st.m[nt][h], om);
            const float um = (nm == kNegInf) ? 0.f : nm;
            a[h] = exp2f(st.m[nt][h] - um);
            bb[h] = exp2f(om - um);
            st.l[nt][h] = st.l[nt][h] * a[h] + ol * bb[h];
            st.m[nt][h] = nm;
          }
#pragma unroll
          for (int mt = 0; mt < 8; ++mt)
#pragma unroll
            for (int e = 0; e < 4; ++e)
              st.o[nt][mt][e] = st.o[nt][mt][e] * a[e & 1] + rb[(nt * 36 + mt * 4 + e) * 32 + lane] * bb[e & 1];
        }
      }
      consumer_sync();
    }
    fence_proxy_async();
    __syncwarp();
    if (lane == 0) mbar_arrive(&sm.empty[last_slot]);
  }
  if (ks == 0) {
    const size_t pf = attend_part_floats(p.mtiles);
    const int rows_pad = 8 * p.mtiles;
    float* pi = p.part + (size_t)it * pf;
#pragma unroll
    for (int nt = 0; nt < NTW; ++nt) {
      const int ntg = grp * NTW + nt;
      if (ntg >= p.mtiles) continue;
      const int r0 = ntg * 8 + 2 * j;
#pragma unroll
      for (int mt = 0; mt < 8; ++mt) {
        const int c0 = 16 * mt + g;
        pi[(r0) * kHeadDim + c0] = st.o[nt][mt][0];
        pi[(r0 + 1) * kHeadDim + c0] = st.o[nt][mt][1];
        pi[(r0) * kHeadDim + c0 + 8] = st.o[nt][mt][2];
        pi[(r0 + 1) * kHeadDim + c0 + 8] = st.o[nt][mt][3];
      }
      if (g == 0) {
        pi[rows_pad * kHeadDim + r0] = st.m[nt][0];
        pi[rows_pad * kHeadDim + r0 + 1] = st.m[nt][1];
        pi[rows_pad * kHeadDim + rows_pad + r0] = st.l[nt][0];
        pi[rows_pad * kHeadDim + rows_pad + r0 + 1] = st.l[nt][1];
      }
    }
  }
}

// All tiles of one item: bf16 rows (BITS = 16: bf16 segments and the tails
// of packed segments) or packed groups (BITS = 4 / 2).
template <int NTW, int BITS>
__device__ __forceinline__ void run_item(const AttnParams& p, AttnSmem& sm, const ItemInfo& ii, int it, int k,
                                         uint32_t& seq, bool& aborted, int NG, int KS, int grp, int ks) {
  const int lane = threadIdx.x & 31;
  uint32_t* qf = NTW == 1 ? reinterpret_cast<uint32_t*>(sm.merge_w)
                          : reinterpret_cast<uint32_t*>(after_ring<NTW>(sm));
  store_q<BITS == 16>(p, qf, qrows_buf<NTW>(sm, k));
  consumer_sync();
  if (lane == 0) mbar_arrive(&sm.item_empty[k]);  // the query rows are no longer needed
  const uint32_t qs = smem_u32(qf) + grp * NTW * 2048;
  WarpState<NTW> st;
  state_init<NTW>(st);
  int last_slot = -1;
  for (int t = ii.tb; t < ii.te; ++t, ++seq) {
    constexpr int ST = stages_for<NTW>();
    const int slot = seq % ST;
    if (!aborted && !mbar_wait(&sm.full[slot], (seq / ST) & 1, p.status, 11, p.wait_ns)) aborted = true;
    const uint32_t sbase = smem_u32(sm.slot[slot]);
    bool wrote = false;  // generic-proxy writes into the slot (zeroed V rows)
    if (!aborted) {
      if constexpr (BITS == 16) {
        const int valid = ii.tail ? (ii.n % kGroup) : min(kTileTok, ii.n - t * kTileTok);
        wrote = valid < kTileTok;
        for (int u = ks; u < 4; u += KS) {
          if (16 * u >= valid) continue;
          if (valid < 16 * u + 16) zero_v_rows(sm.slot[slot], u, valid);
          block_bf16<NTW>(st, qs, sbase, u, valid, p.scale_log2);
        }
      } else {
        constexpr int kTG = quant_groups_per_tile(BITS);
        const int ng = ii.n / kGroup;
        const int ngt = min(kTG, ng - kTG * t);  // quantization groups in this tile
        int gl = ks;
        if constexpr (NTW == 1 && BITS == 2) {
          // the warp's two groups of a full tile share one set of beta MMAs
          if (gl + KS < ngt) {
            float bt[2][NTW][2];
            group_beta_pair<NTW, BITS>(qs, sbase, gl, gl + KS, bt);
#pragma unroll 1
            for (int h = 0; h < 2; ++h, gl += KS) {
              float bh[NTW][2];
#pragma unroll
              for (int nt = 0; nt < NTW; ++nt) {
                bh[nt][0] = h ? bt[1][nt][0] : bt[0][nt][0];
                bh[nt][1] = h ? bt[1][nt][1] : bt[0][nt][1];
              }
              group_quant<NTW, BITS, false>(st, qs, sbase, gl, p.scale_log2, bh);
            }
          }
        }
        const float none[NTW][2] = {};
#pragma unroll 1
        for (; gl < ngt; gl += KS) group_quant<NTW, BITS>(st, qs, sbase, gl, p.scale_log2, none);
      }
    }
    if (t + 1 < ii.te || KS == 1) {
      // reads alone need no proxy fence before the slot is handed back to
      // the copy engine; the zeroed rows of a partial bf16 tile do
      if (wrote) fence_proxy_async();
      __syncwarp();
      if (lane == 0) mbar_arrive(&sm.empty[slot]);
    } else {
      last_slot = slot;
    }
  }
  finish_item<NTW>(p, sm, st, it, last_slot, NG, KS, grp, ks);
}

template <int NTW, class W>
__device__ void consume(const W& w, AttnSmem& sm) {
  const int warp = threadIdx.x >> 5;
  const int mtiles = w.call(0).mtiles;  // the same for every call of a launch
  const int NG = (mtiles + NTW - 1) / NTW <= 1 ? 1 : ((mtiles + NTW - 1) / NTW <= 2 ? 2 : 4);
  const int KS = kConsumers / NG;
  const int grp = warp % NG, ks = warp / NG;
  uint32_t seq = 0;
  bool aborted = false;
  // thread 0: the last arrival (call << 16 | bh), checked one item later
  int prev_key = -1, prev_arrivals = -1;
  if (threadIdx.x == 0) sm.n_pending = 0;
  for (uint32_t iseq = 0;; ++iseq) {
    const int k = iseq % kItemQ;
    if (!mbar_wait(&sm.item_full[k], (iseq / kItemQ) & 1, w.call(0).status, 13, w.call(0).wait_ns)) break;
    const int pos = sm.item_pos[k];
    if (pos < 0) break;
    int it, local, c;
    const AttnParams& p = w.locate(pos, &local, &c);
    const ItemInfo ii = decode_item(p, local, &it);
    const SegDev& sd = p.seg[ii.s];
    if (seg_is_bf16(sd.kind) || ii.tail)
      run_item<NTW, 16>(p, sm, ii, it, k, seq, aborted, NG, KS, grp, ks);
    else if (sd.bits == 4)
      run_item<NTW, 4>(p, sm, ii, it, k, seq, aborted, NG, KS, grp, ks);
    else
      run_item<NTW, 2>(p, sm, ii, it, k, seq, aborted, NG, KS, grp, ks);

    // Arrive on the item's counter; the CTA whose arrival completes a
    // (sequence, KV head) owes its merge, done after its last item so that
    // no warp waits for the atomic here.
    consumer_sync();
    if (threadIdx.x == 0 && !p.defer_merge) {
      if (prev_key >= 0 && prev_arrivals == w.items_per_bh(prev_key >> 16) - 1)
        sm.pending[sm.n_pending++] = prev_key;
      prev_arrivals = counter_arrive_acq_rel(&p.counters[ii.bh]);
      prev_key = (c << 16) | ii.bh;
    }
    if (sm.n_pending == kMaxPendingMerges) {  // list full (not reached for planned grids): merge now
      consumer_sync();
      for (int k = 0; k < kMaxPendingMerges; ++k) {
        const AttnParams& pc = w.call(sm.pending[k] >> 16);
        const int bh = sm.pending[k] & 0xffff;
        final_merge<NTW>(pc, sm, bh, nullptr);
        consumer_sync();
        if (threadIdx.x == 0) pc.counters[bh] = 0;
      }
      if (threadIdx.x == 0) sm.n_pending = 0;
      consumer_sync();
    }
  }
  if (threadIdx.x == 0) {
    if (prev_key >= 0 && prev_arrivals == w.items_per_bh(prev_key >> 16) - 1)
      sm.pending[sm.n_pending++] = prev_key;
  }
  consumer_sync();
  for (int k = 0; k < sm.n_pending; ++k) {
    const AttnParams& pc = w.call(sm.pending[k] >> 16);
    const int bh = sm.pending[k] & 0xffff;
    final_merge<NTW>(pc, sm, bh, &seq);  // the producer has stopped: the ring is idle
    consumer_sync();
    if (threadIdx.x == 0) pc.counters[bh] = 0;
  }
}

template <int NTW, class P>
__global__ void __launch_bounds__(kAttnThreads, ctas_for<NTW>()) attend_kernel(const __grid_constant__ P params) {
  const typename WorkOf<P>::type w{params};
  extern __shared__ uint8_t dyn_smem[];
  AttnSmem& sm = *reinterpret_cast<AttnSmem*>(
      (reinterpret_cast<uintptr_t>(dyn_smem) + 1023) & ~static_cast<uintptr_t>(1023));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // Launched programmatically, this launch may begin while the kernel before
  // it is finishing: nothing below reads memory before that kernel (the
  // append of this call's layer) has completed, and the next launch may
  // begin as soon as this one runs.
  griddep_wait();
  griddep_launch_dependents();

  if (threadIdx.x == 0) {
    for (int s = 0; s < stages_for<NTW>(); ++s) {
      mbar_init(&sm.full[s], 1);
      mbar_init(&sm.empty[s], kConsumers);
    }
    for (int q = 0; q < kItemQ; ++q) {
      mbar_init(&sm.item_full[q], 1);
      mbar_init(&sm.item_empty[q], kConsumers);
    }
    fence_barrier_init();
  }
  __syncthreads();

  if (warp == kConsumers) {
    if (lane == 0) {
      for (int c = 0; c < w.n_calls(); ++c) {
        const AttnParams& p = w.call(c);
        for (int s = 0; s < p.nseg; ++s) {
          prefetch_tmap(&p.tmap[2 * s]);
          prefetch_tmap(&p.tmap[2 * s + 1]);
        }
      }
      produce<NTW>(w, sm);
    }
  } else {
    consume<NTW>(w, sm);
  }
}

static void attend_setup_once() {
  static std::once_flag once;
  std::call_once(once, [] {
    cudaFuncSetAttribute(attend_kernel<1, AttnParams>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         (int)attend_smem_bytes<1>());
    cudaFuncSetAttribute(attend_kernel<2, AttnParams>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         (int)attend_smem_bytes<2>());
    cudaFuncSetAttribute(attend_kernel<1, MultiAttnParams>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         (int)attend_smem_bytes<1>());
    cudaFuncSetAttribute(attend_kernel<2, MultiAttnParams>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         (int)attend_smem_bytes<2>());
  });
}

// Resident CTAs per SM of the instantiation used for `ntiles` n-tiles.
int attend_ctas_per_sm(int ntiles) {
  static int cached[2] = {0, 0};
  const int w = ntiles <= 1 ? 0 : 1;
  if (cached[w] == 0) {
    attend_setup_once();
    int n = 0;
    if (w == 0)
      cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, attend_kernel<1, AttnParams>, kAttnThreads,
                                                    attend_smem_bytes<1>());
    else
      cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, attend_kernel<2, AttnParams>, kAttnThreads,
                                                    attend_smem_bytes<2>());
    cached[w] = n > 0 ? n : 1;
  }
  return cached[w];
}

void launch_attend(const AttnParams& p, int grid, cudaStream_t st) {
  attend_setup_once();
  const bool pdl = pdl_enabled();
  if (p.mtiles <= 1)
    launch_maybe_pdl(pdl, attend_kernel<1, AttnParams>, grid, kAttnThreads, attend_smem_bytes<1>(), st, p);
  else
    launch_maybe_pdl(pdl, attend_kernel<2, AttnParams>, grid, kAttnThreads, attend_smem_bytes<2>(), st, p);
  count_launch();
  if (p.defer_merge) {
    // always launched programmatically: its CTAs take the SM slots the
    // attention CTAs free and wait (griddepcontrol.wait) for that launch to
    // complete, instead of a launch gap after it
    launch_maybe_pdl(true, merge_partials_kernel, p.batch * p.n_kv_heads * p.mtiles * kMergeChunks, 256, 0, st, p);
    count_launch();
  }
}

void launch_attend_multi(const MultiAttnParams& m, int grid, cudaStream_t st) {
  attend_setup_once();
  if (m.call[0].mtiles <= 1)
    attend_kernel<1, MultiAttnParams><<<grid, kAttnThreads, attend_smem_bytes<1>(), st>>>(m);
  else
    attend_kernel<2, MultiAttnParams><<<grid, kAttnThreads, attend_smem_bytes<2>(), st>>>(m);
  count_launch();
}

}  // namespace uc

// ------------------------------------------------------ no-allocation variant
//
// uc_attend_static: decode attention for callers that cannot hand the
// library a workspace. Its scratch (status word, merge counters, partial
// outputs) is this file-scope device array, reserved on every GPU that loads
// the library for as long as the process lives.
namespace uc {

constexpr size_t kStaticScratchBytes = size_t(8) << 20;  // 8 MiB
static __device__ __align__(256) uint8_t g_attend_scratch[kStaticScratchBytes];

// Device address of g_attend_scratch on the current device. In host code the
// array's name is only a host-side handle, so the address is fetched once per
// device (with that device current) and cached.
constexpr int kMaxDevices = 64;  // devices whose scratch address is cached

static uint8_t* attend_static_scratch(uc_status* status) {
  static std::mutex mu;
  static uint8_t* addr[kMaxDevices] = {};
  int dev = -1, n_dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaGetDeviceCount(&n_dev) != cudaSuccess || dev < 0 ||
      dev >= n_dev || dev >= kMaxDevices) {
    set_error("uc_attend_static: no usable current CUDA device");
    *status = UC_ERR_CUDA;
    return nullptr;
  }
  std::lock_guard<std::mutex> lock(mu);
  if (addr[dev] == nullptr) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_attend_scratch);
    if (e != cudaSuccess || p == nullptr) {
      set_error("uc_attend_static: cudaGetSymbolAddress failed: %s", cudaGetErrorString(e));
      *status = UC_ERR_CUDA;
      return nullptr;
    }
    addr[dev] = static_cast<uint8_t*>(p);
  }
  return addr[dev];
}

}  // namespace uc

extern "C" uc_status uc_attend_static(const void* q, int32_t n_q_heads, int32_t n_qtok,
                                      const uc_segment* const* segs, int32_t n_seg, void* out, float* lse,
                                      float* mass, void* stream) {
  UC_TRACE();
  using namespace uc;
  // uc_attend's own argument checks come first: the same inputs give the
  // same statuses, and nothing below runs on a rejected call
  size_t need = 0;
  uc_status st = attend_precheck(q, n_q_heads, n_qtok, segs, n_seg, out, "uc_attend_static", &need);
  if (st != UC_OK) return st;
  uint8_t* scratch = attend_static_scratch(&st);
  if (scratch == nullptr) return st;
  if (need > kStaticScratchBytes) {
    set_error("uc_attend_static: this call needs %zu bytes of scratch, more than the %zu of its static "
              "array; use uc_attend with a caller workspace",
              need, kStaticScratchBytes);
    return UC_ERR_OOM;
  }
  // The array keeps the previous call's contents: clear the status word and
  // the merge counters, which must start at zero.
  const size_t clear = 256 + attend_counter_bytes();
  if (cudaMemsetAsync(scratch, 0, clear, reinterpret_cast<cudaStream_t>(stream)) != cudaSuccess) {
    set_error("uc_attend_static: clearing the scratch failed: %s", cudaGetErrorString(cudaGetLastError()));
    return UC_ERR_CUDA;
  }
  return uc_attend(q, n_q_heads, n_qtok, segs, n_seg, out, lse, mass, scratch, kStaticScratchBytes, stream);
}
