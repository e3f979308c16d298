/*
 * unicache.h — C ABI of the GB300-native UniCache compressed-KV hot path.
 *
 * UniCache (arxiv 2609.32831) splits the attention context of a unified
 * multimodal model into typed segments (§3.1), gives each candidate type one
 * compression policy from offline calibration (§3.2, App. B), shares one
 * storage budget between types by attention mass (§3.3, Eq. 1-3), compresses
 * every segment independently (§3.4) and attends over all of them with one
 * shared softmax (App. E).
 *
 * Conventions for every entry point:
 *  - Device pointers are plain CUDA device addresses owned by the caller; the
 *    library never frees caller memory and allocates device memory only in
 *    uc_compress_budget (a library-owned segment, through the caller's
 *    allocator hook or the stream-ordered CUDA allocator; released by
 *    uc_segment_free). Host pointers are marked "host".
 *  - bf16 tensors are row-major with the last dimension (head_dim = 128)
 *    contiguous. Device arrays must be 16-byte aligned; bf16 row blocks read
 *    by TMA must be 16-byte aligned and tensor bases 128-byte aligned for best
 *    throughput.
 *  - `stream` is a cudaStream_t passed as void*. Calls are asynchronous on
 *    that stream unless stated otherwise.
 *  - Every argument is validated before any launch. On error nothing is
 *    launched, no output is written, the status is returned and a message is
 *    available from uc_last_error() (per host thread).
 *  - Conditions only the device can see (a non-finite value to quantize, a
 *    bounded wait that ran out) are recorded in the first 16 bytes of the
 *    call's workspace and read with uc_workspace_status().
 *  - No entry point ever falls back to a CPU implementation.
 */
#ifndef UNICACHE_H
#define UNICACHE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  UC_OK = 0,
  UC_ERR_ARG = 1,       /* null pointer, bad enum value, misaligned pointer */
  UC_ERR_SHAPE = 2,     /* unsupported or inconsistent sizes */
  UC_ERR_BUDGET = 3,    /* a budget that cannot be met (capacity too small) */
  UC_ERR_RANGE = 4,     /* NaN/Inf input, or fp16 scale / zero-point overflow */
  UC_ERR_OOM = 5,       /* workspace smaller than required, or an allocation failed */
  UC_ERR_CUDA = 6,      /* a CUDA runtime / driver call failed */
  UC_ERR_TIMEOUT = 7    /* a bounded device-side wait ran out */
} uc_status;

/* Segment kinds: how one cache type is stored (App. E, "Physical, type-aware
 * KV storage"). FULL keeps every token in bf16 (protected objects of §3.1 or
 * candidates whose budget is the full size); EVICT keeps the top-k tokens in
 * bf16 with their logical indices; QUANT keeps every token as low-bit codes;
 * EVICT_QUANT keeps the top-k tokens, then quantizes them. */
typedef enum {
  UC_KIND_FULL = 0,
  UC_KIND_EVICT = 1,
  UC_KIND_QUANT = 2,
  UC_KIND_EVICT_QUANT = 3
} uc_kind;

/* Compression policies assigned per task-type pair by calibration (§3.2). */
typedef enum { UC_POLICY_PROTECTED = -1, UC_POLICY_EVICT = 0, UC_POLICY_QUANT = 1 } uc_policy;

#define UC_HEAD_DIM 128   /* the only supported head dimension */
#define UC_GROUP 32       /* quantization group (tokens for K, channels for V) */
#define UC_MAX_BATCH 64   /* sequences per segment */
#define UC_MAX_SEGMENTS 8 /* segments per attend call / types per table */
#define UC_MAX_QTOKENS 8  /* decode-shaped attend calls; more take the dense path */
#define UC_MAX_CALLS 8    /* decode calls per uc_attend_batch launch */

/*
 * One compressed segment: one cache type of one layer, for B sequences and
 * Hkv KV heads. Its storage is caller-allocated device memory (sizes from
 * uc_segment_sizes_of()), or the library's for a segment uc_compress_budget
 * returned. Token counts may differ per sequence (budgets are
 * per sequence) but are equal across the KV heads of one sequence.
 *
 * Packed layout (App. E: "packed low-bit representations with scales,
 * minima, and a short BFloat16 residual tail"), per (b, kvh) block; `cap`
 * is the token capacity per block (a multiple of 64 for quantized kinds):
 *
 *   k, v        bf16 rows [.. , 128]. FULL/EVICT: the kept tokens in
 *               ascending index order, block (b, kvh) starting at row
 *               (b*Hkv + kvh)*row_stride + row_offset. QUANT/EVICT_QUANT: the
 *               residual tail (n_kept mod 32 most recent kept tokens), 32
 *               rows per block, row_stride = 32, row_offset = 0.
 *   k_codes     keys, per-channel groups of 32 consecutive kept tokens, in
 *               tensor-core fragment order: for each 8-token tile, 32 lanes x
 *               (bits*4) bytes; lane (n = lane/4, j = lane%4) holds the codes
 *               of token n of the tile for channels {16i+2j, 16i+2j+1,
 *               16i+2j+8, 16i+2j+9 : i = 0..7}; inside a 32-bit word the
 *               codes of channel pairs sit at bit offsets (p*bits, 16+p*bits).
 *               Block size cap*128*bits/8 bytes.
 *   k_params    fp16 (scale, zero) per (group, channel), 512 bytes per group:
 *               [group][i = 0..7][j = 0..3][s(c0) s(c1) | s(c8) s(c9) |
 *               z(c0) z(c1) | z(c8) z(c9)] with c0 = 16i+2j.
 *   v_codes     values, per-token groups of 32 channels, fragment order: for
 *               each 16-token tile, 32 lanes x (bits*8) bytes; lane
 *               (g = lane/4, j = lane%4) holds tokens {2j, 2j+1, 2j+8, 2j+9}
 *               of the tile for channels {8m+g : m = 0..15}.
 *   v_params    fp16 (scale, zero) per (token, channel group), 16 bytes per
 *               token: [16-token tile][group 0..3][j = 0..3][s(t0) s(t1) |
 *               s(t8) s(t9) | z(t0) z(t1) | z(t8) z(t9)] with t0 = 2j.
 *   kept_idx    int32 logical token indices [B, Hkv, cap], ascending.
 *
 * Quantization (a reading of App. E with the measured workloads' constants):
 * qmax = 2^bits - 1, s = fp16((max - min) / qmax + 0), z = fp16(min + 0) (a
 * zero scale or minimum is stored as +0),
 * code = clamp(rint((x - z) / s), 0, qmax) in IEEE fp32 round-to-nearest-even
 * (code = 0 when s == 0); attention reads x_hat = code * s + z.
 */
typedef struct uc_segment {
  int32_t kind;        /* uc_kind */
  int32_t bits;        /* 16 for FULL/EVICT; 4 or 2 for QUANT/EVICT_QUANT */
  int32_t batch;       /* B, 1..UC_MAX_BATCH */
  int32_t n_kv_heads;  /* Hkv */
  int32_t head_dim;    /* must equal UC_HEAD_DIM */
  int32_t n_src;       /* tokens per (b, kvh) in the uncompressed source */
  int32_t cap;         /* token capacity per (b, kvh) block */
  int32_t label;       /* caller's cache-type id (free use) */
  int32_t n_kept_host[UC_MAX_BATCH]; /* host mirror of n_kept; the library
                                        keeps it in step with its own writes */
  int32_t* n_kept;     /* device int32 [B]: tokens stored per sequence */
  int32_t* kept_idx;   /* device int32 [B, Hkv, cap]; NULL for FULL */
  void* k;             /* device bf16 rows (see layout) */
  void* v;
  int64_t row_stride;  /* rows between consecutive (b, kvh) blocks of k / v */
  int64_t row_offset;  /* first row of the segment inside each block */
  int64_t rows_total;  /* rows addressable from k / v (bounds of the buffer) */
  void* k_codes;       /* device, quantized kinds only */
  void* k_params;
  void* v_codes;
  void* v_params;
  uint64_t cache_key;  /* library-private: zero-initialise, never modify */
  uint8_t cache[256];  /* library-private descriptor cache */
} uc_segment;

/* Byte sizes of the caller-allocated arrays of a segment (0 when unused). */
typedef struct {
  uint64_t k, v, k_codes, k_params, v_codes, v_params, kept_idx, n_kept;
} uc_segment_sizes;

/*
 * Segment table of one task and layer chunk (§3.1-§3.3). Inputs and outputs
 * of the host policy calls; one entry per cache type.
 */
typedef struct uc_segment_table {
  int32_t n_types;
  int32_t candidate[UC_MAX_SEGMENTS];     /* in: 1 candidate, 0 protected (§3.1) */
  int32_t n_tokens[UC_MAX_SEGMENTS];      /* in: tokens per KV head, S_a = 512 * n */
  int32_t policy[UC_MAX_SEGMENTS];        /* in/out: uc_policy */
  double concentration[UC_MAX_SEGMENTS];  /* out: averaged top-share (App. B) */
  double mass[UC_MAX_SEGMENTS];           /* in: m_a^(c), Eq. 1 */
  double budget[UC_MAX_SEGMENTS];         /* in: b_a^(c) bytes per KV head
                                             (S_a for c = 0); out: b_a^(c+1) */
  int32_t keep[UC_MAX_SEGMENTS];          /* out: tokens to keep */
  int32_t bits[UC_MAX_SEGMENTS];          /* out: 16, 4 or 2 */
  int32_t kind[UC_MAX_SEGMENTS];          /* out: uc_kind to build */
} uc_segment_table;

/* ---------------------------------------------------------------- general */

/* Message of the last error on this host thread ("" if none). */
const char* uc_last_error(void);

/* ABI version, currently 1. */
int32_t uc_version(void);

/* Number of kernels this library has launched in this process. */
uint64_t uc_launch_count(void);

/* Issue order of the dense (many-query) attention kernel, process-wide.
 * 1 (default): the issuing thread waits for a Q tile's P V to complete
 * before the next Q K^T of that tile, which overwrites P's tensor-memory
 * columns. 0: that Q K^T is issued right behind the P V; this relies on the
 * tensor pipe reading P before the later MMA writes those columns, an
 * ordering the two MMAs (different accumulators) are not documented to
 * have. On GB300 both orders give bit-identical results (tested) and 0 is
 * 2.8 % faster on the denoising workload. Returns the previous setting. */
int32_t uc_set_dense_serial_pv(int32_t serial);

/* Limit, in nanoseconds, of every bounded wait inside the decode attention
 * kernels (a producer waiting for a free ring slot, consumers waiting for a
 * tile or a work item) and the quantizer (a warp waiting for its staged
 * rows), process-wide; a wait that runs out records UC_ERR_TIMEOUT in the
 * call's workspace status word and the kernel returns without hanging. 0 restores the default (2 s). Read when a call is built
 * (a captured graph keeps the value of its capture). Returns the previous
 * value. */
uint64_t uc_set_wait_limit(uint64_t ns);

/* Programmatic dependent launch of the decode kernels (uc_attend's attention
 * and merge kernels, uc_append / uc_append_next), process-wide, read when a
 * call launches (a captured graph keeps what its capture saw). With 1, the
 * next kernel in the stream may start while the current one's last CTAs are
 * finishing: an attention kernel still waits for the kernel before it (so
 * its layer's append is complete), but an append waits for nothing. The
 * caller therefore orders launches so that an append never overlaps a
 * kernel reading its segment, and gives consecutive attention calls their
 * own workspaces: a multi-layer decode step (append of layer l + 1 after the
 * attention of layer l, one workspace per layer) qualifies. Default 0.
 * Returns the previous setting. */
int32_t uc_set_programmatic_launch(int32_t on);

/* Test hook for the bounded waits (no counterpart in the paper): the next
 * decode attention call leaves the first tile of its work item at processing
 * position `pos` uncopied, or the next group quantization (uc_compress_segment
 * or uc_recompress_segment into a packed segment, whichever comes first)
 * leaves one K row of its group `pos` uncopied (groups counted block by block,
 * each (sequence, KV head) block holding as many groups as the largest keep
 * count has); the waits for it give up after the wait limit
 * and the call reports UC_ERR_TIMEOUT (its outputs are then meaningless).
 * One-shot; a negative `pos` cancels it. */
void uc_debug_withhold_tile(int32_t pos);

/* Synchronises `stream`, reads the status word a kernel may have written into
 * `workspace` (first 16 bytes), clears it and returns it (UC_OK if clean). */
uc_status uc_workspace_status(void* workspace, void* stream);

/* Byte sizes of a segment's arrays for the kind, bits, batch, n_kv_heads and
 * cap filled in `seg` (pointers are ignored). cap must be a multiple of 64
 * for quantized kinds. */
uc_status uc_segment_sizes_of(const uc_segment* seg, uc_segment_sizes* out);

/* ------------------------------------------------------ host policy (L3) */

/*
 * App. B (Calibration Setting): attention concentration is the share of a
 * type's within-type attention mass held by its top ceil(top_frac * n)
 * tokens. `mass` (host, n floats) is one example's per-token mass.
 */
uc_status uc_concentration(const float* mass, int64_t n, double top_frac, double* out);

/*
 * §3.2 / App. B: offline policy assignment. `mass` (host) holds
 * n_examples * table->n_types pointers; mass[e * n_types + a] points to
 * table->n_tokens[a] floats, the per-token mass of type a in calibration
 * example e. Writes table->concentration (mean over examples) and
 * table->policy: UC_POLICY_EVICT when concentration >= threshold, else
 * UC_POLICY_QUANT; protected types get UC_POLICY_PROTECTED.
 */
uc_status uc_calibrate_policy(uc_segment_table* table, const float* const* mass,
                              int32_t n_examples, double top_frac, double threshold);

/*
 * §3.3 Eq. 2 and the redistribution rule, with the shared budget
 * B^(c+1) = rho * sum_a S_a over candidate types (S_a = 512 * n_tokens[a]
 * bytes per KV head, bf16 K + V). For candidate types,
 * b_a = min(b_a^(c), m_a / sum_j m_j * B^(c+1)); budget left by capped types
 * is redistributed in proportion to mass among uncapped types with m > 0
 * until none is left or all are capped (some may stay unused). b_a^(c) is
 * table->budget[a], or S_a when first_chunk != 0 (b^(0) = S). Then §3.4 maps
 * each budget to a policy configuration: eviction keeps floor(b / 512)
 * tokens in bf16; quantization takes int4 if n * 160 <= b, else int2 if
 * n * 96 <= b, else int2 on the floor(b / 96) top tokens. Writes budget,
 * keep, bits, kind. Protected types are untouched (kind FULL, keep = n).
 */
uc_status uc_allocate_budget(uc_segment_table* table, double rho, int32_t first_chunk);

/* §3.3 Eq. 3: rho^(c+1) = min(rho^(c), max(rho_min, rho_init * M^(c) / M^(0))).
 * Requires 0 < rho_min <= rho_init <= 1 and M^(0) > 0. */
uc_status uc_retention_schedule(double rho_prev, double rho_init, double rho_min,
                                double m_c, double m_0, double* rho_out);

/* §3.3 Eq. 3 for one (sequence, layer chunk) from its table: M^(c) is the
 * sum of table->mass over candidate types (§3.3 Eq. 1 summed over the types
 * that can be compressed). With first_chunk != 0 (chunk 0, full KV):
 * *m_0 = M^(0) and *rho_out = rho_init. Otherwise *rho_out is Eq. 3 with
 * M^(c) and *m_0, or rho_prev when *m_0 is 0 (no mass on the candidates at
 * chunk 0). Requires 0 < rho_min <= rho_init <= 1; masses finite, >= 0. */
uc_status uc_retention_step(const uc_segment_table* table, int32_t first_chunk, double rho_prev,
                            double rho_init, double rho_min, double* m_0, double* rho_out);

/* One segment configuration of a cache type for a whole batch. */
typedef struct {
  int32_t kind;      /* uc_kind shared by the batch's sequences */
  int32_t bits;      /* 16, 4 or 2 */
  int32_t full_view; /* 1: every sequence keeps every token in bf16 (a view, nothing to compress) */
  int32_t max_keep;  /* largest per-sequence keep count (the segment's capacity) */
} uc_type_config;

/*
 * §3.4 for a batch (a reading: one segment holds a type of one layer for
 * every sequence of the batch, so it has one kind and bit width while keep
 * counts stay per sequence). `tables`: n_seq tables after uc_allocate_budget
 * (one per sequence, same types). For type `type`: keep[b] = tables[b].keep;
 * the bit width is the lowest any sequence's budget allows; the kind is FULL
 * (full_view = 1) when every sequence's configuration is FULL, else EVICT for
 * bf16, QUANT when every sequence keeps every token, EVICT_QUANT otherwise.
 * Protected types (candidate 0) keep every token (a full view).
 */
uc_status uc_plan_batch(const uc_segment_table* tables, int32_t n_seq, int32_t type, int32_t* keep,
                        uc_type_config* out);

/* Tokens a fixed keep fraction retains (a reading: the paper gives fractions,
 * not a rounding): max(1, floor(keep_frac * n)) for n > 0 (the product
 * guarded against binary rounding by 1e-9), 0 for n = 0. 0 < keep_frac <= 1. */
uc_status uc_keep_count(int32_t n, double keep_frac, int32_t* out);

/* ---------------------------------------------------- device kernels (L1) */

/*
 * Observation-window attention scores (§3.3 Eq. 1's P; App. E "Batched GQA
 * token selection"): for every sequence b, KV head j and context token t,
 *   scores[b, j, t] = sum_{h in heads of j} sum_{w < W} softmax_t(q_{b,h,w} . k_{b,j,t} / sqrt(128))
 * with the softmax over all n_ctx tokens (no mask). Query head h reads KV
 * head h / (Hq / Hkv).
 *   qwin   bf16 [B, Hq, W, 128]
 *   k      bf16, block (b, j) = rows (b*Hkv + j)*k_row_stride .. + n_ctx
 *   scores fp32 [B, Hkv, n_ctx] (written)
 * Requires Hq % Hkv == 0, (Hq / Hkv) * W <= 256, n_ctx >= 1.
 * workspace: uc_score_workspace_size() bytes, 16-byte aligned.
 */
uc_status uc_score_accumulate(const void* qwin, const void* k, int32_t batch, int32_t n_q_heads,
                              int32_t n_kv_heads, int32_t window, int32_t n_ctx,
                              int64_t k_row_stride, float* scores, void* workspace,
                              size_t workspace_bytes, void* stream);
size_t uc_score_workspace_size(int32_t batch, int32_t n_q_heads, int32_t n_kv_heads,
                               int32_t window, int32_t n_ctx);

/*
 * Eq. 1 from observation scores: for one (layer, step) pair the inner term is
 *   m[b, s] = sum_{j, t in [begin_s, end_s)} scores[b, j, t] / (Hq * W)
 * (the mean over heads and window queries of the probability on segment s).
 * The call writes (accumulate = 0) or adds (accumulate = 1) weight * m into
 * mass; calling it for every pair of a chunk with weight = 1 / |chunk| leaves
 * the chunk average m_a^(c) of Eq. 1 in mass. begin / end are host arrays of
 * n_seg token offsets into the context. mass: device fp32 [B, n_seg].
 */
uc_status uc_segment_mass(const float* scores, int32_t batch, int32_t n_kv_heads, int32_t n_ctx,
                          const int32_t* begin, const int32_t* end, int32_t n_seg,
                          int32_t n_q_heads, int32_t window, float weight, int32_t accumulate,
                          float* mass, void* stream);

/*
 * Compress one segment (§3.4; App. E storage and token selection).
 * Source rows: block (b, j) of k_src / v_src starts at row
 * (b*Hkv + j)*src_row_stride + src_row_offset and holds seg->n_src tokens.
 * scores: fp32, block (b, j) at (b*Hkv + j)*scores_stride + scores_offset
 * (ignored for QUANT). Per sequence b, seg->n_kept_host[b] is the number of
 * tokens to keep (<= n_src, <= cap); for EVICT kinds the kept tokens are the
 * n_recent most recent plus the top scores among the rest (ties to the lower
 * index, NaN -> UC_ERR_RANGE in the status word). The kept tokens are stored
 * in ascending index order, quantized for the quantized kinds. Writes every
 * array of `seg` and seg->n_kept. FULL segments are not compressed (use them
 * as views).
 * workspace: uc_compress_workspace_size() bytes.
 */
uc_status uc_compress_segment(const void* k_src, const void* v_src, int64_t src_row_stride,
                              int64_t src_row_offset, const float* scores, int64_t scores_stride,
                              int64_t scores_offset, int32_t n_recent, uc_segment* seg,
                              void* workspace, size_t workspace_bytes, void* stream);
size_t uc_compress_workspace_size(const uc_segment* seg);

/*
 * Device memory for library-owned segments, stream-ordered: alloc returns
 * `bytes` of device memory usable in order on `stream` (NULL on failure;
 * 16-byte alignment required), free returns it in order on `stream`. `ctx`
 * is passed through. A NULL uc_allocator pointer selects cudaMallocAsync /
 * cudaFreeAsync.
 */
typedef struct uc_allocator {
  void* (*alloc)(size_t bytes, void* stream, void* ctx);
  void (*free)(void* ptr, void* stream, void* ctx);
  void* ctx;
} uc_allocator;

/*
 * Segment compression under a budget (§3.4, with App. E storage and token
 * selection): the paper's compress_segment(K, V, scores, budget) -> segment.
 * `tables`: one uc_segment_table per sequence (batch of them) after
 * uc_allocate_budget, i.e. Eq. 2's budgets mapped to keep counts and bit
 * widths; `type` selects the cache type, whose tables' n_tokens must equal
 * n_src. The batch's configuration comes from uc_plan_batch (one kind and bit
 * width, per-sequence keep counts). Source rows, scores and n_recent are as
 * for uc_compress_segment. The call allocates the segment's arrays (capacity:
 * the largest keep count rounded up to 64) and a workspace through
 * `allocator` on `stream`, compresses, synchronises `stream`, releases the
 * workspace and returns the segment in *out, owned by the library until
 * uc_segment_free. Status: the argument, budget and shape errors of
 * uc_plan_batch / uc_compress_segment, UC_ERR_OOM when an allocation fails,
 * or the kernels' status (UC_ERR_RANGE for a NaN score or an fp16 overflow);
 * on any error nothing is returned and everything allocated is released.
 * A type whose every sequence keeps every token in bf16 (protected types and
 * full budgets) becomes a FULL view of the source rows: only its n_kept array
 * is allocated, and k_src / v_src must outlive the segment. A batch whose
 * keep counts are all 0 gives an empty segment; an evicting configuration
 * with some keep counts 0 and others not is UC_ERR_BUDGET.
 */
uc_status uc_compress_budget(const void* k_src, const void* v_src, int32_t batch, int32_t n_kv_heads,
                             int32_t n_src, int64_t src_row_stride, int64_t src_row_offset, const float* scores,
                             int64_t scores_stride, int64_t scores_offset, int32_t n_recent,
                             const uc_segment_table* tables, int32_t type, const uc_allocator* allocator,
                             void* stream, uc_segment** out);

/*
 * Returns a segment from uc_compress_budget to its allocator, in order on
 * the stream it was built on: work queued on that stream before this call
 * may still read it; work on other streams must be ordered before it by the
 * caller. NULL is ignored; a segment the library did not hand out is left
 * untouched (uc_last_error says so).
 */
void uc_segment_free(uc_segment* seg);

/*
 * Progressive re-compression (§3.3 Eq. 2-3 with §3.4): when a later chunk
 * lowers a type's budget, the type's already compressed segment `src` is
 * compressed further into `dst` (eviction is irreversible, so only what src
 * still holds can be kept). Per sequence b:
 *   rows      the n = src->n_kept[b] stored tokens of src as bf16: bf16 rows
 *             as stored; packed groups rebuilt as bf16(fp32(code * s + z))
 *             (the fp32 value is the correctly rounded code * s + z, then
 *             rounded to nearest even in bf16); the residual tail as stored.
 *   selection dst->n_kept_host[b] of those rows: every row for QUANT dst
 *             (which then requires dst keep == n); for EVICT / EVICT_QUANT
 *             the n_recent most recent rows plus the top-scoring older rows,
 *             with the score of stored row i taken from its logical token:
 *             scores[(b*Hkv + kvh)*scores_stride + scores_offset + idx_i],
 *             idx_i = src->kept_idx[b, kvh, i] (i itself for FULL src); ties
 *             go to the lower row, NaN sets UC_ERR_RANGE in the workspace.
 *   output    dst built from the selected rows exactly as uc_compress_segment
 *             builds it from bf16 rows (gather or group quantization), with
 *             dst->kept_idx holding the selected rows' logical indices
 *             (ascending) and dst->n_kept the keep counts.
 * src and dst share batch, n_kv_heads and n_src, may differ in kind, bits and
 * cap, and must not share any storage. src->n_kept_host must mirror
 * src->n_kept (see uc_append_next). keep may be 0 for evicting kinds.
 * workspace: uc_recompress_workspace_size(src, dst) bytes, 16-byte aligned
 * (2 * B * Hkv * src->cap * 256 bytes beyond 256 when src is packed).
 */
uc_status uc_recompress_segment(const uc_segment* src, const float* scores, int64_t scores_stride,
                                int64_t scores_offset, int32_t n_recent, uc_segment* dst,
                                void* workspace, size_t workspace_bytes, void* stream);
size_t uc_recompress_workspace_size(const uc_segment* src, const uc_segment* dst);

/*
 * Heavy-hitter statistics during decode (App. E "heavy-hitter and
 * recent-token selection", applied as decode proceeds): after a decode
 * attention call over a layer's segments, adds each stored token's
 * probability, summed over the query heads of its KV head and the T query
 * tokens, to an accumulator indexed by logical token:
 *   acc[b, kvh, acc_offset + idx_t] +=
 *       sum_{h of kvh, tau < T} exp(q_{b,h,tau} . k_t / sqrt(128) - lse[b, h, tau])
 * with lse the call's log-sum-exp over all of its segments (uc_attend's lse
 * output), so the added values are the call's softmax probabilities. seg is
 * one of that call's bf16 segments (FULL or EVICT); idx_t = kept_idx (row t
 * for FULL). Logits are recomputed in fp32 from the bf16 rows. q bf16
 * [B, Hq, T, 128] with T <= UC_MAX_QTOKENS and (Hq / Hkv) * T <= 64; acc fp32
 * [B, Hkv, acc_stride]. An index outside [0, acc_stride - acc_offset) sets
 * UC_ERR_RANGE in the workspace status word and is skipped. workspace: >= 256
 * bytes (status word). Each token has a single writer: results are
 * deterministic. uc_recompress_segment re-evicts by these scores.
 */
uc_status uc_accumulate_scores(const void* q, int32_t n_q_heads, int32_t n_qtok, const uc_segment* seg,
                               const float* lse, float* acc, int64_t acc_stride, int64_t acc_offset,
                               void* workspace, size_t workspace_bytes, void* stream);

/*
 * Eq. 1 from an attention call's own probabilities: for one (layer, step)
 * pair, the inner term of Eq. 1 for segment s of sequence b is
 *   m[b, s] = Mean_{h, t} mass[b, h, t, s]
 * (mass as written by uc_attend: the probability each query puts on the
 * segment's retained tokens). Writes (accumulate = 0) or adds
 * (accumulate = 1) weight * m into out; with weight = 1 / |chunk| over all
 * pairs of a chunk, out holds m_a^(c). mass: device fp32
 * [B, Hq, T, n_seg]; out: device fp32 [B, n_seg]. Summation order is fixed,
 * so repeated calls give identical results.
 */
uc_status uc_attention_mass(const float* mass, int32_t batch, int32_t n_q_heads, int32_t n_qtok,
                            int32_t n_seg, float weight, int32_t accumulate, float* out, void* stream);

/*
 * Shared-softmax attention over heterogeneous segments (App. E "Attention
 * over heterogeneous cache segments"), for any number T of query tokens:
 *   O[b, h, t]       = softmax(q K^T / sqrt(128)) V over the union of all
 *                      segments' stored tokens for KV head h / (Hq / Hkv)
 *   lse[b, h, t]     = log sum exp(q . k / sqrt(128))           (nullable)
 *   mass[b, h, t, s] = share of the probability on segment s      (nullable;
 *                      the per-(layer, step) term of Eq. 1)
 * q bf16 [B, Hq, T, 128]; O bf16 [B, Hq, T, 128]; lse fp32 [B, Hq, T];
 * mass fp32 [B, Hq, T, n_seg]. All segments share batch and n_kv_heads, and
 * every sequence must see at least one token.
 * T <= UC_MAX_QTOKENS (decode): split-K over token chunks of the packed
 * layout with a log-sum-exp merge, all on the device.
 * T > UC_MAX_QTOKENS (denoising / editing latents): the stored tokens are
 * rebuilt once per call as fp16 rows in the workspace (packed keys as an
 * fp16 hi + lo pair, so the logits keep ~22 bits), then attended on the
 * tensor cores, 128 keys per tile; at most 512 tiles per sequence, each
 * segment padded to a multiple of 128 tokens.
 * workspace: uc_attend_workspace_size() bytes, zero-filled once before first
 * use and used by uc_attend only (it holds merge counters that every call
 * leaves at zero again); calls sharing one workspace must not overlap.
 */
uc_status uc_attend(const void* q, int32_t n_q_heads, int32_t n_qtok, const uc_segment* const* segs,
                    int32_t n_seg, void* out, float* lse, float* mass, void* workspace,
                    size_t workspace_bytes, void* stream);
size_t uc_attend_workspace_size(const uc_segment* const* segs, int32_t n_seg, int32_t n_q_heads,
                                int32_t n_qtok);

/*
 * How uc_attend splits a decode-shaped call (T <= UC_MAX_QTOKENS) into work
 * items (App. E split-K over token chunks): introspection for callers and
 * tests. An item is a run of tiles of one segment of one (sequence, KV
 * head); heavy items split the long segments so that one round of them fills
 * the CTA slots, light items (the bf16 tails of packed segments, segments
 * under half an average heavy item) run last on CTAs that finished early.
 * slots: resident CTAs the launch may use; <= 0 asks this device's
 * occupancy (then a CUDA device must be current; otherwise the call touches
 * no device). Reads kind, bits, batch, n_kv_heads and n_kept_host of each
 * segment only. Errors: UC_ERR_ARG (null pointers), UC_ERR_SHAPE (segment
 * count, query shape or T beyond UC_MAX_QTOKENS).
 */
typedef struct {
  int32_t items_per_bh;                 /* partials per (sequence, KV head), <= 64 */
  int32_t n_heavy, n_light;             /* heavy / light items per (sequence, KV head) */
  int32_t grid;                         /* CTAs the launch starts */
  int32_t merge_kernel;                 /* 1: the split-K merge runs as a kernel of its own */
  int32_t n_chunks[UC_MAX_SEGMENTS];    /* items of each segment */
  int32_t light[UC_MAX_SEGMENTS];       /* 1: every item of the segment is light */
} uc_attend_plan_info;
uc_status uc_attend_plan(const uc_segment* const* segs, int32_t n_seg, int32_t n_q_heads, int32_t n_qtok,
                         int32_t slots, uc_attend_plan_info* out);

/*
 * Several independent decode-shaped attention calls in one launch (App. E,
 * "Batched attention": compatible calls combined into one variable-length
 * launch). Each call is exactly a uc_attend call with its own queries,
 * segment list (its own batch, KV heads, kinds and lengths) and outputs;
 * the calls' work items share one persistent grid, so short calls fill the
 * SMs that long ones leave idle. Requirements: 1 <= n_calls <= UC_MAX_CALLS;
 * every call decode-shaped (n_qtok <= UC_MAX_QTOKENS) with the same number
 * of 8-row query tiles ceil((Hq / Hkv) * T / 8); calls must not write the
 * same outputs. Results equal those of separate uc_attend calls up to the
 * summation order of the split-K merge. workspace:
 * uc_attend_batch_workspace_size() bytes, zero-filled once before first use
 * and used by uc_attend_batch only (its merge counters are left at zero).
 */
typedef struct uc_attend_call {
  const void* q;                /* bf16 [B, Hq, T, 128] */
  int32_t n_q_heads, n_qtok;    /* Hq, T */
  const uc_segment* const* segs;
  int32_t n_seg;
  void* out;                    /* bf16 [B, Hq, T, 128] */
  float* lse;                   /* fp32 [B, Hq, T] (nullable) */
  float* mass;                  /* fp32 [B, Hq, T, n_seg] (nullable) */
} uc_attend_call;

uc_status uc_attend_batch(const uc_attend_call* calls, int32_t n_calls, void* workspace, size_t workspace_bytes,
                          void* stream);
size_t uc_attend_batch_workspace_size(const uc_attend_call* calls, int32_t n_calls);

/*
 * uc_attend without a caller workspace. The paper has no counterpart: this
 * entry point exists for callers that cannot allocate device memory for
 * scratch space, such as a plug-in running inside a host framework that owns
 * the whole device memory pool, or code on a latency-critical path where a
 * cudaMalloc (which may synchronise the device) is not acceptable. It
 * computes exactly what uc_attend computes, with the same arguments minus the
 * workspace, and allocates nothing: its scratch is a static device array of
 * 8 MiB built into the library, which every GPU that loads the library holds
 * until the process exits.
 *  - A call whose scratch need (uc_attend_workspace_size) exceeds 8 MiB is
 *    rejected with UC_ERR_OOM before anything is launched.
 *  - The first call on a device looks up the array's device address (once
 *    per device, with that device current); make that first call before any
 *    stream capture.
 *  - All calls share the one array: calls that overlap on the GPU (for
 *    example on two streams at once) race and give wrong results; order them
 *    on one stream or through events. Each call clears the array's status
 *    word and merge counters before it launches.
 */
uc_status uc_attend_static(const void* q, int32_t n_q_heads, int32_t n_qtok, const uc_segment* const* segs,
                           int32_t n_seg, void* out, float* lse, float* mass, void* stream);

/*
 * Append one decode token per sequence to a segment (the residual tail of
 * App. E): k_new / v_new bf16 [B, Hkv, 128]; the token's logical index is
 * `position`. bf16 kinds store the row; quantized kinds store it in the tail
 * and, when the tail reaches 32 tokens, quantize it into a new group.
 * Increments seg->n_kept (device and host mirror). Requires n_kept < cap.
 */
uc_status uc_append(uc_segment* seg, const void* k_new, const void* v_new, int32_t position,
                    void* workspace, size_t workspace_bytes, void* stream);

/*
 * uc_append for frozen layouts replayed as CUDA graphs (App. E "Cached
 * metadata and execution plans"): the same append, but the token's logical
 * index is base_position + n_kept[b] read on the device, and nothing is
 * checked or updated on the host, so one captured call serves every later
 * decode step. seg->n_kept_host is not advanced (it still holds the count at
 * capture); capacity is checked on the device (UC_ERR_BUDGET in the
 * workspace status word, nothing written). A uc_attend captured in the same
 * graph keeps the plan of the capture-time counts and reads the current
 * counts from the device, so it covers the growing segment.
 */
uc_status uc_append_next(uc_segment* seg, const void* k_new, const void* v_new, int32_t base_position,
                         void* workspace, size_t workspace_bytes, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* UNICACHE_H */
