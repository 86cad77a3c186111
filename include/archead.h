/*
 * archead.h -- C ABI of the GB300 (sm_103a) packed LM-head forward.
 *
 * The packed head replaces a dense output projection W (V x d) by
 *
 *   W_hat = W_d + A_w B_w,      W_d = Q(A_c) Q(B_c) + Q_SC4(W - A_c B_c)
 *
 * (paper, Section 3.2, Eqs. 3 and 6) and the forward evaluates
 *
 *   Y_hat = H W_d^T + (H B_w^T) A_w^T                       (Eq. 7)
 *
 * without ever forming a dense W_hat: the INT4 residual is streamed and
 * dequantised tile by tile, and both rank-r branches are applied as factored
 * products.  In this ABI, H is called x (M tokens x d) and the factors are
 *
 *   core_u = A_c (V x r_c), core_v = B_c^T (d x r_c),
 *   corr_a = A_w (V x r_r), corr_b = B_w^T (d x r_r).
 *
 * Conventions for every entry point:
 *  - Nothing throws across the ABI; every call returns an archead_status.
 *  - Argument and shape checks are synchronous and happen before any work is
 *    queued.  M == 0 is a valid no-op.
 *  - "stream" is a cudaStream_t passed as void* (NULL = legacy default stream).
 *    Device work is queued on it; results are ready when it completes.
 *  - Device pointers must be 16-byte aligned; x rows must be contiguous.
 *  - A pack may be used by one stream at a time (the workspace it owns for
 *    the pre-pass and the cross-entropy partials is not shared safely between
 *    concurrent calls); successive calls may use different streams.  When a
 *    call needs a larger workspace than the pack holds, it synchronises the
 *    device before freeing the old one, so earlier calls on any stream are
 *    done with it.  Different packs are independent.
 *  - Faults detected on the device (an out-of-range target, a pipeline wait
 *    that gave up) are latched in a per-pack device error word and reported
 *    by archead_sync_status().
 */
#ifndef ARCHEAD_H_
#define ARCHEAD_H_

#include <stddef.h>
#include <stdint.h>

/* Version of this interface: 2 added archead_pack_create_ex and
 * archead_abi_version.  archead_desc only grows by appending fields. */
#define ARCHEAD_ABI_VERSION 2

#if defined(__GNUC__)
#define ARCHEAD_API __attribute__((visibility("default")))
#else
#define ARCHEAD_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef struct archead_pack archead_pack; /* opaque, owned by the library */

typedef enum {
  ARCHEAD_OK = 0,
  ARCHEAD_ERR_INVALID_ARG = 1,    /* NULL pointer, bad shape, misaligned pointer      */
  ARCHEAD_ERR_UNSUPPORTED = 2,    /* valid request outside the supported envelope     */
  ARCHEAD_ERR_OOM = 3,            /* a device allocation failed                       */
  ARCHEAD_ERR_CUDA = 4,           /* a CUDA runtime call failed (see last_error)      */
  ARCHEAD_ERR_DEVICE_TIMEOUT = 5, /* a bounded pipeline wait gave up on the device    */
  ARCHEAD_ERR_TARGET_RANGE = 6    /* a CE target was outside [0, V); its ce is NaN     */
} archead_status;

typedef enum {
  ARCHEAD_OUT_BF16 = 0, /* logits rounded to bf16 (nearest even) from fp32 accumulators */
  ARCHEAD_OUT_FP32 = 1  /* logits as the fp32 accumulators                               */
} archead_out_dtype;

/* Stored format of the packed head (archead_desc.format). */
typedef enum {
  ARCHEAD_FORMAT_INT8 = 0, /* INT8 core left factor, one fp16 scale per residual group          */
  ARCHEAD_FORMAT_SC4 = 1   /* the paper's format: 5-bit core left factor, 4-bit scale codes    */
} archead_format;

typedef enum {
  ARCHEAD_PATH_AUTO = 0,    /* decode kernel for M <= 64 (M <= 48 for heads whose
                               shared memory leaves only 16-token launches), prefill
                               kernel above (and for heads too wide for the decode
                               kernel's shared memory)                                 */
  ARCHEAD_PATH_DECODE = 1,  /* decode kernel: one launch per 16, 32 or 64 tokens (by M
                               and the head's width); ARCHEAD_ERR_UNSUPPORTED for
                               heads too wide for it                                   */
  ARCHEAD_PATH_PREFILL = 2  /* tensor-core prefill kernel                               */
} archead_path;

/*
 * The packed head in its canonical layout (paper, Appendix C, Table
 * "Logical contents of the packed ARCHead state dictionary"; Section 3.2).
 * Symmetric quantisers throughout (no zero points); every scale is an IEEE
 * fp16 bit pattern.  Pointers may be host or device memory (anything CUDA's
 * unified addressing resolves); they are read during archead_pack_create only.
 *
 *   res_codes    uint8 [V][d/2]   signed INT4 residual Q_SC4(W - A_c B_c),
 *                                 two's complement, packed along d: byte j of
 *                                 row n holds k = 2j (low nibble) and k = 2j+1
 *   res_scales   fp16  [V][d/g]   one scale per (row, group of g along d)
 *   core_u       int8  [V][r_c]   core left factor codes,  core_u_scale fp16 [r_c] (per column)
 *   core_v       int8  [d][r_c]   core right factor codes, core_v_scale fp16 [r_c] (per column)
 *   corr_a       int8  [V][r_r]   correction left codes,   corr_a_scale fp16 [V]   (per row)
 *   corr_b       int8  [d][r_r]   correction right codes,  corr_b_scale fp16 [d/g][r_r]
 *                                 (per group of g along d and rank column)
 *
 * Dequantised values are code * scale, e.g. W_hat[n,k] =
 *   code[n,k] s_R[n,k/g] + sum_j core_u[n,j] su[j] core_v[k,j] sv[j]
 *                        + sum_j corr_a[n,j] sa[n] corr_b[k,j] sb[k/g,j].
 * A rank of 0 drops that branch (its pointers may then be NULL): r_c = r_r = 0
 * is the plain group-wise INT4 head, r_r = 0 the "core only" variant.
 *
 * format = ARCHEAD_FORMAT_SC4 selects the paper's own packed format
 * (Section 3.2, Eq. 3: Q_5 core left factor and the SC4 residual with
 * quantised group scales; Appendix C).  Three fields change meaning:
 *   res_scales    uint8 [V][ceil(G/2)]  4-bit unsigned group-scale codes q,
 *                                 low nibble = even group, G = d/g;
 *   res_row_scale fp16  [V]       one per row; the group scale is
 *                                 s_R[n, grp] = res_row_scale[n] * (q + 1);
 *   core_u        uint8 [V][ceil(5 r_c / 8)]  5-bit two's complement codes
 *                                 (-16..15), code j in bits 5j..5j+4 of the
 *                                 row's bytes read as one little-endian bit
 *                                 string (unused top bits ignored).
 * Everything else is as above.  res_row_scale is read only in this format
 * (callers of the INT8 format may pass a shorter struct without it).
 *
 * Supported envelope: V >= 1; d a multiple of 64 and of g; g in {32, 64,
 * 128, 256}; 0 <= r_c, r_r <= 256.
 */
typedef struct {
  int64_t vocab;       /* V */
  int64_t hidden;      /* d */
  int32_t core_rank;   /* r_c */
  int32_t corr_rank;   /* r_r */
  int32_t group_size;  /* g */
  int32_t format;      /* archead_format */
  const void *res_codes;
  const void *res_scales;
  const void *core_u;
  const void *core_u_scale;
  const void *core_v;
  const void *core_v_scale;
  const void *corr_a;
  const void *corr_a_scale;
  const void *corr_b;
  const void *corr_b_scale;
  const void *res_row_scale; /* ARCHEAD_FORMAT_SC4 only */
} archead_desc;

/*
 * Build a pack on the current CUDA device: copies every component into
 * library-owned device memory and re-tiles it into the kernels' layouts
 * (one pass on the device).  Returns after the pack is ready; the caller's
 * buffers may be freed as soon as it returns.  On failure *out is NULL.
 */
ARCHEAD_API archead_status archead_pack_create(const archead_desc *desc, void *stream, archead_pack **out);

/*
 * archead_pack_create with the caller's sizeof(archead_desc).  The library
 * reads only the fields that lie within desc_size, so a struct compiled
 * against an older header (appended fields missing) stays valid; the fields
 * of version 1 (up to corr_b_scale) are required (ARCHEAD_ERR_INVALID_ARG if
 * desc_size is smaller), and a field the format needs that lies beyond
 * desc_size (res_row_scale for ARCHEAD_FORMAT_SC4) is ARCHEAD_ERR_INVALID_ARG.
 */
ARCHEAD_API archead_status archead_pack_create_ex(const archead_desc *desc, size_t desc_size, void *stream,
                                                  archead_pack **out);

/* ARCHEAD_ABI_VERSION of the library actually loaded. */
ARCHEAD_API int archead_abi_version(void);

/* Free a pack and everything it owns.  NULL is a no-op. */
ARCHEAD_API void archead_destroy(archead_pack *pack);

/*
 * Logits (Eq. 7): logits[m][n] = sum_k x[m][k] W_hat[n][k] for m < M, n < V.
 *   x       device, bf16 [M][d] row-major
 *   logits  device, [M][V] row-major, bf16 or fp32 per out_dtype
 * fp32 accumulation throughout; bf16 output is rounded once at the end.
 */
ARCHEAD_API archead_status archead_forward(archead_pack *pack, const void *x, int64_t M, void *logits,
                               archead_out_dtype out_dtype, void *stream);

/* archead_forward with an explicit kernel choice (for crossover sweeps and tests). */
ARCHEAD_API archead_status archead_forward_path(archead_pack *pack, const void *x, int64_t M, void *logits,
                                    archead_out_dtype out_dtype, archead_path path, void *stream);

/*
 * Per-token cross entropy in nats (paper, Section 4, "Data and metrics"):
 *   ce[m] = log sum_n exp(y[m][n]) - y[m][targets[m]],   y = logits of Eq. 7,
 * computed from the fp32 accumulators with an online max / sum of exp over
 * vocabulary tiles; no V-wide logits are written to memory.
 *   x        device, bf16 [M][d];  targets device, int32 [M];  ce device, fp32 [M]
 * A target outside [0, V) gives ce = NaN and latches ARCHEAD_ERR_TARGET_RANGE.
 */
ARCHEAD_API archead_status archead_forward_ce(archead_pack *pack, const void *x, int64_t M, const int32_t *targets,
                                  float *ce, void *stream);

ARCHEAD_API archead_status archead_forward_ce_path(archead_pack *pack, const void *x, int64_t M, const int32_t *targets,
                                       float *ce, archead_path path, void *stream);

/*
 * Greedy decoding output without logits: for each token m, index[m] = the
 * vocabulary row of the largest logit of Eq. 7 (the first one on ties, as
 * argmax) and, if value != NULL, value[m] = that logit (fp32, before any
 * bf16 rounding).  The kernels keep a (largest logit, row) pair per token and
 * vocabulary slice instead of writing the V-wide logits, and a second pass
 * merges the slices in a fixed order.  The paper does not define this entry
 * point; it is the generation-time use of the head (greedy next token).
 *   x      device, bf16 [M][d] row-major, 16-byte aligned
 *   index  device, int32 [M], 16-byte aligned (caller-owned)
 *   value  device, float [M], 16-byte aligned, or NULL
 * Returns ARCHEAD_ERR_INVALID_ARG for bad pointers or M < 0; M == 0 is a no-op.
 * `path` as in archead_forward_path.
 */
ARCHEAD_API archead_status archead_forward_argmax(archead_pack *pack, const void *x, int64_t M, int32_t *index,
                                                  float *value, void *stream);
ARCHEAD_API archead_status archead_forward_argmax_path(archead_pack *pack, const void *x, int64_t M, int32_t *index,
                                                       float *value, archead_path path, void *stream);

/*
 * Vocabulary-parallel evaluation.  The forward is row-separable (paper,
 * Section 3.2, Eq. 7: every logit y[m][n] involves only row n of the
 * V-indexed components -- residual codes and scales, core_u, corr_a and its
 * row scales -- and the d-side factors core_v, corr_b, which every shard
 * holds whole).  A head can therefore be cut into P contiguous blocks of
 * vocabulary rows, one pack per block (shard p holds global rows
 * [row0_p, row0_p + V_p) as its rows 0..V_p-1), typically one per GPU:
 * logits need no exchange (each shard writes its own columns), cross entropy
 * and greedy output need one small exchange per token, made by the caller
 * (an all-gather over its process group, for example), followed by one of
 * the combines below.
 *
 * archead_forward_lse_partial: for each token m, over this shard's rows,
 *   parts[3m]     = max_n y[m][n]
 *   parts[3m + 1] = sum_n exp(y[m][n] - parts[3m])
 *   parts[3m + 2] = y[m][targets[m] - row0] if row0 <= targets[m] < row0 + V
 *                   of this pack, else -inf (another shard owns the target).
 *   x device bf16 [M][d]; targets device int32 [M] (GLOBAL rows);
 *   parts device fp32 [M][3], 16-byte aligned (caller-owned).
 *   row0 is this shard's first global row (row0 + V < 2^31).
 *
 * archead_lse_combine: parts device fp32 [num_shards][M][3], the shards'
 * partials in shard order; ce device fp32 [M]:
 *   ce[m] = max + log(sum) - y[m][t_m]   (merged over the shards in order),
 * NaN where no shard (or more than one) reports the target.  Uses the
 * current device; deterministic.
 *
 * archead_argmax_combine: values fp32 [num_shards][M] and indices int32
 * [num_shards][M] from each shard's archead_forward_argmax (shard-local
 * rows), row0 int32 [num_shards] the shards' first global rows, all device
 * memory; writes index[m] = the global row of the largest logit over all
 * shards (the lowest row on ties, as argmax) and, if value != NULL, that
 * logit.  Uses the current device; deterministic.
 */
ARCHEAD_API archead_status archead_forward_lse_partial(archead_pack *pack, const void *x, int64_t M,
                                                       const int32_t *targets, int64_t row0, float *parts,
                                                       archead_path path, void *stream);
ARCHEAD_API archead_status archead_lse_combine(const float *parts, int num_shards, int64_t M, float *ce, void *stream);
ARCHEAD_API archead_status archead_argmax_combine(const float *values, const int32_t *indices, const int32_t *row0,
                                                  int num_shards, int64_t M, int32_t *index, float *value,
                                                  void *stream);

/*
 * End-to-end call with HOST buffers: copies x (host, bf16 [M][d]) to the
 * device, runs archead_forward into logits_host ([M][V], bf16 or fp32) and
 * waits for the stream.  When logits_host is pinned and mapped into the
 * device's address space (cudaHostAlloc / cudaMallocHost, or torch's
 * pin_memory, under unified addressing) the kernels write the logits into it
 * directly; otherwise they go to a device buffer owned by the pack and are
 * copied back.  Either way the call returns with the logits in logits_host.
 */
ARCHEAD_API archead_status archead_forward_host(archead_pack *pack, const void *x_host, int64_t M, void *logits_host,
                                    archead_out_dtype out_dtype, void *stream);

/*
 * Persistent storage of the packed head (paper, Section 3.3, Eq. 10): the
 * sum of numel * element_size over the stored components listed above, in
 * the pack's format.  The correction's row scales count only when r_r > 0.
 */
ARCHEAD_API int64_t archead_pack_bytes(const archead_pack *pack);

/* Bytes of device memory the pack holds now: tiled copies, padding and workspace. */
ARCHEAD_API int64_t archead_device_bytes(const archead_pack *pack);

/*
 * Dequantise rows [row0, row0 + nrows) of one stored component with the
 * kernels' own device unpacking, as fp32 code * scale (exact):
 *   0 residual [nrows][d]   1 core_u [nrows][r_c]   2 core_v [nrows][r_c] (rows are k)
 *   3 corr_a  [nrows][r_r]  4 corr_b [nrows][r_r] (rows are k)
 * out is device memory.
 */
ARCHEAD_API archead_status archead_debug_dequant(const archead_pack *pack, int component, int64_t row0, int64_t nrows,
                                     float *out, void *stream);

/*
 * Wait for the stream, then read and clear the pack's device error word.
 * Returns ARCHEAD_OK, ARCHEAD_ERR_TARGET_RANGE, ARCHEAD_ERR_DEVICE_TIMEOUT,
 * ARCHEAD_ERR_UNSUPPORTED (a kernel found its shared-memory window misaligned
 * for its TMA layout and skipped its work; archead_last_error() says so) or
 * ARCHEAD_ERR_CUDA.
 */
ARCHEAD_API archead_status archead_sync_status(archead_pack *pack, void *stream);

/*
 * Upper bound, in SM clock cycles, on every pipeline wait inside the
 * kernels (default about one second).  A wait that exceeds it latches
 * ARCHEAD_ERR_DEVICE_TIMEOUT and its block returns early.
 */
ARCHEAD_API archead_status archead_set_wait_budget(archead_pack *pack, int64_t cycles);

/*
 * Launch one block whose only job is a bounded wait on a barrier that
 * nothing completes, so the timeout path can be tested without hanging or
 * faulting the device.  Returns after queueing it; follow with
 * archead_sync_status() to read ARCHEAD_ERR_DEVICE_TIMEOUT.
 */
ARCHEAD_API archead_status archead_debug_wait_timeout(archead_pack *pack, void *stream);

/*
 * Allocation-free variant of archead_forward for M <= 16 (the decode path).
 * The paper has no counterpart; this exists for callers that must not
 * allocate device memory while they run the head (all memory reserved up
 * front, a stream being captured into a CUDA graph under a pool that forbids
 * new allocations, latency-critical loops that cannot take cudaMalloc's locks
 * or cudaFree's device synchronisation).  archead_forward grows the pack's
 * workspace with cudaMalloc; this call never allocates: its scratch lives in
 * one fixed 512 KiB array compiled into the library, which every device that
 * loads the library holds until the process exits.
 *   x       device, bf16 [M][d];  logits device, [M][V] (bf16 or fp32), as archead_forward.
 * The first call with a pack (at any M <= 16) looks up that array's device
 * address on the pack's device and prepares every decode kernel the pack can
 * use; make that first call before any stream capture.  The address is kept
 * for the life of the process, so calls after a cudaDeviceReset of that
 * device are not supported.  All calls on a device share the array: calls
 * whose work overlaps on the GPU (other streams, other packs at the same
 * time) race.  Returns ARCHEAD_ERR_UNSUPPORTED (see
 * archead_last_error) when M > 16 or the head needs more than 512 KiB of
 * scratch (pre-pass partial sums: 2 KB per 32 rank columns per 256 of d, plus
 * 1 KB per 16 rank columns; 174 KB for d=4096, r_c+r_r=160).
 */
ARCHEAD_API archead_status archead_forward_decode_noalloc(archead_pack *pack, const void *x, int64_t M,
                                                          void *logits, archead_out_dtype out_dtype, void *stream);

/*
 * Offline construction of a packed head (paper, Section 3.4, Algorithm 1;
 * Appendix B steps 3-7): the quantisation and packing steps, on the device.
 * The dense linear algebra around them (H^T H, the eigendecomposition of the
 * damped covariance, the randomized SVDs of W and of E T_p) is done by library
 * routines in paper_2608_02703_gb300/construct.py, which calls these.  All
 * pointers are device memory; inputs are fp32, row-major.
 *
 * archead_quantize_symmetric: codes int8 [rows][cols] and fp16 scales
 *   [rows/group_rows][cols/group_cols] of x, one scale per group_rows x
 *   group_cols block: scale = fp16(max|x| / qmax) (fp32 division, round to
 *   nearest even), code = clamp(rint(x / scale), -qmax, qmax) with the
 *   division in fp32 and ties to even; code 0 where the scale is 0.
 *   bits 8 (qmax 127: Q_8 and the INT8 correction factors), 5 (qmax 15: the
 *   paper's Q_5 core left factor) or 4 (qmax 7: the INT4 residual).
 *   Row-wise: group_rows = 1, group_cols = cols; per column: group_rows =
 *   rows, group_cols = 1; B_w^T group-wise along d: group_rows = g,
 *   group_cols = 1; residual with one scale per group: 1 x g.
 * archead_quantize_residual_sc4: the residual in the paper's format: per row
 *   s_row = fp16(max|r| / 112), per group q = clamp(ceil(max_group|r| /
 *   (7 s_row)) - 1, 0, 15), codes against s_row (q + 1) in [-7, 7];
 *   codes int8 [rows][cols], scale_codes uint8 [rows][cols/group_size]
 *   (unpacked, 0..15), row_scale fp16 [rows].  cols/group_size <= 1024.
 * archead_pack_codes: bits 4: two's complement nibbles, byte j of a row =
 *   columns 2j (low) and 2j+1 (high), [rows][ceil(cols/2)]; bits 5: code j in
 *   bits 5j..5j+4 of the row's little-endian bit string,
 *   [rows][ceil(5 cols / 8)] (the canonical layouts of archead_desc).
 * archead_dequant_symmetric / archead_dequant_residual_sc4: code * scale in
 *   fp32 (exact), the inverse maps of the two quantisers.
 * Return ARCHEAD_ERR_INVALID_ARG for shapes that the groups do not divide;
 * device work is queued on the stream.
 */
ARCHEAD_API archead_status archead_quantize_symmetric(const float *x, int64_t rows, int64_t cols, int64_t group_rows,
                                                      int64_t group_cols, int bits, int8_t *codes, uint16_t *scales,
                                                      void *stream);
ARCHEAD_API archead_status archead_quantize_residual_sc4(const float *r, int64_t rows, int64_t cols, int group_size,
                                                         int8_t *codes, uint8_t *scale_codes, uint16_t *row_scale,
                                                         void *stream);
ARCHEAD_API archead_status archead_pack_codes(const int8_t *codes, int64_t rows, int64_t cols, int bits,
                                              uint8_t *packed, void *stream);
ARCHEAD_API archead_status archead_dequant_symmetric(const int8_t *codes, const uint16_t *scales, int64_t rows,
                                                     int64_t cols, int64_t group_rows, int64_t group_cols, float *out,
                                                     void *stream);
ARCHEAD_API archead_status archead_dequant_residual_sc4(const int8_t *codes, const uint8_t *scale_codes,
                                                        const uint16_t *row_scale, int64_t rows, int64_t cols,
                                                        int group_size, float *out, void *stream);

/* Per-kernel timing with CUDA events on the launch stream (off by default). */
typedef struct {
  const char *name;  /* static string */
  int64_t launches;
  double total_ms;
} archead_kernel_stat;

ARCHEAD_API archead_status archead_profile_enable(archead_pack *pack, int enable);
/* Collect timings of completed launches; returns the number of entries written. */
ARCHEAD_API int archead_profile_read(archead_pack *pack, archead_kernel_stat *out, int max_entries);

ARCHEAD_API const char *archead_status_string(archead_status status);
/* Message of the last CUDA error seen by this thread (empty if none). */
ARCHEAD_API const char *archead_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* ARCHEAD_H_ */
