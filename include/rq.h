/*
 * rq.h -- C ABI of librq, the GB300 (sm_103a) hot path of RateQuant
 * (arXiv 2605.06675): per-head mixed-bit KV-cache quantization chosen by
 * reverse waterfilling, bit-packing, and decode attention that reads the
 * packed cache directly.
 *
 * Conventions for every entry point
 * ---------------------------------
 * - Plain C types only. Device pointers are ordinary pointers into device
 *   memory the caller owns; `stream` is a cudaStream_t passed as void*
 *   (NULL = legacy default stream). librq never allocates memory and keeps no
 *   state between calls apart from a cached per-device SM count and the fixed
 *   device array used by rq_decode_attention_static.
 * - Arguments are validated on the host before anything is launched; a bad
 *   argument returns an error code and launches nothing. A failed launch
 *   returns RQ_ERR_CUDA. Device entry points are asynchronous on `stream`.
 * - Conditions the device detects (non-finite input, a bit-width outside
 *   1..8 in the device table) are OR-ed into `*status_dev` (a device uint32;
 *   may be NULL) as RQ_STATUS_* bits; the kernels still write defined values
 *   and never trap or spin.
 * - Host-only functions are pure and thread-safe.
 *
 * Indexing
 * --------
 * - Component index of (layer l, kv head h, kind): i = (l * H_kv + h) * 2 + kind,
 *   kind 0 = K, 1 = V (Sec. 3.4 "K/V separation": 2N components share one budget).
 * - Bit table: uint8 bits[L][H_kv][2], the paper's static per-head lookup
 *   table (Sec. 3.4 "Pipeline summary"; App. M "No runtime overhead").
 * - GQA: query head j reads kv head j / (H_q / H_kv) (Sec. 4.1 "Models").
 * - Caches: one layer's K and V are [B][H_kv][S][d] contiguous, fp16 or bf16.
 */
#ifndef RQ_H
#define RQ_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define RQ_ABI_VERSION 2
#define RQ_HEAD_DIM 128
#define RQ_GROUP 32
#define RQ_MAX_GQA 8

typedef enum {
  RQ_OK = 0,
  RQ_ERR_INVALID_ARG = 1, /* NULL pointer, bad enum, n <= 0, ... */
  RQ_ERR_INFEASIBLE = 2,  /* budget not reachable with the allowed bit set */
  RQ_ERR_SHAPE = 3,       /* unsupported shape (d != 128, S % 32 != 0, ...) */
  RQ_ERR_ALIGNMENT = 4,   /* a device pointer is not 16-byte aligned */
  RQ_ERR_WORKSPACE = 5,   /* workspace smaller than the *_workspace_bytes query */
  RQ_ERR_CUDA = 6         /* a CUDA runtime call or launch failed */
} rq_status;

/* bits OR-ed into *status_dev by the kernels */
#define RQ_STATUS_NUMERIC 1u  /* a group held NaN/inf or its fp16 scale/zero overflowed */
#define RQ_STATUS_BAD_BITS 2u /* a device bit-table entry was outside 1..8; stream skipped */
#define RQ_STATUS_BAD_POSITION 4u /* a per-row position or token count (rq_append_rows,
                                     rq_decode_attention_rows) was out of range; row skipped */

typedef enum { RQ_F16 = 0, RQ_BF16 = 1 } rq_dtype;

/* RQ_PER_TOKEN: a group is 32 consecutive channels of one token (KIVI values,
 * QuaRot); RQ_PER_CHANNEL: 32 consecutive tokens of one channel (KIVI keys).
 * Sec. 2 "KV cache quantization", App. W "KIVI kernel".
 * RQ_PER_TOKEN_64 / RQ_PER_TOKEN_128: 64 consecutive channels of one token /
 * a token's whole 128-channel row, the value / key group sizes of App. W
 * "TurboQuant kernel" (min-max or absmax, not Lloyd-Max). They are stored
 * like RQ_PER_TOKEN: every group of 32 channels carries its wide group's
 * fp16 (scale, zero), so the block format and its size are unchanged. */
typedef enum {
  RQ_PER_TOKEN = 0,
  RQ_PER_CHANNEL = 1,
  RQ_PER_TOKEN_64 = 2,
  RQ_PER_TOKEN_128 = 3
} rq_grouping;

/* Per-group quantizer of a kind (keys or values), groups of 32 either way.
 * RQ_MINMAX: asymmetric min-max, scale = fp16(fp32(max - min) / (2^b - 1)),
 *   zero = fp16(min), codes 0 .. 2^b - 1 (KIVI values, Sec. 2).
 * RQ_ABSMAX: the symmetric absmax form of App. W ("TurboQuant kernel"),
 *   x_hat = round(x M / a) a / M, a = max |x|, M = 2^(b-1) - 1 (KIVI's
 *   "per-channel symmetric" keys, Sec. 2; QuaRot / RTN per-token symmetric,
 *   Sec. 4.1, Table 16). Stored like a min-max group: scale = fp16(a / M),
 *   zero = fp16(0 - M * scale), codes q + M in 0 .. 2M; b = 1 (M = 0) has
 *   the single level 0 (scale 0, zero 0, codes 0).
 * Codes are c = clamp(rint((x - zero) * (1/scale)), 0, c_max) in fp32 with
 * one rounding of the product, from the stored fp16 scale and zero, for
 * both; the decoder reads both the same way (x_hat = c * scale + zero).
 * For the wide per-token groupings the group's min, max or max |x| is taken
 * over its 64 or 128 values, and the codes from its stored scale and zero.
 * RQ_LLOYDMAX: the 2^b-level Lloyd-Max codebook of a unit Gaussian (App. F
 *   Table 8; TurboQuant's scalar quantizer, App. W) scaled by the group's
 *   RMS: scale = fp16(sqrt(s2 / 32)) with s2 the fp32 sum of squares of
 *   values 0..15 plus that of values 16..31 (each summed in order), zero = 0,
 *   code = the number of thresholds fp32(fp32((L_{i-1} + L_i) / 2) * scale)
 *   at or below the value (L = the fp16 levels of rq_lloydmax_levels),
 *   x_hat = L_code * scale. Per-token groups only (RQ_ERR_INVALID_ARG with
 *   per-channel groups), the grouping TurboQuant uses. */
typedef enum { RQ_MINMAX = 0, RQ_ABSMAX = 1, RQ_LLOYDMAX = 2 } rq_quantizer;

/* allocation flags */
#define RQ_CAP_5X 1u /* w_i <- min(w_i, 5 * mean w) first (App. W "Mitigation") */

typedef struct {
  int32_t L;          /* layers */
  int32_t B;          /* batch */
  int32_t H_kv;       /* kv heads */
  int32_t H_q;        /* query heads; H_q % H_kv == 0, H_q / H_kv <= 8 */
  int32_t S;          /* cached tokens; S % 32 == 0 */
  int32_t d;          /* head dim; must be 128 */
  int32_t group;      /* group size; must be 32 */
  int32_t dtype;      /* rq_dtype of K, V and q */
  int32_t k_grouping; /* rq_grouping of keys */
  int32_t v_grouping; /* rq_grouping of values */
  int32_t hadamard;   /* 1: rotate K and V per token by R = diag(signs) H / sqrt(128)
                         before quantizing (QuaRot, App. W "QuaRot kernel") */
  int32_t k_quantizer; /* rq_quantizer of keys */
  int32_t v_quantizer; /* rq_quantizer of values */
} rq_cache_desc;

const char* rq_status_string(rq_status s);
int32_t rq_abi_version(void);

/* The fp16 levels (bit patterns, ascending, 2^b of them) of the RQ_LLOYDMAX
 * codebook at b bits: the Lloyd-Max quantizer of N(0, 1), computed by the
 * library on first use (Lloyd's iteration, then Newton's method on the same
 * fixed point, in fp64) and rounded to nearest fp16. levels: host array of
 * 2^b entries. Errors: RQ_ERR_INVALID_ARG (b outside 1..8, NULL). */
rq_status rq_lloydmax_levels(int32_t b, uint16_t* levels);

/* ---------------------------------------------------------------- host ---- */

/* Fit D(b) = alpha * beta^-b per component by unweighted least squares of
 * ln D on b over b in [b_lo, b_hi] with D(b) > 0 (Assumption 1; Alg. 1 stage 2;
 * Sec. 3.4 "Distortion calibration"). mse: host [n][8], column k = D(k+1).
 * R^2 on ln D is returned in r2. If r2_min > 0, a component with
 * R^2 < r2_min gets beta = min(beta, mean fitted beta of its class)
 * (App. W "Outlier heads"); classes: host [n] (NULL = one class).
 * Fewer than two positive points: alpha = 0, beta = +inf, r2 = 1.
 * Outputs: host arrays of n doubles. Errors: RQ_ERR_INVALID_ARG. */
rq_status rq_fit_distortion(int32_t n, const double* mse, int32_t b_lo, int32_t b_hi,
                            double r2_min, const int32_t* classes, double* alpha,
                            double* beta, double* r2);

/* Integer allocation of Eq. 1: minimise sum_i w_i alpha_i beta_i^-b_i with
 * sum_i b_i = B = floor(avg_bits * n + 0.5) and every b_i in the allowed set
 * (bit k of allowed_mask set <=> k bits allowed, k in 1..8).
 * A contiguous set uses the greedy max-heap of Alg. 2 (marginal gain
 * w alpha beta^-b (1 - 1/beta), ties to the lower index; optimal by Prop. 3).
 * A non-contiguous set (e.g. {2,3,4,8}) uses an exact dynamic programme
 * (ties: the larger bit-width for the lower index).
 * flags: RQ_CAP_5X. Inputs/outputs are host arrays; bits_out: n uint8;
 * objective_out (nullable): the minimised objective.
 * Errors: RQ_ERR_INVALID_ARG, RQ_ERR_INFEASIBLE (B not reachable). */
rq_status rq_alloc(int32_t n, const double* w, const double* alpha, const double* beta,
                   double avg_bits, uint32_t allowed_mask, uint32_t flags, uint8_t* bits_out,
                   double* objective_out);

/* Continuous reverse waterfilling (Thm. 1, Eq. 2; App. B.1): free components
 * satisfy w_i alpha_i ln(beta_i) beta_i^-b_i = lambda with sum b_i = avg_bits * n;
 * components leaving [b_min, b_max] are clipped, fixed, and the rest
 * re-solved until none leaves (App. B.1 "Iterative waterfilling").
 * Requires beta_i > 1, w_i, alpha_i > 0. b_out: host n doubles.
 * Errors: RQ_ERR_INVALID_ARG, RQ_ERR_INFEASIBLE. */
rq_status rq_alloc_continuous(int32_t n, const double* w, const double* alpha,
                              const double* beta, double avg_bits, double b_min, double b_max,
                              double* b_out);

/* Byte offsets of every packed stream and the buffer size.
 * bits: host [L][H_kv][2]. offsets: host [L][B][H_kv][2] (uint64), filled in
 * (layer, batch, head, kind) order. A stream of S tokens at b bits is S/32
 * blocks of 512*(b+1) bytes: 512*b bytes of codes (32 lanes x 4b words in
 * MMA-fragment order) then 512 bytes of fp16 scale/zero metadata.
 * Errors: RQ_ERR_INVALID_ARG, RQ_ERR_SHAPE. */
rq_status rq_packed_layout(const rq_cache_desc* desc, const uint8_t* bits, uint64_t* offsets,
                           uint64_t* total_bytes);

/* -------------------------------------------------------------- device ---- */

/* Size of the workspace rq_calibrate_distortion needs for n components of T
 * tokens: n * (T/32) * 8 doubles. */
size_t rq_calibrate_workspace_bytes(int32_t n, int32_t T);

/* Distortion sweep (Alg. 1 stage 2; Sec. 3.4 "Distortion calibration"):
 * for every component i and b = 1..8, quantize-dequantize every group with
 * the kind's quantizer (after the per-token Hadamard rotation when
 * `hadamard`) and store mse_dev[i][b-1] = mean over the component's T*128
 * elements of (y - y_hat)^2 in the quantizer's domain, fp64. Each quantizer
 * gets its own curve and so its own fitted beta (Sec. 3.4, Sec. 4.3, App. C).
 * x: device [n][T][128] of `dtype`; component i is a key (grouping
 * k_grouping, quantizer k_quantizer) when i is even, a value (v_grouping,
 * v_quantizer) when odd.
 * signs_dev: device int8 [128] of +-1 (NULL = all +1; used when hadamard).
 * ws: device workspace of rq_calibrate_workspace_bytes(n, T) bytes.
 * Deterministic (fixed reduction order).
 * Errors: RQ_ERR_INVALID_ARG, RQ_ERR_SHAPE (T % 32), RQ_ERR_ALIGNMENT,
 * RQ_ERR_WORKSPACE, RQ_ERR_CUDA. */
rq_status rq_calibrate_distortion(const void* x, int32_t dtype, int32_t n, int32_t T,
                                  int32_t k_grouping, int32_t v_grouping, int32_t hadamard,
                                  int32_t k_quantizer, int32_t v_quantizer,
                                  const int8_t* signs_dev, double* mse_dev, void* ws,
                                  size_t ws_bytes, uint32_t* status_dev, void* stream);

/* Quantize and pack one layer (the quantizer kernel indexing the per-head
 * table, App. M / App. U): for every (batch, kv head, kind) stream, every
 * group gets the scale, zero and codes of the kind's rq_quantizer, e.g.
 * for min-max scale = fp16(fp32(max - min) / (2^b - 1)), zero = fp16(min),
 * codes c = clamp(rint((x - zero) * (1/scale)), 0, 2^b - 1) in fp32, written
 * to packed + offsets[layer][batch][head][kind] in the block format of
 * rq_packed_layout. k, v: [B][H_kv][S][128] of desc->dtype (16-byte
 * aligned) in device memory, or in page-locked host memory the device can
 * address (cudaHostAlloc / cudaHostRegister under unified addressing): the
 * kernel then reads the cache over the host link itself, with no staging
 * copy (on GB300's NVLink-C2C about twice the rate of copy-engine transfers
 * of the same buffers). bits_dev: device [L][H_kv][2]; offsets_dev: device copy of the
 * rq_packed_layout offsets; packed: device buffer of total_bytes (16-byte
 * aligned). signs_dev as in rq_calibrate_distortion.
 * Errors: RQ_ERR_INVALID_ARG, RQ_ERR_SHAPE, RQ_ERR_ALIGNMENT, RQ_ERR_CUDA. */
rq_status rq_quantize_pack(const rq_cache_desc* desc, int32_t layer, const void* k,
                           const void* v, const int8_t* signs_dev, const uint8_t* bits_dev,
                           const uint64_t* offsets_dev, void* packed, uint32_t* status_dev,
                           void* stream);

/* How this process issues its decode calls (a library setting; the paper
 * has no counterpart). It sets how the split kernel deals the splits of a
 * call to the four split groups of its CTAs, and where the merge kernel's
 * CTAs start; results are bit-identical either way. Process-wide, read by every later decode call on any device;
 * the default is RQ_DECODE_BACK_TO_BACK.
 *  - RQ_DECODE_BACK_TO_BACK: decode calls follow one another on the stream
 *    (a loop over layers): a CTA takes consecutive splits of the plan, all of
 *    one size, so the CTAs of the smaller splits leave their SMs early to
 *    the next call's splits.
 *  - RQ_DECODE_INTERLEAVED: other kernels run between the calls (a model's
 *    layers): every CTA takes one split from each quarter of the plan, the
 *    same work per SM, and the merge CTAs start where split CTAs have left
 *    (the split kernel keeps all 128 registers a thread), so a call on its
 *    own ends sooner.
 * Errors: RQ_ERR_INVALID_ARG (another value). */
typedef enum { RQ_DECODE_BACK_TO_BACK = 0, RQ_DECODE_INTERLEAVED = 1 } rq_decode_pattern;
rq_status rq_decode_set_pattern(int32_t pattern);

/* Workspace rq_decode_attention needs on the current device (the split-K
 * partial records). */
rq_status rq_decode_workspace_bytes(const rq_cache_desc* desc, size_t* bytes);

/* Decode attention of one query per (batch, query head) over all S cached
 * tokens of one layer, reading the packed mixed-bit cache directly
 * (App. W "Kernel fusion"): out[b][j] = sum_t softmax_t(q_j . k_hat_t / sqrt(128)) v_hat_t
 * with k_hat, v_hat the dequantized cache of kv head j / (H_q / H_kv)
 * (x_hat = c * scale + zero, or L_c * scale for RQ_LLOYDMAX groups); with
 * desc->hadamard the rotated cache is used as Q(XR)R^T (App. W "QuaRot kernel").
 * Split-K over the sequence, then a log-sum-exp merge kernel launched as a
 * programmatic dependent of the split kernel (it overlaps the split grid's
 * tail and waits for it before reading; where its shared memory fits, its
 * CTAs start beside the split CTAs and wait there).
 * q: device [B][H_q][128] of desc->dtype; out: device fp32 [B][H_q][128];
 * ws: device workspace of at least rq_decode_workspace_bytes, 16-byte
 * aligned, contents arbitrary on entry; one call at a time per workspace.
 * Errors: RQ_ERR_INVALID_ARG, RQ_ERR_SHAPE (S == 0, S % 32, GQA > 8),
 * RQ_ERR_ALIGNMENT, RQ_ERR_WORKSPACE, RQ_ERR_CUDA. */
rq_status rq_decode_attention(const rq_cache_desc* desc, int32_t layer, const void* q,
                              const void* packed, const uint8_t* bits_dev,
                              const uint64_t* offsets_dev, const int8_t* signs_dev, float* out,
                              void* ws, size_t ws_bytes, uint32_t* status_dev, void* stream);

/* Allocation-free variant of rq_decode_attention (the paper has no counterpart;
 * this is a library convenience). Some callers cannot allocate device memory
 * where they decode: embedding runtimes whose device allocator belongs to
 * someone else, and plugins that are handed only the tensors they read and
 * write. This entry point takes the same arguments minus the workspace: the
 * split-K partials live in a fixed device array inside librq of
 * RQ_STATIC_SCRATCH_BYTES bytes, reserved on every GPU that loads the
 * library until the process exits. It calls no cudaMalloc/cudaFree.
 *  - Limit: the rq_decode_workspace_bytes of the shape must fit in
 *    RQ_STATIC_SCRATCH_BYTES; larger shapes return RQ_ERR_WORKSPACE before
 *    anything is launched.
 *  - The first call on a device looks up the array's device address
 *    (cudaGetSymbolAddress, a host-side runtime call) with that device
 *    current. The address is cached for the life of the process: a device
 *    reset (cudaDeviceReset) invalidates it and is not supported.
 *  - Every call on a device shares the one array, which keeps the previous
 *    call's contents (each call overwrites every record it reads, so nothing
 *    needs clearing). Calls that can overlap on the GPU (different streams
 *    without ordering) race on the array and give wrong results: serialise
 *    them, or use rq_decode_attention with separate workspaces.
 * Other arguments, results and errors as rq_decode_attention. */
#define RQ_STATIC_SCRATCH_BYTES (8u << 20)
rq_status rq_decode_attention_static(const rq_cache_desc* desc, int32_t layer, const void* q,
                                     const void* packed, const uint8_t* bits_dev,
                                     const uint64_t* offsets_dev, const int8_t* signs_dev,
                                     float* out, uint32_t* status_dev, void* stream);

/* ---- Decode-time append (KIVI-style residual window) ----------------------
 * The paper allocates bits per head uniformly over token positions (appendix
 * "Scope and Extensions", "Design choices"), so a token appended during
 * decoding is stored at its head's widths like every other. Per-channel key
 * groups span 32 tokens, so the open block of every stream stays unquantized
 * in a residual window of 32 tokens (the KIVI residual, Sec. 2) until it is
 * full; it is then quantized and packed exactly as rq_quantize_pack packs
 * that block. desc->S is the cache's capacity in tokens (a multiple of 32);
 * the packed buffer and offsets are those of rq_packed_layout(desc). */

/* Bytes of the residual windows of a cache: [L][B][H_kv][2][32][128] values of
 * desc->dtype, K then V per (layer, batch, kv head); token t sits in slot
 * t % 32. 0 for an invalid descriptor. */
size_t rq_residual_bytes(const rq_cache_desc* desc);

/* Append the token at position pos (0 <= pos < desc->S, the same position for
 * every batch row) of one layer: k_new, v_new: device [B][H_kv][128] of
 * desc->dtype (16-byte aligned) are written to slot pos % 32 of the layer's
 * residual windows (device, rq_residual_bytes, 16-byte aligned). When
 * pos % 32 == 31 the windows are full and block pos / 32 of every stream of
 * the layer is quantized (and rotated with desc->hadamard) and packed into
 * `packed` at the widths of bits_dev; the windows are then free for the next
 * block. signs_dev, status_dev as in rq_quantize_pack.
 * Errors: RQ_ERR_INVALID_ARG (null pointers, layer or pos out of range),
 * RQ_ERR_SHAPE, RQ_ERR_ALIGNMENT, RQ_ERR_CUDA. */
rq_status rq_append(const rq_cache_desc* desc, int32_t layer, int32_t pos, const void* k_new,
                    const void* v_new, void* residual, const int8_t* signs_dev,
                    const uint8_t* bits_dev, const uint64_t* offsets_dev, void* packed,
                    uint32_t* status_dev, void* stream);

/* Decode attention over the first n_tokens (1 <= n_tokens <= desc->S) of one
 * layer: tokens below 32 * (n_tokens / 32) from the packed blocks, the last
 * n_tokens % 32 from the residual windows (unquantized; slots 0..). Otherwise
 * as rq_decode_attention (same workspace size, ws of
 * rq_decode_workspace_bytes(desc)); residual may be NULL when
 * n_tokens % 32 == 0. */
rq_status rq_decode_attention_len(const rq_cache_desc* desc, int32_t layer, int32_t n_tokens,
                                  const void* q, const void* packed, const uint8_t* bits_dev,
                                  const uint64_t* offsets_dev, const int8_t* signs_dev,
                                  const void* residual, float* out, void* ws, size_t ws_bytes,
                                  uint32_t* status_dev, void* stream);

/* Decode-time append for a batch whose rows are at different lengths (a
 * ragged decode batch): as rq_append, with one position per batch row in
 * pos_dev (device int32 [B], 4-byte aligned). Row b's new token goes to slot
 * pos_dev[b] % 32 of its windows; when that is slot 31 the row's windows are
 * quantized and packed as block pos_dev[b] / 32 of its streams. A negative
 * position appends nothing for that row (a row that is not decoding this
 * step); a position at or past desc->S sets RQ_STATUS_BAD_POSITION and skips
 * the row. Always launches (the positions are read on the device).
 * Errors: as rq_append. */
rq_status rq_append_rows(const rq_cache_desc* desc, int32_t layer, const int32_t* pos_dev,
                         const void* k_new, const void* v_new, void* residual,
                         const int8_t* signs_dev, const uint8_t* bits_dev,
                         const uint64_t* offsets_dev, void* packed, uint32_t* status_dev,
                         void* stream);

/* Decode attention with one token count per batch row: row b attends its
 * first n_dev[b] tokens (device int32 [B], 4-byte aligned; 1 <= n <= desc->S):
 * the packed blocks below 32 * (n / 32) and the last n % 32 from its residual
 * windows, as rq_decode_attention_len does for one n. residual is required.
 * The split plan is that of the capacity desc->S; each row's splits stop at
 * its own packed length. A count outside 1..desc->S sets
 * RQ_STATUS_BAD_POSITION and that row's output is 0. Workspace and other
 * arguments as rq_decode_attention_len. */
rq_status rq_decode_attention_rows(const rq_cache_desc* desc, int32_t layer, const int32_t* n_dev,
                                   const void* q, const void* packed, const uint8_t* bits_dev,
                                   const uint64_t* offsets_dev, const int8_t* signs_dev,
                                   const void* residual, float* out, void* ws, size_t ws_bytes,
                                   uint32_t* status_dev, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* RQ_H */
