// Device code of the quantizer (quantize + bit-pack one layer of the KV cache
// at per-head bit-widths) and the pieces the distortion sweep shares with it.
// Each (dtype, rotation) instance of quantize_pack_kernel is compiled in its
// own translation unit (quantize_k_*.cu), in parallel.
//
// RateQuant (arXiv 2605.06675): the quantizer kernel reads the per-head
// bit-width from the static allocation table (App. M "No runtime overhead",
// App. U "Runtime Analysis"); keys are quantized per channel and values per
// token (KIVI, Sec. 2 and App. W), optionally after a per-token Hadamard
// rotation (QuaRot, App. W "QuaRot kernel"); the sweep measures the MSE at
// every b for the fit of D(b) = alpha beta^-b (Alg. 1 stage 2, Sec. 3.4).
//
// quantize_pack_kernel: persistent CTAs of 128 threads; a CTA walks a
// contiguous range of 32-token x 128-channel tiles (one packed block each)
// one stream at a time, each stream with a loop compiled for its layout and
// width; a tile is staged raw in shared memory by cp.async one tile ahead.
// Per tile:
//   phase 1, one group per thread: min / max with NaN-propagating fp16x2 or
//     bf16x2 compares on the raw values, the group's fp16 scale and zero
//     (its meta words go straight to global memory) and (-zero, 1/scale)
//     into a shared table;
//   phase 2, one unit of the packed format (16 two-code registers of one
//     decoder lane, format.cuh) per thread: code = low bits of
//     RN(fp32(v - zero) * inv + 1.5 * 2^23) (fp32x2 add + fma), two codes
//     per register by one byte permute, OR-ed into the unit's words, stored
//     with vector stores. Codes never pass through shared memory.
// Phase 1 flags a tile whose codes could leave [0, largest code], or that holds a
// degenerate group; such a tile takes the clamping variant of phase 2.
// Lloyd-Max groups (per token): phase 1 computes the group's RMS scale, phase 2
// finds each code by a binary search over the scaled level midpoints.
#pragma once

#include <algorithm>
#include <cstddef>

#include "format.cuh"
#include "rq_internal.cuh"

namespace rq {

// kernel arguments (shared by the translation units)
struct QuantArgs {
  const void* k;
  const void* v;
  const int8_t* signs;
  const uint8_t* bits;       // [L][H][2]
  const uint64_t* offsets;   // [L][B][H][2]
  uint8_t* packed;
  uint32_t* status;
  int layer, B, H, S, nblk, kg, vg, hadamard;   // kg, vg: the stored grouping
  int kspan, vspan;          // groups of 32 channels per per-token group (1, 2 or 4)
  int kq, vq;                // rq_quantizer of keys / values
  int j_dst0;                // packed block index of each stream's first tile
  const int32_t* row_pos;    // decode-time append per batch row (or null): the window of row
                             // b is packed as block row_pos[b] / 32 when row_pos[b] % 32 == 31
                             // and 0 <= row_pos[b] < cap, and skipped otherwise
  int cap;                   // the cache's capacity in tokens (row_pos only)
  long long ntiles;
  LMBook lm;                 // RQ_LLOYDMAX codebooks
};

struct CalibArgs {
  const void* x;             // [n][T][128]
  const int8_t* signs;
  double* partial;           // [n][T/32][8]
  uint32_t* status;
  int n, T, ntile, kg, vg, hadamard;   // kg, vg: the stored grouping
  int kspan, vspan;          // groups of 32 channels per per-token group (1, 2 or 4)
  int kq, vq;                // rq_quantizer of keys / values
  long long ntiles;
  LMBook lm;                 // RQ_LLOYDMAX codebooks
};

// one launcher per quantize_pack_kernel instance (quantize_k_*.cu)
rq_status launch_quantize_f16(const QuantArgs& a, cudaStream_t s);
rq_status launch_quantize_f16_rot(const QuantArgs& a, cudaStream_t s);
rq_status launch_quantize_bf16(const QuantArgs& a, cudaStream_t s);
rq_status launch_quantize_bf16_rot(const QuantArgs& a, cudaStream_t s);
// the same, when both kinds of the layer are Lloyd-Max
rq_status launch_quantize_lm_f16(const QuantArgs& a, cudaStream_t s);
rq_status launch_quantize_lm_f16_rot(const QuantArgs& a, cudaStream_t s);
rq_status launch_quantize_lm_bf16(const QuantArgs& a, cudaStream_t s);
rq_status launch_quantize_lm_bf16_rot(const QuantArgs& a, cudaStream_t s);

namespace {

constexpr int kThreads = 128;
// CTAs per SM the quantizer's register budget is sized for: 6 (80 registers)
// measured faster than 8 (64 registers, spilling) or 4-5 on GB300
#ifndef RQ_QUANT_MIN_BLOCKS
#define RQ_QUANT_MIN_BLOCKS 6
#endif
// staged tile row: 256 bytes of values + 64 bytes, so that rows 1 apart land
// 16 banks apart (conflict-free 16-byte reads of neighbouring tokens)
constexpr int kRowBytes = 320;
constexpr int kTileBytes = kTile * kRowBytes;
// Rotated fp32 tile: channel c of token t at x32_at(t, c) = 164 t + c. The
// row stride (4 mod 32 banks) keeps reads of neighbouring tokens apart; the
// four quarters of a token are written in the chunk order i ^ G of
// phase1_rotated, which puts each quarter-warp's 16-byte stores on distinct
// banks.
constexpr int kX32S = 164;
__device__ __forceinline__ int x32_at(int t, int c) { return t * kX32S + c; }

// layouts: keys per channel / per token, values per token / per channel, and
// the Lloyd-Max codebook quantizer on per-token keys / values
enum { kModeKC = 0, kModeKT = 1, kModeVT = 2, kModeVC = 3, kModeKTL = 4, kModeVTL = 5 };

// 16-byte multiple: the rotated fp32 tile follows it (float4 accesses)
struct alignas(16) QSmem {
  uint8_t tile[2][kTileBytes];
  float nz[kD];                 // -zero of every group (channel c, or 32 G + t)
  float inv[kD];                // 1 / scale (0 for a group without codes)
  union {
    uint2 xchg[kThreads];       // per-channel min/max of half the tokens (rotated tiles)
    uint8_t lm_lut[1024];       // Lloyd-Max kernel (per-token groups only): code bucket of x / scale
  };
  float top;                    // magic + the largest code of the tile's quantizer
  float lm_mid[257];            // Lloyd-Max: midpoints of the width's levels (+inf after, Lloyd-Max kernel)
  alignas(16) uint32_t negw[4][16];   // rotation signs (read as uint4): word k of row G flips the sign bits (15, 31)
                                //   of the raw pair of channels 32 G + 2k, 32 G + 2k + 1
};

static_assert(sizeof(QSmem) % 16 == 0, "the rotated tile after QSmem must stay 16-byte aligned");
static_assert(offsetof(QSmem, tile) % 16 == 0 && offsetof(QSmem, negw) % 16 == 0 &&
              offsetof(QSmem, xchg) % 16 == 0, "16-byte shared-memory accesses");

// sm.top, read where it is used (a volatile load from a fixed shared address,
// so the clamping variant keeps no register for it)
__device__ __forceinline__ float clamp_top() {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  return *reinterpret_cast<volatile const float*>(smem_raw + offsetof(QSmem, top));
}



// ------------------------------------------------------------- helpers ----

__device__ __forceinline__ float fmin_nan(float a, float b) {
  float r;
  asm("min.NaN.f32 %0, %1, %2;" : "=f"(r) : "f"(a), "f"(b));
  return r;
}
__device__ __forceinline__ float fmax_nan(float a, float b) {
  float r;
  asm("max.NaN.f32 %0, %1, %2;" : "=f"(r) : "f"(a), "f"(b));
  return r;
}
__device__ __forceinline__ float fmin3_nan(float a, float b, float c) {
  float r;
  asm("min.NaN.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
  return r;
}
__device__ __forceinline__ float fmax3_nan(float a, float b, float c) {
  float r;
  asm("max.NaN.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
  return r;
}

// min / max of a wide per-token group (64 or 128 channels of one token) from
// its quarters: thread 4 t + G holds quarter G (channels 32 G .. 32 G + 31) of
// token t; span 2 joins quarters (0, 1) and (2, 3), span 4 all four (NaN
// propagates). Every lane of the warp takes part.
__device__ __forceinline__ void join_quarters(float& mn, float& mx, int span) {
  if (span >= 2) {
    mn = fmin_nan(mn, __shfl_xor_sync(0xffffffffu, mn, 1));
    mx = fmax_nan(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
  }
  if (span >= 4) {
    mn = fmin_nan(mn, __shfl_xor_sync(0xffffffffu, mn, 2));
    mx = fmax_nan(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
  }
}

// NaN-propagating min / max of two packed 16-bit pairs
template <typename T>
__device__ __forceinline__ uint32_t min2_nan(uint32_t a, uint32_t b);
template <typename T>
__device__ __forceinline__ uint32_t max2_nan(uint32_t a, uint32_t b);
template <>
__device__ __forceinline__ uint32_t min2_nan<__nv_bfloat16>(uint32_t a, uint32_t b) {
  uint32_t r;
  asm("min.NaN.bf16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
  return r;
}
template <>
__device__ __forceinline__ uint32_t max2_nan<__nv_bfloat16>(uint32_t a, uint32_t b) {
  uint32_t r;
  asm("max.NaN.bf16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
  return r;
}
template <>
__device__ __forceinline__ uint32_t min2_nan<__half>(uint32_t a, uint32_t b) {
  uint32_t r;
  asm("min.NaN.f16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
  return r;
}
template <>
__device__ __forceinline__ uint32_t max2_nan<__half>(uint32_t a, uint32_t b) {
  uint32_t r;
  asm("max.NaN.f16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
  return r;
}

// the low / high 16-bit value of a packed pair as fp32 (exact)
template <typename T>
__device__ __forceinline__ float lo_f32(uint32_t w);
template <typename T>
__device__ __forceinline__ float hi_f32(uint32_t w);
template <>
__device__ __forceinline__ float lo_f32<__nv_bfloat16>(uint32_t w) { return __uint_as_float(w << 16); }
template <>
__device__ __forceinline__ float hi_f32<__nv_bfloat16>(uint32_t w) {
  return __uint_as_float(w & 0xFFFF0000u);
}
template <>
__device__ __forceinline__ float lo_f32<__half>(uint32_t w) {
  return __half2float(__ushort_as_half(static_cast<unsigned short>(w & 0xFFFFu)));
}
template <>
__device__ __forceinline__ float hi_f32<__half>(uint32_t w) {
  return __half2float(__ushort_as_half(static_cast<unsigned short>(w >> 16)));
}

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(dst), "l"(src));
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::); }
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_group 0;\n" ::); }

// the 8 KB tile into a staging buffer: thread tau copies 16-byte chunks
// tau + 128 i (row = chunk / 16)
__device__ __forceinline__ void issue_tile(uint8_t* buf, const void* src) {
  const uint32_t dst = smem_u32(buf);
  const uint8_t* s = static_cast<const uint8_t*>(src);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int ch = threadIdx.x + kThreads * i;
    cp_async16(dst + (ch >> 4) * kRowBytes + 16 * (ch & 15), s + 16 * ch);
  }
}

// ------------------------------------------------------------- phase 1 ----
// phase 1's grouping argument: RQ_PER_TOKEN, RQ_PER_CHANNEL, or per-token
// Lloyd-Max groups
constexpr int kGroupingLM = 2;

struct GroupOut {
  bool slow, bad;
};

// quantizer of a tile at b bits: absmax when SYM, else min-max
template <bool SYM>
struct TileQ {
  int b;
};

// Scale/zero of one group: meta words to global memory (packed format),
// (-zero, 1/scale) to the table. `slow`: no codes (bad or zero range) or
// codes that could fall outside [0, cmax] (they are monotone in v, so the
// group's min and max bound them).
template <bool SYM>
__device__ __forceinline__ GroupOut finish_group(int kind, int grouping, int t, int G, int c,
                                                 float mn, float mx, bool finite, TileQ<SYM> q,
                                                 uint8_t* meta, QSmem& sm) {
  const GroupParams g = group_params(mn, mx, finite, q.b, SYM);
  const uint32_t sb = __half_as_ushort(g.scale), zb = __half_as_ushort(g.zero);
  uint16_t* m16 = reinterpret_cast<uint16_t*>(meta);
  uint32_t* m32 = reinterpret_cast<uint32_t*>(meta);
  int slot;
  if (grouping == RQ_PER_CHANNEL) {
    slot = c;
    if (kind == 0) {                          // pair P = c / 2: zeros at word 2P, scales at 2P + 1
      const int P = c >> 1, hh = c & 1;
      m16[4 * P + 2 + hh] = static_cast<uint16_t>(sb);
      m16[4 * P + hh] = static_cast<uint16_t>(zb);
    } else {
      m32[c] = sb | (zb << 16);
    }
  } else {
    slot = 32 * G + t;
    if (kind == 0) {
      m32[16 * (t & 7) + 4 * G + (t >> 3)] = sb | (zb << 16);
    } else {                                  // scale / zero pairs of tokens (t, t^1)
      const int Q = t >> 1;
      const int zw = 64 + 32 * (Q >> 3) + 8 * (Q & 3) + 4 * (G >> 1) + 2 * ((Q >> 2) & 1) + (G & 1);
      m16[2 * (4 * Q + G) + (t & 1)] = static_cast<uint16_t>(sb);
      m16[2 * zw + (t & 1)] = static_cast<uint16_t>(zb);
    }
  }
  sm.nz[slot] = -g.zf;
  sm.inv[slot] = g.inv;
  GroupOut o;
  o.bad = g.bad;
  if (!g.ok) {
    o.slow = true;
    return o;
  }
  const float um = __fmaf_rn(__fsub_rn(mn, g.zf), g.inv, kRoundMagic);
  const float uM = __fmaf_rn(__fsub_rn(mx, g.zf), g.inv, kRoundMagic);
  o.slow = um < kRoundMagic || uM > kRoundMagic + g.cmax;
  return o;
}

// Lloyd-Max group (per-token groups only): scale = fp16(sqrt(s2 / 32)) of the
// fp32 sum of squares s2 = (v0^2 + ... + v15^2) + (v16^2 + ... + v31^2), each
// half summed in order; zero = +0. The table gets sf (codes come from the
// thresholds mid * sf). No clamping variant is needed.
__device__ __forceinline__ float sumsq16(const float* v) {
  float s = 0.0f;
#pragma unroll
  for (int i = 0; i < 16; ++i) s = __fadd_rn(s, __fmul_rn(v[i], v[i]));
  return s;
}

__device__ __forceinline__ GroupOut finish_group_lm(int kind, int t, int G, const float (&v)[kG],
                                                    bool finite, uint8_t* meta, QSmem& sm) {
  const float s2 = __fadd_rn(sumsq16(v), sumsq16(v + 16));
  const float rms = __fsqrt_rn(__fmul_rn(s2, 0.03125f));
  __half scale = __float2half_rn(rms);
  float sf = __half2float(scale);
  GroupOut o;
  o.bad = !finite || !isfinite(sf);
  o.slow = false;
  if (o.bad) {
    scale = __float2half_rn(0.0f);
    sf = 0.0f;
  }
  const uint32_t sb = __half_as_ushort(scale);
  uint16_t* m16 = reinterpret_cast<uint16_t*>(meta);
  uint32_t* m32 = reinterpret_cast<uint32_t*>(meta);
  if (kind == 0) {
    m32[16 * (t & 7) + 4 * G + (t >> 3)] = sb;            // (scale, zero = +0)
  } else {
    const int Q = t >> 1;
    const int zw = 64 + 32 * (Q >> 3) + 8 * (Q & 3) + 4 * (G >> 1) + 2 * ((Q >> 2) & 1) + (G & 1);
    m16[2 * (4 * Q + G) + (t & 1)] = static_cast<uint16_t>(sb);
    m16[2 * zw + (t & 1)] = 0;
  }
  sm.nz[32 * G + t] = sf;
  return o;
}

// per-token Lloyd-Max groups on the raw tile: thread 4 t + G, values in order
template <typename T>
__device__ __forceinline__ GroupOut phase1_rows_lm(const uint8_t* tile, int kind, uint8_t* meta,
                                                   QSmem& sm) {
  const int tau = threadIdx.x, t = tau >> 2, G = tau & 3;
  const uint8_t* row = tile + t * kRowBytes + 64 * G;
  float v[kG];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const uint4 u = *reinterpret_cast<const uint4*>(row + 16 * i);
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      v[8 * i + 2 * e] = lo_f32<T>(w[e]);
      v[8 * i + 2 * e + 1] = hi_f32<T>(w[e]);
    }
  }
  bool finite = true;
#pragma unroll
  for (int i = 0; i < kG; ++i) {
    finite = finite && isfinite(v[i]);
    v[i] = __fadd_rn(v[i], 0.0f);
  }
  return finish_group_lm(kind, t, G, v, finite, meta, sm);
}

// Per-channel groups on the raw tile: thread 2p + hv (channel pair p, token
// half hv) takes channels 2p, 2p+1 over 16 tokens; the two halves of a pair
// are neighbouring lanes and meet by one shuffle, and the thread finishes
// channel 2p + hv. Half 1 walks its rows starting one row later, which puts
// the two halves of a warp's read on disjoint banks (rows are 80 words apart).
template <typename T, bool SYM>
__device__ __forceinline__ GroupOut phase1_cols(const uint8_t* tile, int kind, TileQ<SYM> q,
                                                uint8_t* meta, QSmem& sm) {
  const int tau = threadIdx.x, p = tau >> 1, hv = tau & 1;
  const uint8_t* col = tile + 4 * p + hv * 16 * kRowBytes;
  uint32_t mn2 = *reinterpret_cast<const uint32_t*>(col + hv * kRowBytes), mx2 = mn2;
#pragma unroll
  for (int i = 1; i < 16; ++i) {
    const uint32_t x = *reinterpret_cast<const uint32_t*>(col + ((i + hv) & 15) * kRowBytes);
    mn2 = min2_nan<T>(mn2, x);
    mx2 = max2_nan<T>(mx2, x);
  }
  mn2 = min2_nan<T>(mn2, __shfl_xor_sync(0xffffffffu, mn2, 1));
  mx2 = max2_nan<T>(mx2, __shfl_xor_sync(0xffffffffu, mx2, 1));
  float mn = hv ? hi_f32<T>(mn2) : lo_f32<T>(mn2);
  float mx = hv ? hi_f32<T>(mx2) : lo_f32<T>(mx2);
  const bool finite = isfinite(mn) && isfinite(mx);
  mn = __fadd_rn(mn, 0.0f);     // -0 -> +0
  mx = __fadd_rn(mx, 0.0f);
  return finish_group(kind, RQ_PER_CHANNEL, 0, 0, tau, mn, mx, finite, q, meta, sm);
}

// Per-token groups on the raw tile: thread 4 t + G takes token t, channels
// 32 G .. 32 G + 31 as four 16-byte reads in the chunk order i ^ G, which
// puts the eight threads of a quarter-warp (two tokens x four quarters, rows
// 320 bytes apart) on eight distinct 16-byte bank groups; min / max do not
// depend on the order.
template <typename T, bool SYM>
__device__ __forceinline__ GroupOut phase1_rows(const uint8_t* tile, int kind, TileQ<SYM> q,
                                                uint8_t* meta, QSmem& sm, int span) {
  const int tau = threadIdx.x, t = tau >> 2, G = tau & 3;
  const uint8_t* row = tile + t * kRowBytes + 64 * G;
  uint32_t w[16];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const uint4 u = *reinterpret_cast<const uint4*>(row + 16 * (i ^ G));
    w[4 * i] = u.x;
    w[4 * i + 1] = u.y;
    w[4 * i + 2] = u.z;
    w[4 * i + 3] = u.w;
  }
  uint32_t lo[8], hi[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    lo[i] = min2_nan<T>(w[2 * i], w[2 * i + 1]);
    hi[i] = max2_nan<T>(w[2 * i], w[2 * i + 1]);
  }
#pragma unroll
  for (int s = 4; s >= 1; s >>= 1)
#pragma unroll
    for (int i = 0; i < s; ++i) {
      lo[i] = min2_nan<T>(lo[i], lo[i + s]);
      hi[i] = max2_nan<T>(hi[i], hi[i + s]);
    }
  float mn = fmin_nan(lo_f32<T>(lo[0]), hi_f32<T>(lo[0]));
  float mx = fmax_nan(lo_f32<T>(hi[0]), hi_f32<T>(hi[0]));
  join_quarters(mn, mx, span);
  const bool finite = isfinite(mn) && isfinite(mx);
  mn = __fadd_rn(mn, 0.0f);
  mx = __fadd_rn(mx, 0.0f);
  return finish_group(kind, RQ_PER_TOKEN, t, G, 0, mn, mx, finite, q, meta, sm);
}

// min / max of 32 fp32 values; NaN propagates. Three-input min / max
// (exact and order-free): 32 -> 12 -> 4 -> 2 -> 1 values, 16 each.
__device__ __forceinline__ void minmax32(const float (&v)[kG], float& mn, float& mx) {
  float lo[12], hi[12];
#pragma unroll
  for (int i = 0; i < 10; ++i) {
    lo[i] = fmin3_nan(v[3 * i], v[3 * i + 1], v[3 * i + 2]);
    hi[i] = fmax3_nan(v[3 * i], v[3 * i + 1], v[3 * i + 2]);
  }
  lo[10] = hi[10] = v[30];
  lo[11] = hi[11] = v[31];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    lo[i] = fmin3_nan(lo[3 * i], lo[3 * i + 1], lo[3 * i + 2]);
    hi[i] = fmax3_nan(hi[3 * i], hi[3 * i + 1], hi[3 * i + 2]);
  }
  mn = fmin_nan(fmin3_nan(lo[0], lo[1], lo[2]), lo[3]);
  mx = fmax_nan(fmax3_nan(hi[0], hi[1], hi[2]), hi[3]);
}

// RN(a - b) per component: the product b * -1 is exact and the fused add
// rounds once (no fp32x2 subtract instruction)
__device__ __forceinline__ float2 fsub2_rn(float2 a, float2 b) {
  return __ffma2_rn(b, make_float2(-1.0f, -1.0f), a);
}

// the butterflies of rotate_group on values whose signs are already applied.
// Stride 1 pairs the two halves of a register pair, so it runs on scalars;
// strides 2..16 and the two lane stages run on pairs (v[2k], v[2k + 1]) with
// fp32x2 instructions, each component rounded exactly as the scalar form.
__device__ __forceinline__ void rotate_group_signed(float (&v)[kG], int G) {
  float2 p[kG / 2];
#pragma unroll
  for (int k = 0; k < kG / 2; ++k)
    p[k] = make_float2(__fadd_rn(v[2 * k], v[2 * k + 1]), __fsub_rn(v[2 * k], v[2 * k + 1]));
#pragma unroll
  for (int h = 1; h < kG / 2; h <<= 1) {
#pragma unroll
    for (int k = 0; k < kG / 2; ++k) {
      if (k & h) continue;
      const float2 a = p[k], b = p[k + h];
      p[k] = __fadd2_rn(a, b);
      p[k + h] = fsub2_rn(a, b);
    }
  }
#pragma unroll
  for (int s = 1; s <= 2; s <<= 1) {
    // lower channel of a pair: v + o; upper: o - v; both as fma(v, +-1, o)
    const float sg = (G & s) ? -1.0f : 1.0f;
    const float2 sg2 = make_float2(sg, sg);
#pragma unroll
    for (int k = 0; k < kG / 2; ++k) {
      const float2 o = make_float2(__shfl_xor_sync(0xffffffffu, p[k].x, s),
                                   __shfl_xor_sync(0xffffffffu, p[k].y, s));
      p[k] = __ffma2_rn(p[k], sg2, o);
    }
  }
  const float2 r = make_float2(kInvSqrt128, kInvSqrt128);
#pragma unroll
  for (int k = 0; k < kG / 2; ++k) {
    const float2 y = __fmul2_rn(p[k], r);
    v[2 * k] = y.x;
    v[2 * k + 1] = y.y;
  }
}

// y = FWHT(x * sigma) / sqrt(128) of token t's channels 32 G .. 32 G + 31
// held by thread 4 t + G: butterflies of stride 1..16 in registers, strides
// 32 and 64 with the lanes holding G ^ 1, G ^ 2 (the lower channel of a
// pair takes a + b, the upper a - b), in that order.
__device__ __forceinline__ void rotate_group(float (&v)[kG], int G, const int8_t* signs) {
#pragma unroll
  for (int i = 0; i < kG; ++i)
    if (signs[32 * G + i] < 0) v[i] = -v[i];
  rotate_group_signed(v, G);
}

// Strides 1 .. 16 of the FWHT of a thread's quarter whose 8-value chunks are
// permuted: slot 8 i + j holds channel 32 G + 8 (i ^ G) + j. Strides 1, 2, 4
// are as in rotate_group_signed. At strides 8 and 16 the lower channel of a
// slot pair sits in the upper slot when bit 0 / bit 1 of G is set, so each
// output is fma(own, +-1, other) with the lane's signs (the same single
// rounding as a + b, a - b). The values stay unscaled; strides 32 and 64
// follow in rotate_lanes_x32.
__device__ __forceinline__ void rotate_quarter_perm(float (&v)[kG], int G) {
  float2 p[kG / 2];
#pragma unroll
  for (int k = 0; k < kG / 2; ++k)
    p[k] = make_float2(__fadd_rn(v[2 * k], v[2 * k + 1]), __fsub_rn(v[2 * k], v[2 * k + 1]));
#pragma unroll
  for (int h = 1; h <= 2; h <<= 1) {          // strides 2, 4
#pragma unroll
    for (int k = 0; k < kG / 2; ++k) {
      if (k & h) continue;
      const float2 a = p[k], b = p[k + h];
      p[k] = __fadd2_rn(a, b);
      p[k + h] = fsub2_rn(a, b);
    }
  }
#pragma unroll
  for (int h = 4; h <= 8; h <<= 1) {          // strides 8, 16
    const float sg = (G & (h >> 2)) ? -1.0f : 1.0f;
    const float2 s2 = make_float2(sg, sg), n2 = make_float2(-sg, -sg);
#pragma unroll
    for (int k = 0; k < kG / 2; ++k) {
      if (k & h) continue;
      const float2 a = p[k], b = p[k + h];
      p[k] = __ffma2_rn(a, s2, b);
      p[k + h] = __ffma2_rn(b, n2, a);
    }
  }
#pragma unroll
  for (int k = 0; k < kG / 2; ++k) {
    v[2 * k] = p[k].x;
    v[2 * k + 1] = p[k].y;
  }
}

// Strides 32 and 64 of token t's FWHT through the fp32 tile, in place: the
// four quarters (after strides 1 .. 16) are in x32; thread 4 t + G takes
// channel offsets 8 G .. 8 G + 7 of all four quarters, runs stride 32 on the
// quarter pairs (0, 1), (2, 3) and stride 64 on (0, 2), (1, 3) (the
// oracle's butterfly order, each output one fp32 rounding), scales by
// fp32(1/sqrt(128)) and writes the results back to the same places. The four
// threads of a token are consecutive lanes, so a warp barrier orders the
// exchange; the 16-byte accesses of a quarter-warp fall on distinct bank
// groups (rows 164 words apart). Returns each quarter's min / max over the
// thread's eight values.
__device__ __forceinline__ void rotate_lanes_x32(float* x32, int t, int G, float (&mnq)[4],
                                                 float (&mxq)[4]) {
  __syncwarp();
  float2 y[4][4];                            // [quarter][pair of offsets]
#pragma unroll
  for (int Q = 0; Q < 4; ++Q) {
    const float* src = x32 + x32_at(t, 32 * Q + 8 * G);
    const float4 a = *reinterpret_cast<const float4*>(src);
    const float4 b = *reinterpret_cast<const float4*>(src + 4);
    y[Q][0] = make_float2(a.x, a.y);
    y[Q][1] = make_float2(a.z, a.w);
    y[Q][2] = make_float2(b.x, b.y);
    y[Q][3] = make_float2(b.z, b.w);
  }
  const float2 r = make_float2(kInvSqrt128, kInvSqrt128);
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const float2 s01 = __fadd2_rn(y[0][k], y[1][k]), d01 = fsub2_rn(y[0][k], y[1][k]);
    const float2 s23 = __fadd2_rn(y[2][k], y[3][k]), d23 = fsub2_rn(y[2][k], y[3][k]);
    y[0][k] = __fmul2_rn(__fadd2_rn(s01, s23), r);
    y[2][k] = __fmul2_rn(fsub2_rn(s01, s23), r);
    y[1][k] = __fmul2_rn(__fadd2_rn(d01, d23), r);
    y[3][k] = __fmul2_rn(fsub2_rn(d01, d23), r);
  }
#pragma unroll
  for (int Q = 0; Q < 4; ++Q) {
    float* dst = x32 + x32_at(t, 32 * Q + 8 * G);
    *reinterpret_cast<float4*>(dst) = make_float4(y[Q][0].x, y[Q][0].y, y[Q][1].x, y[Q][1].y);
    *reinterpret_cast<float4*>(dst + 4) = make_float4(y[Q][2].x, y[Q][2].y, y[Q][3].x, y[Q][3].y);
    mnq[Q] = fmin_nan(fmin3_nan(fmin3_nan(y[Q][0].x, y[Q][0].y, y[Q][1].x), y[Q][1].y, y[Q][2].x),
                      fmin3_nan(y[Q][2].y, y[Q][3].x, y[Q][3].y));
    mxq[Q] = fmax_nan(fmax3_nan(fmax3_nan(y[Q][0].x, y[Q][0].y, y[Q][1].x), y[Q][1].y, y[Q][2].x),
                      fmax3_nan(y[Q][2].y, y[Q][3].x, y[Q][3].y));
  }
}

// Rotated tiles: every thread rotates one 32-channel quarter of a token and
// writes it to the fp32 tile x32; groups are then formed on x32. The thread
// takes its quarter's 16-byte chunks in the order i ^ G, which puts the
// reads and writes of each quarter-warp on distinct banks.
template <typename T, bool SYM>
__device__ __forceinline__ GroupOut phase1_rotated(const uint8_t* tile, float* x32, int kind,
                                                   int grouping, TileQ<SYM> q, uint8_t* meta,
                                                   QSmem& sm, int span) {
  const int tau = threadIdx.x, t = tau >> 2, G = tau & 3;
  float v[kG];
  const uint8_t* row = tile + t * kRowBytes + 64 * G;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    // sign flips on the raw pairs (bits 15 and 31 are the two signs)
    const int c = i ^ G;
    const uint4 u = *reinterpret_cast<const uint4*>(row + 16 * c);
    const uint4 n = *reinterpret_cast<const uint4*>(&sm.negw[G][4 * c]);
    const uint32_t w[4] = {u.x ^ n.x, u.y ^ n.y, u.z ^ n.z, u.w ^ n.w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      v[8 * i + 2 * e] = lo_f32<T>(w[e]);
      v[8 * i + 2 * e + 1] = hi_f32<T>(w[e]);
    }
  }
  rotate_quarter_perm(v, G);
  float* xr = x32 + x32_at(t, 32 * G);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    float* xc = xr + 8 * (i ^ G);
    *reinterpret_cast<float4*>(xc) = make_float4(v[8 * i], v[8 * i + 1], v[8 * i + 2], v[8 * i + 3]);
    *reinterpret_cast<float4*>(xc + 4) =
        make_float4(v[8 * i + 4], v[8 * i + 5], v[8 * i + 6], v[8 * i + 7]);
  }
  float mnq[4], mxq[4];
  rotate_lanes_x32(x32, t, G, mnq, mxq);
  if (grouping == RQ_PER_TOKEN) {             // min / max: any order
    // reduce-scatter over the token's four threads: thread G ends with
    // quarter G's min / max (lane G ^ 2 first takes the other half of the
    // quarters, lane G ^ 1 then the other quarter of the pair); wide
    // groups then join quarters as in the plain layout
    float mn, mx;
    {
      const bool h = G & 2, l = G & 1;
      float a0 = h ? mnq[2] : mnq[0], a1 = h ? mnq[3] : mnq[1];
      float b0 = h ? mxq[2] : mxq[0], b1 = h ? mxq[3] : mxq[1];
      a0 = fmin_nan(a0, __shfl_xor_sync(0xffffffffu, h ? mnq[0] : mnq[2], 2));
      a1 = fmin_nan(a1, __shfl_xor_sync(0xffffffffu, h ? mnq[1] : mnq[3], 2));
      b0 = fmax_nan(b0, __shfl_xor_sync(0xffffffffu, h ? mxq[0] : mxq[2], 2));
      b1 = fmax_nan(b1, __shfl_xor_sync(0xffffffffu, h ? mxq[1] : mxq[3], 2));
      mn = fmin_nan(l ? a1 : a0, __shfl_xor_sync(0xffffffffu, l ? a0 : a1, 1));
      mx = fmax_nan(l ? b1 : b0, __shfl_xor_sync(0xffffffffu, l ? b0 : b1, 1));
    }
    join_quarters(mn, mx, span);
    const bool finite = isfinite(mn) && isfinite(mx);
    return finish_group(kind, RQ_PER_TOKEN, t, G, 0, __fadd_rn(mn, 0.0f), __fadd_rn(mx, 0.0f),
                        finite, q, meta, sm);
  }
  if (grouping == kGroupingLM) {            // Lloyd-Max, per token, on the rotated values
    // the sum of squares is ordered: the quarter back from x32 in channel order
    // (written by the token's four threads)
    __syncwarp();
#pragma unroll
    for (int i = 0; i < kG; i += 4) {
      const float4 y = *reinterpret_cast<const float4*>(xr + i);
      v[i] = y.x;
      v[i + 1] = y.y;
      v[i + 2] = y.z;
      v[i + 3] = y.w;
    }
    bool finite = true;
#pragma unroll
    for (int i = 0; i < kG; ++i) {
      finite = finite && isfinite(v[i]);
      v[i] = __fadd_rn(v[i], 0.0f);
    }
    return finish_group_lm(kind, t, G, v, finite, meta, sm);
  }
  __syncthreads();
  const int p = tau & 63, hv = tau >> 6;
  const float* col = x32 + x32_at(16 * hv, 2 * p);
  float2 lo = *reinterpret_cast<const float2*>(col), hi = lo;
#pragma unroll
  for (int i = 1; i < 16; ++i) {
    const float2 x = *reinterpret_cast<const float2*>(col + i * kX32S);
    lo = make_float2(fmin_nan(lo.x, x.x), fmin_nan(lo.y, x.y));
    hi = make_float2(fmax_nan(hi.x, x.x), fmax_nan(hi.y, x.y));
  }
  const float mnh = hv ? lo.y : lo.x, mxh = hv ? hi.y : hi.x;
  sm.xchg[tau] = make_uint2(__float_as_uint(hv ? lo.x : lo.y), __float_as_uint(hv ? hi.x : hi.y));
  __syncthreads();
  // the partner (other token half) left this thread's channel in xchg
  const uint2 o = sm.xchg[tau ^ 64];
  const float mn = fmin_nan(mnh, __uint_as_float(o.x));
  const float mx = fmax_nan(mxh, __uint_as_float(o.y));
  const bool finite = isfinite(mn) && isfinite(mx);
  return finish_group(kind, RQ_PER_CHANNEL, 0, 0, 2 * p + hv, __fadd_rn(mn, 0.0f),
                      __fadd_rn(mx, 0.0f), finite, q, meta, sm);
}

// The rotated phase 1 is large (the FWHT unrolled over 32 values) and runs
// once per tile: one out-of-line copy per (dtype, quantizer form), shared by
// every layout and width, keeps the kernel's code within the instruction
// cache. Shared memory is re-derived from the dynamic-shared symbol so its
// accesses stay shared-memory instructions.
template <typename T, bool SYM>
__device__ __noinline__ GroupOut phase1_rot_call(int buf, int kind, int grouping, int b,
                                                 uint8_t* meta, int span) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  QSmem& sm = *reinterpret_cast<QSmem*>(smem_raw);
  float* x32 = reinterpret_cast<float*>(smem_raw + sizeof(QSmem));
  const TileQ<SYM> q{b};
  return phase1_rotated<T>(sm.tile[buf], x32, kind, grouping, q, meta, sm, span);
}

template <typename T, bool HAD, bool SYM>
__device__ __forceinline__ GroupOut phase1(const uint8_t* tile, float* x32, int kind, int grouping,
                                              int b, uint8_t* meta, QSmem& sm, int buf, int span) {
  const TileQ<SYM> q{b};
  if constexpr (HAD) return phase1_rot_call<T, SYM>(buf, kind, grouping, b, meta, span);
  else if (grouping == kGroupingLM) return phase1_rows_lm<T>(tile, kind, meta, sm);
  else if (grouping == RQ_PER_CHANNEL) return phase1_cols<T>(tile, kind, q, meta, sm);
  else return phase1_rows<T>(tile, kind, q, meta, sm, span);
}

// ------------------------------------------------------------- phase 2 ----

// four channel pairs (c .. c + 7) of token t as fp32 pairs
template <typename T, bool F32>
__device__ __forceinline__ void load_pairs(const uint8_t* tile, const float* x32, int t, int c,
                                           float2 (&v)[4]) {
  if constexpr (F32) {
    const float4 a = *reinterpret_cast<const float4*>(x32 + x32_at(t, c));
    const float4 b = *reinterpret_cast<const float4*>(x32 + x32_at(t, c) + 4);
    v[0] = make_float2(a.x, a.y);
    v[1] = make_float2(a.z, a.w);
    v[2] = make_float2(b.x, b.y);
    v[3] = make_float2(b.z, b.w);
  } else {
    const uint4 u = *reinterpret_cast<const uint4*>(tile + t * kRowBytes + 2 * c);
    v[0] = make_float2(lo_f32<T>(u.x), hi_f32<T>(u.x));
    v[1] = make_float2(lo_f32<T>(u.y), hi_f32<T>(u.y));
    v[2] = make_float2(lo_f32<T>(u.z), hi_f32<T>(u.z));
    v[3] = make_float2(lo_f32<T>(u.w), hi_f32<T>(u.w));
  }
}

// four channels (c .. c + 3) of token t as fp32
template <typename T, bool F32>
__device__ __forceinline__ void load_quad(const uint8_t* tile, const float* x32, int t, int c,
                                          float (&v)[4]) {
  if constexpr (F32) {
    const float4 a = *reinterpret_cast<const float4*>(x32 + x32_at(t, c));
    v[0] = a.x;
    v[1] = a.y;
    v[2] = a.z;
    v[3] = a.w;
  } else {
    const uint2 u = *reinterpret_cast<const uint2*>(tile + t * kRowBytes + 2 * c);
    v[0] = lo_f32<T>(u.x);
    v[1] = hi_f32<T>(u.x);
    v[2] = lo_f32<T>(u.y);
    v[3] = hi_f32<T>(u.y);
  }
}

// codes of register (x, y) from its two values: RN(fp32(v - zero) * inv +
// magic) has the code in its low byte (and 0 in the next) when in range
template <int B, bool CLAMP>
__device__ __forceinline__ void emit(uint32_t (&uw)[B], int x, int y, float2 v, float2 nz,
                                     float2 iv) {
  const float2 d = __fadd2_rn(v, nz);
  float2 q = __ffma2_rn(d, iv, make_float2(kRoundMagic, kRoundMagic));
  if constexpr (CLAMP) {
    q.x = fminf(fmaxf(q.x, kRoundMagic), clamp_top());
    q.y = fminf(fmaxf(q.y, kRoundMagic), clamp_top());
  }
  fmt::place<B>(uw, x, y, __byte_perm(__float_as_uint(q.x), __float_as_uint(q.y), 0x5410u));
}

// Lloyd-Max code: the number of thresholds fp32(mid_i * sf), i = 0..2^B - 2,
// at or below v (binary search over the ascending thresholds); 0 for a group
// without a scale
template <int B>
__device__ __forceinline__ uint32_t lm_code(float v, float sf, const float* mid) {
  int c = 0;
#pragma unroll
  for (int k = B - 1; k >= 0; --k) {
    const int cand = c + (1 << k);
    c = v >= __fmul_rn(mid[cand - 1], sf) ? cand : c;
  }
  return sf != 0.0f ? static_cast<uint32_t>(c) : 0u;
}

template <int B>
__device__ __forceinline__ void emit_lm(uint32_t (&uw)[B], int x, int y, float2 v, float2 sf,
                                        const float* mid) {
  fmt::place<B>(uw, x, y, lm_code<B>(v.x, sf.x, mid) | (lm_code<B>(v.y, sf.y, mid) << 16));
}

// The same code in the Lloyd-Max kernel (every stream of the layer Lloyd-Max),
// found in two steps: the bucket of u = v / sf among 1024 equal bins over
// [-5, 5) (lm_lut: c0 = the number of midpoints below the bin's lower edge by
// more than 1e-5), then one exact comparison with threshold c0. Exact because
// no window [edge_k - 1e-5, edge_k+1 + 1e-5) holds more than one of the
// codebooks' fp32 midpoints (the narrowest gap, at 8 bits, is 0.0169 against
// bins of 0.0098; none lies beyond +-4.4), while u and the thresholds are
// within 2e-6 of their exact values; a host test checks the property on the
// library's codebooks. (In the general kernel this code's extra registers
// raised the spills of the min-max loops, so it has a kernel of its own.)
constexpr int kLmBins = 1024;
constexpr float kLmBinScale = 102.4f;          // bins per unit of u
constexpr float kLmBinStep = 0.009765625f;     // 1 / 102.4, exact
constexpr float kLmDelta = 1e-5f;

template <int B>
__device__ __forceinline__ uint32_t lm_code_lut(float v, float sf, float inv, const float* mid,
                                                const uint8_t* lut) {
  const float t = __fmaf_rn(__fmul_rn(v, inv), kLmBinScale, 0.5f * kLmBins);
  const int k = min(max(__float2int_rd(t), 0), kLmBins - 1);
  const int c0 = lut[k];
  const int c = c0 + (v >= __fmul_rn(mid[c0], sf) ? 1 : 0);
  return sf != 0.0f ? static_cast<uint32_t>(c) : 0u;
}

template <int B, bool LUT>
__device__ __forceinline__ void emit_lm2(uint32_t (&uw)[B], int x, int y, float2 v, float2 sf,
                                         float2 inv, const QSmem& sm) {
  if constexpr (LUT)
    fmt::place<B>(uw, x, y, lm_code_lut<B>(v.x, sf.x, inv.x, sm.lm_mid, sm.lm_lut) |
                                (lm_code_lut<B>(v.y, sf.y, inv.y, sm.lm_mid, sm.lm_lut) << 16));
  else
    emit_lm<B>(uw, x, y, v, sf, sm.lm_mid);
}

// lm_lut from the segment's midpoints (sm.lm_mid, nmid of them): bin kb gets
// the number of midpoints below its lower edge by more than kLmDelta.
__device__ __forceinline__ void lm_lut_build(QSmem& sm, int nmid) {
  for (int kb = threadIdx.x; kb < kLmBins; kb += kThreads) {
    const float e = __fsub_rn(static_cast<float>(kb - kLmBins / 2) * kLmBinStep, kLmDelta);
    int lo = 0, hi = nmid;
    while (lo < hi) {
      const int md = (lo + hi) >> 1;
      if (sm.lm_mid[md] < e) lo = md + 1;
      else hi = md;
    }
    sm.lm_lut[kb] = static_cast<uint8_t>(lo);
  }
}

// Thread -> (lane gid/tig of the packed format, unit u). K: warp = unit,
// lane = format lane. V: a half warp is (gid 0..7) x (two units), so the
// 8-byte reads of one token row hit 16 distinct bank pairs.
template <int MODE, typename T, int B, bool CLAMP, bool F32, bool LUT = false>
__device__ __forceinline__ void phase2(const uint8_t* tile, const float* x32, const QSmem& sm,
                                       uint32_t* blk) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int gid, tig, u;
  if (MODE == kModeKC || MODE == kModeKT || MODE == kModeKTL) {
    gid = lane >> 2;
    tig = lane & 3;
    u = warp;
  } else {
    gid = lane & 7;
    u = 2 * (warp & 1) + ((lane >> 3) & 1);
    tig = 2 * (warp >> 1) + (lane >> 4);
  }
  uint32_t uw[B];
#pragma unroll
  for (int i = 0; i < B; ++i) uw[i] = 0u;

  if constexpr (MODE == kModeKC) {
    // channels 32u + 8tig + 2x + h, token 8y + gid; group = channel
    const int c = 32 * u + 8 * tig;
    const float4 z0 = *reinterpret_cast<const float4*>(sm.nz + c);
    const float4 z1 = *reinterpret_cast<const float4*>(sm.nz + c + 4);
    const float4 i0 = *reinterpret_cast<const float4*>(sm.inv + c);
    const float4 i1 = *reinterpret_cast<const float4*>(sm.inv + c + 4);
    const float2 nz[4] = {make_float2(z0.x, z0.y), make_float2(z0.z, z0.w),
                          make_float2(z1.x, z1.y), make_float2(z1.z, z1.w)};
    const float2 iv[4] = {make_float2(i0.x, i0.y), make_float2(i0.z, i0.w),
                          make_float2(i1.x, i1.y), make_float2(i1.z, i1.w)};
#pragma unroll
    for (int y = 0; y < 4; ++y) {
      float2 v[4];
      load_pairs<T, F32>(tile, x32, 8 * y + gid, c, v);
#pragma unroll
      for (int x = 0; x < 4; ++x) emit<B, CLAMP>(uw, x, y, v[x], nz[x], iv[x]);
    }
  } else if constexpr (MODE == kModeKTL) {
    // as kModeKT, codes from the Lloyd-Max thresholds (the table holds sf)
    const int c = 32 * u + 8 * tig;
#pragma unroll
    for (int x = 0; x < 4; ++x) {
      const int t = 8 * x + gid;
      const float sf = sm.nz[32 * u + t], inv = LUT ? __frcp_rn(sf) : 0.0f;
      float2 v[4];
      load_pairs<T, F32>(tile, x32, t, c, v);
#pragma unroll
      for (int y = 0; y < 4; ++y)
        emit_lm2<B, LUT>(uw, x, y, v[y], make_float2(sf, sf), make_float2(inv, inv), sm);
    }
  } else if constexpr (MODE == kModeKT) {
    // token 8x + gid, channels 32u + 8tig + 2y + h; group = (token, G = u)
    const int c = 32 * u + 8 * tig;
#pragma unroll
    for (int x = 0; x < 4; ++x) {
      const int t = 8 * x + gid;
      const float z = sm.nz[32 * u + t], i = sm.inv[32 * u + t];
      float2 v[4];
      load_pairs<T, F32>(tile, x32, t, c, v);
#pragma unroll
      for (int y = 0; y < 4; ++y) emit<B, CLAMP>(uw, x, y, v[y], make_float2(z, z), make_float2(i, i));
    }
  } else {
    // channel 32u + 4gid + x, tokens 8y + 2tig + h
    const int c = 32 * u + 4 * gid;
    float4 zc, ic;
    if constexpr (MODE == kModeVC) {
      zc = *reinterpret_cast<const float4*>(sm.nz + c);
      ic = *reinterpret_cast<const float4*>(sm.inv + c);
    }
#pragma unroll
    for (int y = 0; y < 4; ++y) {
      const int t = 8 * y + 2 * tig;
      float a[4], b[4];
      load_quad<T, F32>(tile, x32, t, c, a);
      load_quad<T, F32>(tile, x32, t + 1, c, b);
      if constexpr (MODE == kModeVTL) {
        const float2 sf = *reinterpret_cast<const float2*>(sm.nz + 32 * u + t);
        const float2 inv = LUT ? make_float2(__frcp_rn(sf.x), __frcp_rn(sf.y)) : make_float2(0.0f, 0.0f);
#pragma unroll
        for (int x = 0; x < 4; ++x) emit_lm2<B, LUT>(uw, x, y, make_float2(a[x], b[x]), sf, inv, sm);
      } else if constexpr (MODE == kModeVT) {
        const float2 nz = *reinterpret_cast<const float2*>(sm.nz + 32 * u + t);
        const float2 iv = *reinterpret_cast<const float2*>(sm.inv + 32 * u + t);
#pragma unroll
        for (int x = 0; x < 4; ++x) emit<B, CLAMP>(uw, x, y, make_float2(a[x], b[x]), nz, iv);
      } else {
        const float zz[4] = {zc.x, zc.y, zc.z, zc.w}, ii[4] = {ic.x, ic.y, ic.z, ic.w};
#pragma unroll
        for (int x = 0; x < 4; ++x)
          emit<B, CLAMP>(uw, x, y, make_float2(a[x], b[x]), make_float2(zz[x], zz[x]),
                         make_float2(ii[x], ii[x]));
      }
    }
  }

  // lane word w = B u + i of lane L lives at block word 128 (w / 4) + 4 L + w % 4
  const int L = 4 * gid + tig;
  if constexpr (B == 2) {
    const int w = 2 * u;
    *reinterpret_cast<uint2*>(blk + 128 * (w >> 2) + 4 * L + (w & 3)) = make_uint2(uw[0], uw[1]);
  } else if constexpr (B == 4) {
    *reinterpret_cast<uint4*>(blk + 128 * u + 4 * L) = make_uint4(uw[0], uw[1], uw[2], uw[3]);
  } else if constexpr (B == 8) {
    *reinterpret_cast<uint4*>(blk + 128 * (2 * u) + 4 * L) = make_uint4(uw[0], uw[1], uw[2], uw[3]);
    *reinterpret_cast<uint4*>(blk + 128 * (2 * u + 1) + 4 * L) = make_uint4(uw[4], uw[5], uw[6], uw[7]);
  } else {
#pragma unroll
    for (int i = 0; i < B; ++i) {
      const int w = B * u + i;
      blk[128 * (w >> 2) + 4 * L + (w & 3)] = uw[i];
    }
  }
}

// The clamping variant of phase 2 (rare: degenerate groups, codes that could
// leave their range): out of line, so each layout and width carries one
// inlined phase 2 only.
template <int MODE, typename T, int B, bool F32>
__device__ __noinline__ void phase2_clamp_call(int buf, uint32_t* blk) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  const QSmem& sm = *reinterpret_cast<const QSmem*>(smem_raw);
  const float* x32 = F32 ? reinterpret_cast<const float*>(smem_raw + sizeof(QSmem)) : nullptr;
  phase2<MODE, T, B, true, F32>(sm.tile[buf], x32, sm, blk);
}

// Per-stream constants (recomputed when the walk crosses into a stream).
struct StreamState {
  const uint8_t* src;     // first tile of the stream (raw values)
  uint8_t* dst;           // first packed block of the stream
  int b, kind, grouping;
  bool skip;              // row_pos: this row's window is not full (nothing to write)
};

template <typename T>
__device__ __forceinline__ StreamState stream_state(const QuantArgs& a, int sk) {
  StreamState st;
  st.kind = sk & 1;
  const int h = (sk >> 1) % a.H;
  st.b = a.bits[(a.layer * a.H + h) * 2 + st.kind];
  st.grouping = st.kind ? a.vg : a.kg;
  st.src = reinterpret_cast<const uint8_t*>(static_cast<const T*>(st.kind ? a.v : a.k) +
                                            static_cast<long long>(sk >> 1) * a.S * kD);
  int j = a.j_dst0;
  st.skip = false;
  if (a.row_pos) {
    const int p = a.row_pos[(sk >> 1) / a.H];
    st.skip = !(p >= 0 && p < a.cap && p % kTile == kTile - 1);
    j = st.skip ? 0 : p / kTile;
  }
  // offsets[layer][batch][h][kind] = offsets[layer * B * H * 2 + sk]
  st.dst = a.packed + a.offsets[static_cast<long long>(a.layer) * a.B * a.H * 2 + sk] +
           static_cast<long long>(j) * (512 * (st.b + 1));
  return st;
}

// The tiles a CTA walks inside one stream: n tiles from src (raw) to dst
// (packed blocks), ring position `it` (tile buffer it & 1 holds the first,
// already issued), and the first tile after the segment (null: none).
struct Segment {
  const uint8_t* src;
  uint8_t* dst;
  const uint8_t* next;
  int n;
};

__host__ __device__ constexpr int mode_of(int kind, int grouping, bool lloydmax) {
  return lloydmax ? (kind == 0 ? kModeKTL : kModeVTL)
                  : kind == 0 ? (grouping == RQ_PER_CHANNEL ? kModeKC : kModeKT)
                              : (grouping == RQ_PER_TOKEN ? kModeVT : kModeVC);
}

// One stream's tiles with the layout (MODE) and width (B) fixed at compile
// time: per tile, wait for it, prefetch the next, phase 1 (group
// parameters, meta words), phase 2 (codes) in the clamping variant only when
// phase 1 flagged the tile. Returns the ring position after the segment.
template <typename T, bool HAD, int MODE, int B, bool LUT = false>
__device__ __forceinline__ int run_segment(const QuantArgs& a, QSmem& sm, float* x32,
                                           const Segment& seg, int it) {
  constexpr int kTileSrcBytes = kTile * kD * static_cast<int>(sizeof(T));
  constexpr int kBlkBytes = 512 * (B + 1);
  constexpr int kind = (MODE == kModeKC || MODE == kModeKT || MODE == kModeKTL) ? 0 : 1;
  constexpr bool LM = MODE == kModeKTL || MODE == kModeVTL;
  constexpr int grouping = LM ? kGroupingLM
                              : (MODE == kModeKC || MODE == kModeVC) ? RQ_PER_CHANNEL : RQ_PER_TOKEN;
  const bool sym = (kind ? a.vq : a.kq) == RQ_ABSMAX;      // kernel parameters, no register
  for (int k = 0; k < seg.n; ++k, ++it) {
    const uint8_t* buf = sm.tile[it & 1];
    cp_async_wait_all();
    __syncthreads();             // tile visible; every thread is past the previous tile
    if (k + 1 < seg.n) issue_tile(sm.tile[(it + 1) & 1], seg.src + static_cast<long long>(k + 1) * kTileSrcBytes);
    else if (seg.next) issue_tile(sm.tile[(it + 1) & 1], seg.next);
    cp_async_commit();
    uint8_t* blk = seg.dst + static_cast<long long>(k) * kBlkBytes;
    uint8_t* meta = blk + 512 * B;
    if (threadIdx.x == 0)        // read by phase 2, after the barrier below
      sm.top = kRoundMagic + static_cast<float>(sym ? (1 << B) - 2 : (1 << B) - 1);
    if constexpr (LM && !LUT) {  // the thresholds' midpoints, exact in fp32
      for (int i = threadIdx.x; i < (1 << B) - 1; i += kThreads) {
        const float l0 = __half2float(__ushort_as_half(a.lm.lv[lm_offset(B) + i]));
        const float l1 = __half2float(__ushort_as_half(a.lm.lv[lm_offset(B) + i + 1]));
        sm.lm_mid[i] = __fmul_rn(__fadd_rn(l0, l1), 0.5f);
      }
    }
    if constexpr (LM && LUT) {
      if (k == 0) {              // once per segment (one width): midpoints, then buckets
        for (int i = threadIdx.x; i < (1 << B); i += kThreads) {
          float m = INFINITY;    // exact in fp32; +inf after the last
          if (i < (1 << B) - 1) {
            const float l0 = __half2float(__ushort_as_half(a.lm.lv[lm_offset(B) + i]));
            const float l1 = __half2float(__ushort_as_half(a.lm.lv[lm_offset(B) + i + 1]));
            m = __fmul_rn(__fadd_rn(l0, l1), 0.5f);
          }
          sm.lm_mid[i] = m;
        }
        __syncthreads();
        lm_lut_build(sm, (1 << B) - 1);
      }
    }
    GroupOut g;
    const int span = kind ? a.vspan : a.kspan;             // kernel parameters, no register
    if (sym) g = phase1<T, HAD, true>(buf, x32, kind, grouping, B, meta, sm, it & 1, span);
    else g = phase1<T, HAD, false>(buf, x32, kind, grouping, B, meta, sm, it & 1, span);
    if (g.bad) set_status(a.status, RQ_STATUS_NUMERIC);
    const bool slow = __syncthreads_or(g.slow) != 0;
    uint32_t* blk32 = reinterpret_cast<uint32_t*>(blk);
    if (slow) phase2_clamp_call<MODE, T, B, HAD>(it & 1, blk32);
    else phase2<MODE, T, B, false, HAD, LUT>(buf, x32, sm, blk32);
  }
  return it;
}

// a stream whose device bit-width is outside 1..8 (reported), or a window
// with nothing to pack: keep the tile pipeline going, write nothing
__device__ __forceinline__ int skip_segment(const QuantArgs& a, QSmem& sm, const Segment& seg,
                                            int it, int tile_bytes, bool report) {
  for (int k = 0; k < seg.n; ++k, ++it) {
    cp_async_wait_all();
    __syncthreads();
    if (k + 1 < seg.n) issue_tile(sm.tile[(it + 1) & 1], seg.src + static_cast<long long>(k + 1) * tile_bytes);
    else if (seg.next) issue_tile(sm.tile[(it + 1) & 1], seg.next);
    cp_async_commit();
  }
  if (report && threadIdx.x == 0) set_status(a.status, RQ_STATUS_BAD_BITS);
  return it;
}

template <typename T, bool HAD, int MODE, bool LUT = false>
__device__ __forceinline__ int run_segment_b(const QuantArgs& a, QSmem& sm, float* x32,
                                             const Segment& seg, int it, int b) {
  switch (b) {
    case 1: return run_segment<T, HAD, MODE, 1, LUT>(a, sm, x32, seg, it);
    case 2: return run_segment<T, HAD, MODE, 2, LUT>(a, sm, x32, seg, it);
    case 3: return run_segment<T, HAD, MODE, 3, LUT>(a, sm, x32, seg, it);
    case 4: return run_segment<T, HAD, MODE, 4, LUT>(a, sm, x32, seg, it);
    case 5: return run_segment<T, HAD, MODE, 5, LUT>(a, sm, x32, seg, it);
    case 6: return run_segment<T, HAD, MODE, 6, LUT>(a, sm, x32, seg, it);
    case 7: return run_segment<T, HAD, MODE, 7, LUT>(a, sm, x32, seg, it);
    default: return run_segment<T, HAD, MODE, 8, LUT>(a, sm, x32, seg, it);
  }
}

// A CTA owns a contiguous range of tiles (block j of stream sk = (batch * H
// + h) * 2 + kind, tile index sk * nblk + j); the range is walked one stream
// segment at a time, each with its own compile-time loop.
// LMK: the Lloyd-Max kernel, launched when both kinds of the layer are
// Lloyd-Max (every segment then is); it holds the Lloyd-Max loops only.
template <typename T, bool HAD, bool LMK = false>
__global__ void __launch_bounds__(kThreads, RQ_QUANT_MIN_BLOCKS) quantize_pack_kernel(QuantArgs a) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  QSmem& sm = *reinterpret_cast<QSmem*>(smem_raw);
  float* x32 = HAD ? reinterpret_cast<float*>(smem_raw + sizeof(QSmem)) : nullptr;
  const long long t0 = a.ntiles * blockIdx.x / gridDim.x;
  const long long t1 = a.ntiles * (blockIdx.x + 1) / gridDim.x;
  if (t0 >= t1) return;
  if (HAD) {                     // warp w's ballot is the sign mask of channels 32 w .. 32 w + 31
    const bool neg = a.signs && a.signs[threadIdx.x] < 0;
    const uint32_t m = __ballot_sync(0xffffffffu, neg);
    const int k = threadIdx.x & 31;
    if (k < 16)
      sm.negw[threadIdx.x >> 5][k] = ((m >> (2 * k)) & 1u) << 15 | ((m >> (2 * k + 1)) & 1u) << 31;
  }

  const int nblk = a.nblk;
  constexpr int kTileSrcBytes = kTile * kD * static_cast<int>(sizeof(T));
  int sk = static_cast<int>(t0 / nblk), j = static_cast<int>(t0 % nblk);
  StreamState cur = stream_state<T>(a, sk);
  issue_tile(sm.tile[0], cur.src + static_cast<long long>(j) * kTileSrcBytes);
  cp_async_commit();
  int it = 0;
  for (long long t = t0; t < t1;) {
    const long long end = t1 < static_cast<long long>(sk + 1) * nblk ? t1 : static_cast<long long>(sk + 1) * nblk;
    const bool more = end < t1;
    const StreamState nxt = more ? stream_state<T>(a, sk + 1) : cur;
    Segment seg;
    seg.src = cur.src + static_cast<long long>(j) * kTileSrcBytes;
    seg.dst = cur.dst + static_cast<long long>(j) * (512 * (cur.b + 1));
    seg.next = more ? nxt.src : nullptr;
    seg.n = static_cast<int>(end - t);
    const int b = cur.b;
    if (cur.skip || b < 1 || b > 8) {
      it = skip_segment(a, sm, seg, it, kTileSrcBytes, !cur.skip);
    } else {
      const bool lm = (cur.kind ? a.vq : a.kq) == RQ_LLOYDMAX;
      if constexpr (LMK) {
        if (cur.kind == 0) it = run_segment_b<T, HAD, kModeKTL, true>(a, sm, x32, seg, it, b);
        else it = run_segment_b<T, HAD, kModeVTL, true>(a, sm, x32, seg, it, b);
      } else {
        switch (mode_of(cur.kind, cur.grouping, lm)) {
          case kModeKC: it = run_segment_b<T, HAD, kModeKC>(a, sm, x32, seg, it, b); break;
          case kModeKT: it = run_segment_b<T, HAD, kModeKT>(a, sm, x32, seg, it, b); break;
          case kModeVT: it = run_segment_b<T, HAD, kModeVT>(a, sm, x32, seg, it, b); break;
          case kModeKTL: it = run_segment_b<T, HAD, kModeKTL>(a, sm, x32, seg, it, b); break;
          case kModeVTL: it = run_segment_b<T, HAD, kModeVTL>(a, sm, x32, seg, it, b); break;
          default: it = run_segment_b<T, HAD, kModeVC>(a, sm, x32, seg, it, b); break;
        }
      }
    }
    t = end;
    ++sk;
    j = 0;
    cur = nxt;
  }
}


template <typename Kern, typename Args>
rq_status launch_persistent(Kern kern, const Args& a, size_t smem, cudaStream_t stream) {
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(smem)) != cudaSuccess)
    return RQ_ERR_CUDA;
  int sms = 0;
  if (current_sm_count(&sms) != RQ_OK) return RQ_ERR_CUDA;
  int per_sm = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kThreads, smem) != cudaSuccess)
    return RQ_ERR_CUDA;
  per_sm = std::max(per_sm, 1);
  const long long grid = std::min<long long>(a.ntiles, static_cast<long long>(sms) * per_sm);
  kern<<<static_cast<unsigned>(grid), kThreads, smem, stream>>>(a);
  return launch_status();
}

inline size_t quant_smem_bytes(bool hadamard) {
  return sizeof(QSmem) + (hadamard ? kTile * kX32S * sizeof(float) : 0);
}

}  // namespace
}  // namespace rq
