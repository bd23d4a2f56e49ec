// Quantize + bit-pack one layer of the KV cache at per-head bit-widths, and
// the distortion sweep that calibrates D(b) per component.
//
// RateQuant (arXiv 2605.06675): the quantizer kernel reads the per-head
// bit-width from the static allocation table (App. M "No runtime overhead",
// App. U "Runtime Analysis"); keys are quantized per channel and values per
// token (KIVI, Sec. 2 and App. W), optionally after a per-token Hadamard
// rotation (QuaRot, App. W "QuaRot kernel"); the sweep measures the MSE at
// every b for the fit of D(b) = alpha beta^-b (Alg. 1 stage 2, Sec. 3.4).
//
// quantize_pack_kernel: persistent CTAs of 128 threads; a CTA owns one
// 32-token x 128-channel tile (one packed block) at a time, staged raw in
// shared memory by cp.async one tile ahead. Per tile:
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
#include <algorithm>

#include "format.cuh"
#include "rq_internal.cuh"

namespace rq {
namespace {

constexpr int kThreads = 128;
// CTAs per SM the quantizer's register budget is sized for
#ifndef RQ_QUANT_MIN_BLOCKS
#define RQ_QUANT_MIN_BLOCKS 8
#endif
// staged tile row: 256 bytes of values + 64 bytes, so that rows 1 apart land
// 16 banks apart (conflict-free 16-byte reads of neighbouring tokens)
constexpr int kRowBytes = 320;
constexpr int kTileBytes = kTile * kRowBytes;
constexpr int kX32S = kD + 4;           // rotated fp32 row (floats)

enum { kModeKC = 0, kModeKT = 1, kModeVT = 2, kModeVC = 3 };

// 16-byte multiple: the rotated fp32 tile follows it (float4 accesses)
struct alignas(16) QSmem {
  uint8_t tile[2][kTileBytes];
  float nz[kD];                 // -zero of every group (channel c, or 32 G + t)
  float inv[kD];                // 1 / scale (0 for a group without codes)
  uint2 xchg[kThreads];         // per-channel min/max of half the tokens
  float top;                    // magic + the largest code of the tile's quantizer
  int8_t signs[kD];
};

static_assert(sizeof(QSmem) % 16 == 0, "the rotated tile after QSmem must stay 16-byte aligned");

// sm.top, read where it is used (a volatile load from a fixed shared address,
// so the clamping variant keeps no register for it)
__device__ __forceinline__ float clamp_top() {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  return *reinterpret_cast<volatile const float*>(smem_raw + offsetof(QSmem, top));
}

struct QuantArgs {
  const void* k;
  const void* v;
  const int8_t* signs;
  const uint8_t* bits;       // [L][H][2]
  const uint64_t* offsets;   // [L][B][H][2]
  uint8_t* packed;
  uint32_t* status;
  int layer, B, H, S, nblk, kg, vg, hadamard;
  int kq, vq;                // rq_quantizer of keys / values
  int j_dst0;                // packed block index of each stream's first tile
  long long ntiles;
};

struct CalibArgs {
  const void* x;             // [n][T][128]
  const int8_t* signs;
  double* partial;           // [n][T/32][8]
  uint32_t* status;
  int n, T, ntile, kg, vg, hadamard;
  int kq, vq;                // rq_quantizer of keys / values
  long long ntiles;
};

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

// Per-channel groups on the raw tile: thread (pair p, token half hv) takes
// channels 2p, 2p+1 over tokens 16 hv .. 16 hv + 15, the two halves meet
// through shared memory, and the thread finishes channel 2p + hv.
template <typename T, bool SYM>
__device__ __forceinline__ GroupOut phase1_cols(const uint8_t* tile, int kind, TileQ<SYM> q,
                                                uint8_t* meta, QSmem& sm) {
  const int tau = threadIdx.x, p = tau & 63, hv = tau >> 6;
  const uint8_t* col = tile + 4 * p + hv * 16 * kRowBytes;
  uint32_t mn2 = *reinterpret_cast<const uint32_t*>(col), mx2 = mn2;
#pragma unroll
  for (int i = 1; i < 16; ++i) {
    const uint32_t x = *reinterpret_cast<const uint32_t*>(col + i * kRowBytes);
    mn2 = min2_nan<T>(mn2, x);
    mx2 = max2_nan<T>(mx2, x);
  }
  sm.xchg[tau] = make_uint2(mn2, mx2);
  __syncthreads();
  const uint2 o = sm.xchg[tau ^ 64];
  mn2 = min2_nan<T>(mn2, o.x);
  mx2 = max2_nan<T>(mx2, o.y);
  float mn = hv ? hi_f32<T>(mn2) : lo_f32<T>(mn2);
  float mx = hv ? hi_f32<T>(mx2) : lo_f32<T>(mx2);
  const bool finite = isfinite(mn) && isfinite(mx);
  mn = __fadd_rn(mn, 0.0f);     // -0 -> +0
  mx = __fadd_rn(mx, 0.0f);
  return finish_group(kind, RQ_PER_CHANNEL, 0, 0, 2 * p + hv, mn, mx, finite, q, meta, sm);
}

// Per-token groups on the raw tile: thread 4 t + G takes token t, channels
// 32 G .. 32 G + 31 (four 16-byte reads, started at a rotating chunk so the
// eight threads of a read phase hit distinct banks).
template <typename T, bool SYM>
__device__ __forceinline__ GroupOut phase1_rows(const uint8_t* tile, int kind, TileQ<SYM> q,
                                                uint8_t* meta, QSmem& sm) {
  const int tau = threadIdx.x, t = tau >> 2, G = tau & 3;
  const uint8_t* row = tile + t * kRowBytes + 64 * G;
  uint32_t w[16];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const uint4 u = *reinterpret_cast<const uint4*>(row + 16 * ((i + (t >> 1)) & 3));
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
  const bool finite = isfinite(mn) && isfinite(mx);
  mn = __fadd_rn(mn, 0.0f);
  mx = __fadd_rn(mx, 0.0f);
  return finish_group(kind, RQ_PER_TOKEN, t, G, 0, mn, mx, finite, q, meta, sm);
}

// min / max of 32 fp32 values; NaN propagates
__device__ __forceinline__ void minmax32(const float (&v)[kG], float& mn, float& mx) {
  float lo[16], hi[16];
#pragma unroll
  for (int i = 0; i < 16; ++i) {
    lo[i] = fmin_nan(v[2 * i], v[2 * i + 1]);
    hi[i] = fmax_nan(v[2 * i], v[2 * i + 1]);
  }
#pragma unroll
  for (int w = 8; w >= 1; w >>= 1)
#pragma unroll
    for (int i = 0; i < w; ++i) {
      lo[i] = fmin_nan(lo[i], lo[i + w]);
      hi[i] = fmax_nan(hi[i], hi[i + w]);
    }
  mn = lo[0];
  mx = hi[0];
}

// y = FWHT(x * sigma) / sqrt(128) of token t's channels 32 G .. 32 G + 31
// held by thread 4 t + G: butterflies of stride 1..16 in registers, strides
// 32 and 64 with the lanes holding G ^ 1, G ^ 2 (the lower channel of a
// pair takes a + b, the upper a - b), in that order.
__device__ __forceinline__ void rotate_group(float (&v)[kG], int G, const int8_t* signs) {
#pragma unroll
  for (int i = 0; i < kG; ++i)
    if (signs[32 * G + i] < 0) v[i] = -v[i];
#pragma unroll
  for (int h = 1; h < kG; h <<= 1) {
#pragma unroll
    for (int i = 0; i < kG; ++i) {
      if (i & h) continue;
      const float a = v[i], b = v[i + h];
      v[i] = __fadd_rn(a, b);
      v[i + h] = __fsub_rn(a, b);
    }
  }
#pragma unroll
  for (int s = 1; s <= 2; s <<= 1) {
    const bool upper = (G & s) != 0;
#pragma unroll
    for (int i = 0; i < kG; ++i) {
      const float o = __shfl_xor_sync(0xffffffffu, v[i], s);
      v[i] = upper ? __fsub_rn(o, v[i]) : __fadd_rn(v[i], o);
    }
  }
#pragma unroll
  for (int i = 0; i < kG; ++i) v[i] = __fmul_rn(v[i], kInvSqrt128);
}

// Rotated tiles: every thread rotates one 32-channel quarter of a token and
// writes it to the fp32 tile x32; groups are then formed on x32.
template <typename T, bool SYM>
__device__ __forceinline__ GroupOut phase1_rotated(const uint8_t* tile, float* x32, int kind,
                                                   int grouping, TileQ<SYM> q, uint8_t* meta,
                                                   QSmem& sm) {
  const int tau = threadIdx.x, t = tau >> 2, G = tau & 3;
  float v[kG];
  const uint8_t* row = tile + t * kRowBytes + 64 * G;
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
  rotate_group(v, G, sm.signs);
  float* xr = x32 + t * kX32S + 32 * G;
#pragma unroll
  for (int i = 0; i < kG; i += 4)
    *reinterpret_cast<float4*>(xr + i) = make_float4(v[i], v[i + 1], v[i + 2], v[i + 3]);
  if (grouping == RQ_PER_TOKEN) {
    float mn, mx;
    minmax32(v, mn, mx);
    const bool finite = isfinite(mn) && isfinite(mx);
    return finish_group(kind, RQ_PER_TOKEN, t, G, 0, __fadd_rn(mn, 0.0f), __fadd_rn(mx, 0.0f),
                        finite, q, meta, sm);
  }
  __syncthreads();
  const int p = tau & 63, hv = tau >> 6;
  const float* col = x32 + 16 * hv * kX32S + 2 * p;
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

template <typename T, bool HAD, bool SYM>
__device__ __forceinline__ GroupOut phase1(const uint8_t* tile, float* x32, int kind, int grouping,
                                           int b, uint8_t* meta, QSmem& sm) {
  const TileQ<SYM> q{b};
  if constexpr (HAD) return phase1_rotated<T>(tile, x32, kind, grouping, q, meta, sm);
  else if (grouping == RQ_PER_CHANNEL) return phase1_cols<T>(tile, kind, q, meta, sm);
  else return phase1_rows<T>(tile, kind, q, meta, sm);
}

// ------------------------------------------------------------- phase 2 ----

// four channel pairs (c .. c + 7) of token t as fp32 pairs
template <typename T, bool F32>
__device__ __forceinline__ void load_pairs(const uint8_t* tile, const float* x32, int t, int c,
                                           float2 (&v)[4]) {
  if constexpr (F32) {
    const float4 a = *reinterpret_cast<const float4*>(x32 + t * kX32S + c);
    const float4 b = *reinterpret_cast<const float4*>(x32 + t * kX32S + c + 4);
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
    const float4 a = *reinterpret_cast<const float4*>(x32 + t * kX32S + c);
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

// Thread -> (lane gid/tig of the packed format, unit u). K: warp = unit,
// lane = format lane. V: a half warp is (gid 0..7) x (two units), so the
// 8-byte reads of one token row hit 16 distinct bank pairs.
template <int MODE, typename T, int B, bool CLAMP, bool F32>
__device__ __forceinline__ void phase2(const uint8_t* tile, const float* x32, const QSmem& sm,
                                       uint32_t* blk) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int gid, tig, u;
  if (MODE == kModeKC || MODE == kModeKT) {
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
      if constexpr (MODE == kModeVT) {
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

template <typename T, bool CLAMP, bool F32>
__device__ __forceinline__ void phase2_dispatch(int mode, int b, const uint8_t* tile,
                                                const float* x32, const QSmem& sm, uint32_t* blk) {
#define RQ_P2_WIDTHS(MODE)                                                          \
  switch (b) {                                                                      \
    case 1: phase2<MODE, T, 1, CLAMP, F32>(tile, x32, sm, blk); break;              \
    case 2: phase2<MODE, T, 2, CLAMP, F32>(tile, x32, sm, blk); break;              \
    case 3: phase2<MODE, T, 3, CLAMP, F32>(tile, x32, sm, blk); break;              \
    case 4: phase2<MODE, T, 4, CLAMP, F32>(tile, x32, sm, blk); break;              \
    case 5: phase2<MODE, T, 5, CLAMP, F32>(tile, x32, sm, blk); break;              \
    case 6: phase2<MODE, T, 6, CLAMP, F32>(tile, x32, sm, blk); break;              \
    case 7: phase2<MODE, T, 7, CLAMP, F32>(tile, x32, sm, blk); break;              \
    default: phase2<MODE, T, 8, CLAMP, F32>(tile, x32, sm, blk); break;             \
  }
  switch (mode) {
    case kModeKC: RQ_P2_WIDTHS(kModeKC) break;
    case kModeKT: RQ_P2_WIDTHS(kModeKT) break;
    case kModeVT: RQ_P2_WIDTHS(kModeVT) break;
    default: RQ_P2_WIDTHS(kModeVC) break;
  }
#undef RQ_P2_WIDTHS
}

// Per-stream constants of the tiles a CTA walks (recomputed only when the
// walk crosses into the next stream).
struct StreamState {
  const uint8_t* src;     // first tile of the stream (raw values)
  uint8_t* dst;           // first packed block of the stream
  int b, kind, grouping, blk_bytes;
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
  // offsets[layer][batch][h][kind] = offsets[layer * B * H * 2 + sk]
  st.blk_bytes = 512 * (st.b + 1);
  st.dst = a.packed + a.offsets[static_cast<long long>(a.layer) * a.B * a.H * 2 + sk] +
           static_cast<long long>(a.j_dst0) * st.blk_bytes;
  return st;
}

// A CTA owns a contiguous range of tiles (block j of stream sk = (batch * H
// + h) * 2 + kind, tile index sk * nblk + j), so consecutive tiles share
// their stream's constants.
template <typename T, bool HAD>
__global__ void __launch_bounds__(kThreads, RQ_QUANT_MIN_BLOCKS) quantize_pack_kernel(QuantArgs a) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  QSmem& sm = *reinterpret_cast<QSmem*>(smem_raw);
  float* x32 = HAD ? reinterpret_cast<float*>(smem_raw + sizeof(QSmem)) : nullptr;
  const long long t0 = a.ntiles * blockIdx.x / gridDim.x;
  const long long t1 = a.ntiles * (blockIdx.x + 1) / gridDim.x;
  if (t0 >= t1) return;
  if (HAD && threadIdx.x < kD) sm.signs[threadIdx.x] = a.signs ? a.signs[threadIdx.x] : int8_t(1);

  const int nblk = a.nblk;
  constexpr int kTileSrcBytes = kTile * kD * static_cast<int>(sizeof(T));
  int sk = static_cast<int>(t0 / nblk), j = static_cast<int>(t0 % nblk);
  StreamState cur = stream_state<T>(a, sk);
  StreamState nxt = cur;
  int nj = j;
  issue_tile(sm.tile[0], cur.src + static_cast<long long>(j) * kTileSrcBytes);
  cp_async_commit();

  for (long long t = t0; t < t1; ++t) {
    const int it = static_cast<int>(t - t0);
    const uint8_t* buf = sm.tile[it & 1];
    cp_async_wait_all();
    __syncthreads();             // tile visible; every thread is past the previous tile
    if (t + 1 < t1) {
      if (++nj == nblk) {
        nj = 0;
        nxt = stream_state<T>(a, ++sk);
      }
      issue_tile(sm.tile[(it + 1) & 1], nxt.src + static_cast<long long>(nj) * kTileSrcBytes);
    }
    cp_async_commit();

    const int b = cur.b;
    if (b >= 1 && b <= 8) {
      uint8_t* blk = cur.dst + static_cast<long long>(j) * cur.blk_bytes;
      uint8_t* meta = blk + 512 * b;
      const int kind = cur.kind, grouping = cur.grouping;
      GroupOut g;
      const bool sym = (kind ? a.vq : a.kq) == RQ_ABSMAX;   // kernel parameters, no register
      if (threadIdx.x == 0)        // read by phase 2, after the barrier below
        sm.top = kRoundMagic + static_cast<float>(sym ? (1 << b) - 2 : (1 << b) - 1);
      if (sym) g = phase1<T, HAD, true>(buf, x32, kind, grouping, b, meta, sm);
      else g = phase1<T, HAD, false>(buf, x32, kind, grouping, b, meta, sm);
      if (g.bad) set_status(a.status, RQ_STATUS_NUMERIC);
      const bool slow = __syncthreads_or(g.slow) != 0;

      const int mode = kind == 0 ? (grouping == RQ_PER_CHANNEL ? kModeKC : kModeKT)
                                 : (grouping == RQ_PER_TOKEN ? kModeVT : kModeVC);
      uint32_t* blk32 = reinterpret_cast<uint32_t*>(blk);
      if (slow) phase2_dispatch<T, true, HAD>(mode, b, buf, x32, sm, blk32);
      else phase2_dispatch<T, false, HAD>(mode, b, buf, x32, sm, blk32);
    } else if (threadIdx.x == 0) {
      set_status(a.status, RQ_STATUS_BAD_BITS);
    }
    j = nj;
    cur = nxt;
  }
}

// ------------------------------------------------------ distortion sweep ----
// Per component and b = 1..8: sum over the component's groups of
// (y - y_hat)^2 with y_hat = fp32(fp32(c * scale) + zero). A group's 32
// squared errors are summed in fp32 (two interleaved partial sums, fixed
// order) and the per-group sums in fp64; per-tile partials are reduced in a
// fixed order (deterministic). One group per thread: per-token groups are
// loaded as rows (thread 4 t + G), per-channel groups as columns of the
// tile staged in shared memory.

struct CalibSmem {
  uint16_t x16[kTile * (kD + 8)];       // raw tile (column mode), rows 272 bytes apart
  int8_t signs[kD];
  double red[kThreads / 32][8];
};
constexpr int kX16Stride = kD + 8;

template <typename T>
__device__ __forceinline__ void calib_load(const T* tile_base, bool row_mode, uint4 (&ld)[4]) {
  const uint4* src = row_mode
      ? reinterpret_cast<const uint4*>(tile_base + (threadIdx.x >> 2) * kD + 32 * (threadIdx.x & 3))
      : reinterpret_cast<const uint4*>(tile_base) + threadIdx.x;
  const int stride = row_mode ? 1 : kThreads;
#pragma unroll
  for (int i = 0; i < 4; ++i) ld[i] = ldg_stream(src + i * stride);
}

// The 32 values of this thread's group in the quantizer's domain (rotated
// when `hadamard`); contains __syncthreads (call uniformly).
template <typename T>
__device__ __forceinline__ void calib_group_values(const uint4 (&ld)[4], bool row_mode,
                                                   int grouping, bool hadamard, CalibSmem& sm,
                                                   float* x32, float (&v)[kG]) {
  const int tau = threadIdx.x;
  if (row_mode) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      float f[8];
      unpack8<T>(ld[i], f);
#pragma unroll
      for (int e = 0; e < 8; ++e) v[8 * i + e] = f[e];
    }
    if (hadamard) {
      rotate_group(v, tau & 3, sm.signs);
      if (grouping == RQ_PER_CHANNEL) {       // regroup the rotated tile by column
        const int t = tau >> 2, G = tau & 3;
#pragma unroll
        for (int i = 0; i < kG; ++i) x32[t * (kD + 1) + 32 * G + i] = v[i];
        __syncthreads();
#pragma unroll
        for (int i = 0; i < kG; ++i) v[i] = x32[i * (kD + 1) + tau];
      }
    }
  } else {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int ch = tau + kThreads * i;
      *reinterpret_cast<uint4*>(&sm.x16[(ch >> 4) * kX16Stride + (ch & 15) * 8]) = ld[i];
    }
    __syncthreads();
#pragma unroll
    for (int i = 0; i < kG; ++i) {
      const uint16_t raw = sm.x16[i * kX16Stride + tau];
      v[i] = to_f32<T>(*reinterpret_cast<const T*>(&raw));
    }
  }
}

template <typename T>
__global__ void __launch_bounds__(kThreads) calib_sweep_kernel(CalibArgs a) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  CalibSmem& sm = *reinterpret_cast<CalibSmem*>(smem_raw);
  float* x32 = reinterpret_cast<float*>(smem_raw + sizeof(CalibSmem));
  const long long stride = gridDim.x;
  long long tile = blockIdx.x;
  if (tile >= a.ntiles) return;
  if (threadIdx.x < kD) sm.signs[threadIdx.x] = a.signs ? a.signs[threadIdx.x] : int8_t(1);
  __syncthreads();
  const bool had = a.hadamard != 0;
  const T* xbase = static_cast<const T*>(a.x);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;

  int grouping = (static_cast<int>(tile / a.ntile) & 1) ? a.vg : a.kg;
  bool sym = ((static_cast<int>(tile / a.ntile) & 1) ? a.vq : a.kq) == RQ_ABSMAX;
  bool row_mode = grouping == RQ_PER_TOKEN || had;
  uint4 ld[4];
  calib_load<T>(xbase + tile * kTile * kD, row_mode, ld);
  for (; tile < a.ntiles; tile += stride) {
    float v[kG];
    calib_group_values<T>(ld, row_mode, grouping, had, sm, x32, v);
    const long long next = tile + stride;
    const bool sym_now = sym;
    if (next < a.ntiles) {
      sym = ((static_cast<int>(next / a.ntile) & 1) ? a.vq : a.kq) == RQ_ABSMAX;
      grouping = (static_cast<int>(next / a.ntile) & 1) ? a.vg : a.kg;
      row_mode = grouping == RQ_PER_TOKEN || had;
      calib_load<T>(xbase + next * kTile * kD, row_mode, ld);
    }
    float mn, mx;
    minmax32(v, mn, mx);
    const bool finite = isfinite(mn) && isfinite(mx);
    mn = __fadd_rn(mn, 0.0f);
    mx = __fadd_rn(mx, 0.0f);
    double acc[8];
#pragma unroll
    for (int b = 1; b <= 8; ++b) {
      const GroupParams g = group_params(mn, mx, finite, b, sym_now);
      if (b == 1 && g.bad) set_status(a.status, RQ_STATUS_NUMERIC);
      const float2 sf = make_float2(g.sf, g.sf), zf = make_float2(g.zf, g.zf);
      float2 s2 = make_float2(0.0f, 0.0f);
#pragma unroll
      for (int i = 0; i < kG; i += 2) {
        // code = clamp(rint(fp32(v - zero) * inv)), one rounding of the product
        const float c0 = round_magic_clamped(__fsub_rn(v[i], g.zf), g.inv, g.cmax) - kRoundMagic;
        const float c1 = round_magic_clamped(__fsub_rn(v[i + 1], g.zf), g.inv, g.cmax) - kRoundMagic;
        const float2 xh = __fadd2_rn(__fmul2_rn(make_float2(c0, c1), sf), zf);
        const float2 e = __fadd2_rn(make_float2(v[i], v[i + 1]), make_float2(-xh.x, -xh.y));
        s2 = __ffma2_rn(e, e, s2);
      }
      acc[b - 1] = static_cast<double>(s2.x) + static_cast<double>(s2.y);
    }
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      double t = acc[k];
#pragma unroll
      for (int o = 16; o >= 1; o >>= 1) t = __dadd_rn(t, __shfl_xor_sync(0xffffffffu, t, o));
      if (lane == 0) sm.red[warp][k] = t;
    }
    __syncthreads();
    if (threadIdx.x < 8) {
      double t = sm.red[0][threadIdx.x];
#pragma unroll
      for (int w = 1; w < kThreads / 32; ++w) t = __dadd_rn(t, sm.red[w][threadIdx.x]);
      a.partial[tile * 8 + threadIdx.x] = t;
    }
    __syncthreads();
  }
}

// mse[i][k] = (sum_j partial[i][j][k], j ascending) / (T * 128)
__global__ void calib_finalize_kernel(const double* partial, double* mse, int n, int ntile,
                                      double count) {
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= n * 8) return;
  const int i = idx >> 3, k = idx & 7;
  double s = 0.0;
  for (int j = 0; j < ntile; ++j) s = __dadd_rn(s, partial[(static_cast<long long>(i) * ntile + j) * 8 + k]);
  mse[idx] = __ddiv_rn(s, count);
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

size_t quant_smem_bytes(bool hadamard) {
  return sizeof(QSmem) + (hadamard ? kTile * kX32S * sizeof(float) : 0);
}

size_t calib_smem_bytes(bool hadamard, int kg, int vg) {
  const bool x32 = hadamard && (kg == RQ_PER_CHANNEL || vg == RQ_PER_CHANNEL);
  return sizeof(CalibSmem) + (x32 ? kTile * (kD + 1) * sizeof(float) : 0);
}

}  // namespace
}  // namespace rq

extern "C" rq_status rq_quantize_pack(const rq_cache_desc* desc, int32_t layer, const void* k,
                                      const void* v, const int8_t* signs_dev,
                                      const uint8_t* bits_dev, const uint64_t* offsets_dev,
                                      void* packed, uint32_t* status_dev, void* stream) {
  using namespace rq;
  if (!desc || !k || !v || !bits_dev || !offsets_dev || !packed) return RQ_ERR_INVALID_ARG;
  if (desc->L <= 0 || desc->B < 0 || desc->H_kv <= 0 || desc->S < 0) return RQ_ERR_INVALID_ARG;
  if (layer < 0 || layer >= desc->L) return RQ_ERR_INVALID_ARG;
  if (desc->dtype != RQ_F16 && desc->dtype != RQ_BF16) return RQ_ERR_INVALID_ARG;
  for (int g : {desc->k_grouping, desc->v_grouping})
    if (g != RQ_PER_TOKEN && g != RQ_PER_CHANNEL) return RQ_ERR_INVALID_ARG;
  for (int qz : {desc->k_quantizer, desc->v_quantizer})
    if (qz != RQ_MINMAX && qz != RQ_ABSMAX) return RQ_ERR_INVALID_ARG;
  if (desc->d != kD || desc->group != kG || desc->S % kTile != 0) return RQ_ERR_SHAPE;
  if (!aligned16(k) || !aligned16(v) || !aligned16(packed)) return RQ_ERR_ALIGNMENT;
  QuantArgs a;
  a.k = k;
  a.v = v;
  a.signs = signs_dev;
  a.bits = bits_dev;
  a.offsets = offsets_dev;
  a.packed = static_cast<uint8_t*>(packed);
  a.status = status_dev;
  a.layer = layer;
  a.B = desc->B;
  a.H = desc->H_kv;
  a.S = desc->S;
  a.nblk = desc->S / kTile;
  a.kg = desc->k_grouping;
  a.vg = desc->v_grouping;
  a.kq = desc->k_quantizer;
  a.vq = desc->v_quantizer;
  a.hadamard = desc->hadamard ? 1 : 0;
  a.j_dst0 = 0;
  a.ntiles = static_cast<long long>(desc->B) * desc->H_kv * 2 * a.nblk;
  if (a.ntiles == 0) return RQ_OK;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const size_t smem = quant_smem_bytes(a.hadamard != 0);
  if (desc->dtype == RQ_F16)
    return a.hadamard ? launch_persistent(quantize_pack_kernel<__half, true>, a, smem, st)
                      : launch_persistent(quantize_pack_kernel<__half, false>, a, smem, st);
  return a.hadamard ? launch_persistent(quantize_pack_kernel<__nv_bfloat16, true>, a, smem, st)
                    : launch_persistent(quantize_pack_kernel<__nv_bfloat16, false>, a, smem, st);
}

extern "C" size_t rq_calibrate_workspace_bytes(int32_t n, int32_t T) {
  if (n <= 0 || T <= 0) return 0;
  return static_cast<size_t>(n) * static_cast<size_t>((T + rq::kTile - 1) / rq::kTile) * 8 *
         sizeof(double);
}

extern "C" rq_status rq_calibrate_distortion(const void* x, int32_t dtype, int32_t n, int32_t T,
                                             int32_t k_grouping, int32_t v_grouping,
                                             int32_t hadamard, int32_t k_quantizer,
                                             int32_t v_quantizer, const int8_t* signs_dev,
                                             double* mse_dev, void* ws, size_t ws_bytes,
                                             uint32_t* status_dev, void* stream) {
  using namespace rq;
  if (!x || !mse_dev || !ws || n <= 0 || T <= 0) return RQ_ERR_INVALID_ARG;
  if (dtype != RQ_F16 && dtype != RQ_BF16) return RQ_ERR_INVALID_ARG;
  for (int g : {k_grouping, v_grouping})
    if (g != RQ_PER_TOKEN && g != RQ_PER_CHANNEL) return RQ_ERR_INVALID_ARG;
  for (int qz : {k_quantizer, v_quantizer})
    if (qz != RQ_MINMAX && qz != RQ_ABSMAX) return RQ_ERR_INVALID_ARG;
  if (T % kTile != 0) return RQ_ERR_SHAPE;
  if (!aligned16(x) || !aligned16(ws) || (reinterpret_cast<uintptr_t>(mse_dev) & 7u))
    return RQ_ERR_ALIGNMENT;
  if (ws_bytes < rq_calibrate_workspace_bytes(n, T)) return RQ_ERR_WORKSPACE;
  CalibArgs a;
  a.x = x;
  a.signs = signs_dev;
  a.partial = static_cast<double*>(ws);
  a.status = status_dev;
  a.n = n;
  a.T = T;
  a.ntile = T / kTile;
  a.kg = k_grouping;
  a.vg = v_grouping;
  a.kq = k_quantizer;
  a.vq = v_quantizer;
  a.hadamard = hadamard ? 1 : 0;
  a.ntiles = static_cast<long long>(n) * a.ntile;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const size_t smem = calib_smem_bytes(a.hadamard != 0, a.kg, a.vg);
  const rq_status s = dtype == RQ_F16
                          ? launch_persistent(calib_sweep_kernel<__half>, a, smem, st)
                          : launch_persistent(calib_sweep_kernel<__nv_bfloat16>, a, smem, st);
  if (s != RQ_OK) return s;
  calib_finalize_kernel<<<(n * 8 + 127) / 128, 128, 0, st>>>(a.partial, mse_dev, n, a.ntile,
                                                              static_cast<double>(T) * kD);
  return launch_status();
}

// ---------------------------------------------------------- decode append ----
// Residual windows: [L][B][H][2][32][128] values, K then V per (layer, batch,
// kv head); token t in slot t % 32. One CTA of 32 threads per (batch, head):
// threads 0..15 copy the new key's 16-byte chunks, 16..31 the value's.
namespace rq {
namespace {

__global__ void append_token_kernel(const uint4* k_new, const uint4* v_new, uint4* residual_layer,
                                    int slot) {
  const int bh = blockIdx.x, t = threadIdx.x, kind = t >> 4, ch = t & 15;
  const uint4* src = (kind ? v_new : k_new) + bh * 16 + ch;
  // 16-byte chunks: a token row is 16, a window 32 * 16, a (batch, head) 2 windows
  residual_layer[(bh * 2 + kind) * 32 * 16 + slot * 16 + ch] = *src;
}

size_t residual_layer_elems(const rq_cache_desc* desc) {
  return static_cast<size_t>(desc->B) * desc->H_kv * 2 * kTile * kD;
}

}  // namespace
}  // namespace rq

extern "C" size_t rq_residual_bytes(const rq_cache_desc* desc) {
  using namespace rq;
  if (!desc || desc->L <= 0 || desc->B < 0 || desc->H_kv <= 0) return 0;
  if (desc->dtype != RQ_F16 && desc->dtype != RQ_BF16) return 0;
  return static_cast<size_t>(desc->L) * residual_layer_elems(desc) * 2;
}

extern "C" rq_status rq_append(const rq_cache_desc* desc, int32_t layer, int32_t pos,
                               const void* k_new, const void* v_new, void* residual,
                               const int8_t* signs_dev, const uint8_t* bits_dev,
                               const uint64_t* offsets_dev, void* packed, uint32_t* status_dev,
                               void* stream) {
  using namespace rq;
  if (!desc || !k_new || !v_new || !residual || !bits_dev || !offsets_dev || !packed)
    return RQ_ERR_INVALID_ARG;
  if (desc->L <= 0 || desc->B < 0 || desc->H_kv <= 0 || desc->S < 0) return RQ_ERR_INVALID_ARG;
  if (layer < 0 || layer >= desc->L || pos < 0 || pos >= desc->S) return RQ_ERR_INVALID_ARG;
  if (desc->dtype != RQ_F16 && desc->dtype != RQ_BF16) return RQ_ERR_INVALID_ARG;
  for (int g : {desc->k_grouping, desc->v_grouping})
    if (g != RQ_PER_TOKEN && g != RQ_PER_CHANNEL) return RQ_ERR_INVALID_ARG;
  for (int qz : {desc->k_quantizer, desc->v_quantizer})
    if (qz != RQ_MINMAX && qz != RQ_ABSMAX) return RQ_ERR_INVALID_ARG;
  if (desc->d != kD || desc->group != kG || desc->S % kTile != 0) return RQ_ERR_SHAPE;
  if (!aligned16(k_new) || !aligned16(v_new) || !aligned16(residual) || !aligned16(packed))
    return RQ_ERR_ALIGNMENT;
  if (desc->B == 0) return RQ_OK;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const size_t layer_bytes = residual_layer_elems(desc) * 2;
  uint8_t* res_layer = static_cast<uint8_t*>(residual) + static_cast<size_t>(layer) * layer_bytes;
  const int slot = pos % kTile;
  append_token_kernel<<<static_cast<unsigned>(desc->B * desc->H_kv), 32, 0, st>>>(
      static_cast<const uint4*>(k_new), static_cast<const uint4*>(v_new),
      reinterpret_cast<uint4*>(res_layer), slot);
  if (launch_status() != RQ_OK) return RQ_ERR_CUDA;
  if (slot != kTile - 1) return RQ_OK;
  // the windows are full: quantize + pack them as block pos / 32 of every
  // stream (a stream's source is its window: K at +0, V at +32 tokens, the
  // next (batch, head) 64 tokens on)
  QuantArgs a;
  a.k = res_layer;
  a.v = res_layer + static_cast<size_t>(kTile) * kD * 2;
  a.signs = signs_dev;
  a.bits = bits_dev;
  a.offsets = offsets_dev;
  a.packed = static_cast<uint8_t*>(packed);
  a.status = status_dev;
  a.layer = layer;
  a.B = desc->B;
  a.H = desc->H_kv;
  a.S = 2 * kTile;
  a.nblk = 1;
  a.kg = desc->k_grouping;
  a.vg = desc->v_grouping;
  a.kq = desc->k_quantizer;
  a.vq = desc->v_quantizer;
  a.hadamard = desc->hadamard ? 1 : 0;
  a.j_dst0 = pos / kTile;
  a.ntiles = static_cast<long long>(desc->B) * desc->H_kv * 2;
  const size_t smem = quant_smem_bytes(a.hadamard != 0);
  if (desc->dtype == RQ_F16)
    return a.hadamard ? launch_persistent(quantize_pack_kernel<__half, true>, a, smem, st)
                      : launch_persistent(quantize_pack_kernel<__half, false>, a, smem, st);
  return a.hadamard ? launch_persistent(quantize_pack_kernel<__nv_bfloat16, true>, a, smem, st)
                    : launch_persistent(quantize_pack_kernel<__nv_bfloat16, false>, a, smem, st);
}
