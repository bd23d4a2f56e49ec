// Internal helpers shared by librq's CUDA translation units (sm_103a only).
#pragma once

#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <cstdint>

#include "rq.h"

namespace rq {

constexpr int kD = 128;             // head dim
constexpr int kG = 32;              // group size
constexpr int kTile = 32;           // tokens per packed block
constexpr float kInvSqrt128 = 0.08838834764831845f;  // fp32 RN of 2^-3.5
constexpr float kLog2e = 1.4426950408889634f;

// ------------------------------------------------------------ host side ----

inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// SM count of the current device (cached per device ordinal).
rq_status current_sm_count(int* sms);

inline rq_status launch_status() {
  return cudaGetLastError() == cudaSuccess ? RQ_OK : RQ_ERR_CUDA;
}

// The Lloyd-Max codebooks (RQ_LLOYDMAX) of every width, passed to the kernels
// by value: fp16 bit patterns, ascending, width b at lv[2^b - 2 ..].
struct LMBook {
  uint16_t lv[510];
};
__host__ __device__ constexpr int lm_offset(int b) { return (1 << b) - 2; }
// the library's codebook (host.cpp), and one filled LMBook
const uint16_t* lloydmax_levels(int b);
// rq_grouping values; the wide per-token groupings (64 or 128 channels of
// one token) are stored as per-token groups of 32 that repeat their wide
// group's scale and zero
inline bool grouping_ok(int g) {
  return g == RQ_PER_TOKEN || g == RQ_PER_CHANNEL || g == RQ_PER_TOKEN_64 || g == RQ_PER_TOKEN_128;
}
// the grouping of the packed format (RQ_PER_TOKEN or RQ_PER_CHANNEL)
__host__ __device__ constexpr int stored_grouping(int g) {
  return g == RQ_PER_CHANNEL ? RQ_PER_CHANNEL : RQ_PER_TOKEN;
}
// groups of 32 channels in one group of a per-token grouping (1, 2 or 4)
__host__ __device__ constexpr int token_span(int g) {
  return g == RQ_PER_TOKEN_128 ? 4 : g == RQ_PER_TOKEN_64 ? 2 : 1;
}
// a quantizer choice of keys and values is supported: min-max and absmax with
// any grouping, Lloyd-Max with per-token groups of 32
inline bool quantizers_ok(int kq, int kg, int vq, int vg) {
  for (int i = 0; i < 2; ++i) {
    const int q = i ? vq : kq, g = i ? vg : kg;
    if (!grouping_ok(g)) return false;
    if (q != RQ_MINMAX && q != RQ_ABSMAX && q != RQ_LLOYDMAX) return false;
    if (q == RQ_LLOYDMAX && g != RQ_PER_TOKEN) return false;
  }
  return true;
}
inline void fill_lm_book(LMBook& book) {
  for (int b = 1; b <= 8; ++b) {
    const uint16_t* lv = lloydmax_levels(b);
    for (int i = 0; i < (1 << b); ++i) book.lv[lm_offset(b) + i] = lv[i];
  }
}

// ---------------------------------------------------------- device side ----

template <typename T>
__device__ __forceinline__ float to_f32(T x);
template <>
__device__ __forceinline__ float to_f32<__half>(__half x) { return __half2float(x); }
template <>
__device__ __forceinline__ float to_f32<__nv_bfloat16>(__nv_bfloat16 x) {
  return __bfloat162float(x);
}

// the 8 elements of one 16-byte chunk as fp32 (exact for fp16 and bf16)
template <typename T>
__device__ __forceinline__ void unpack8(const uint4& u, float (&f)[8]) {
  const T* e = reinterpret_cast<const T*>(&u);
#pragma unroll
  for (int i = 0; i < 8; ++i) f[i] = to_f32<T>(e[i]);
}

__device__ __forceinline__ uint4 ldg_stream(const void* p) {
  uint4 r;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];\n"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p));
  return r;
}

__device__ __forceinline__ void set_status(uint32_t* status, uint32_t bits) {
  if (status) atomicOr(status, bits);
}

// Quantizer parameters of one group (every step rounded as stated).
//   min-max:  s32 = fp32(mx - mn) / L, scale = fp16(s32), zero = fp16(mn),
//             codes 0 .. L = 2^b - 1;
//   absmax (sym): a = max(|mn|, |mx|), M = 2^(b-1) - 1, s32 = a / M (0 when
//             M = 0), scale = fp16(s32), zero = fp16(0 - M * fp32(scale))
//             (the product is exact), codes 0 .. 2M;
//   inv = 1 / fp32(scale); a group is "bad" when it held a non-finite value
//   or scale/zero overflowed fp16 (then codes, scale and zero are all 0).
struct GroupParams {
  __half scale, zero;
  float sf, zf, inv;
  float cmax;  // largest code
  bool ok;     // codes are computed (not bad and scale != 0)
  bool bad;
};

// RN(1 / (2^k - 1)), k = 0..8 (index 0 unused): the divisors of the scale
static __constant__ float kInvPow2m1[9] = {1.0f,         1.0f / 1.0f,   1.0f / 3.0f,
                                           1.0f / 7.0f,  1.0f / 15.0f,  1.0f / 31.0f,
                                           1.0f / 63.0f, 1.0f / 127.0f, 1.0f / 255.0f};

// RN(x / y) for y = 2^k - 1 (k = 1..8) and yi = RN(1 / y): Markstein's
// correction step, q0 = RN(x yi), r = x - q0 y (exact in one FMA),
// q = RN(q0 + r yi). Checked equal to IEEE division for every fp32
// significand of x and each of these divisors (tests/test_lib_host.py);
// exact scaling by powers of two carries it to every exponent of a normal
// quotient, and quotients below the fp32 normal range round to fp16 zero
// either way.
__device__ __forceinline__ float div_pow2m1(float x, float y, float yi) {
  const float q0 = __fmul_rn(x, yi);
  const float r = __fmaf_rn(-q0, y, x);
  return __fmaf_rn(r, yi, q0);
}

__device__ __forceinline__ GroupParams group_params(float mn, float mx, bool finite, int b,
                                                    bool sym) {
  GroupParams g;
  // one division for both forms: (mx - mn) / L, or a / M (0 when M = 0)
  const float M = static_cast<float>((1 << (b - 1)) - 1);
  const float L = static_cast<float>((1 << b) - 1);
  const float a = fmaxf(fabsf(mn), fabsf(mx));
  const float num = sym ? (M > 0.0f ? a : 0.0f) : __fsub_rn(mx, mn);
  const float den = sym ? fmaxf(M, 1.0f) : L;
  const float deni = kInvPow2m1[sym ? (b > 1 ? b - 1 : 1) : b];
  g.scale = __float2half_rn(div_pow2m1(num, den, deni));
  g.sf = __half2float(g.scale);
  g.zero = __float2half_rn(sym ? __fsub_rn(0.0f, __fmul_rn(M, g.sf)) : mn);
  g.cmax = sym ? 2.0f * M : L;
  g.zf = __half2float(g.zero);
  g.bad = !finite || !isfinite(g.sf) || !isfinite(g.zf);
  g.ok = !g.bad && g.sf != 0.0f;
  g.inv = g.ok ? __fdiv_rn(1.0f, g.sf) : 0.0f;
  if (g.bad) {
    g.scale = __float2half_rn(0.0f);
    g.zero = __float2half_rn(0.0f);
    g.sf = 0.0f;
    g.zf = 0.0f;
  }
  return g;
}

// 1.5 * 2^23: RN(t * inv + kRoundMagic) = kRoundMagic + rint_half_even(t * inv)
// (exact product, one rounding) for |t * inv| < 2^22, so the code is the low
// bits of the result; out-of-range values are clamped to [magic, magic + cmax]
// (NaN from a bad group clamps to magic: code 0).
constexpr float kRoundMagic = 12582912.0f;

__device__ __forceinline__ float round_magic_clamped(float t, float inv, float cmax) {
  const float u = __fmaf_rn(t, inv, kRoundMagic);
  return fminf(fmaxf(u, kRoundMagic), kRoundMagic + cmax);
}

}  // namespace rq
