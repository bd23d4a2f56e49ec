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

// Quantizer parameters of one group (every step rounded as stated):
//   s32 = fp32(mx - mn) / L, scale = fp16(s32), zero = fp16(mn),
//   inv = 1 / fp32(scale); a group is "bad" when it held a non-finite value
//   or scale/zero overflowed fp16 (then codes, scale and zero are all 0).
struct GroupParams {
  __half scale, zero;
  float sf, zf, inv;
  bool ok;   // codes are computed (not bad and scale != 0)
  bool bad;
};

__device__ __forceinline__ GroupParams group_params(float mn, float mx, bool finite, int b) {
  GroupParams g;
  const float L = static_cast<float>((1 << b) - 1);
  const float s32 = __fdiv_rn(__fsub_rn(mx, mn), L);
  g.scale = __float2half_rn(s32);
  g.zero = __float2half_rn(mn);
  g.sf = __half2float(g.scale);
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
// bits of the result; out-of-range values are clamped to [magic, magic + L]
// (NaN from a bad group clamps to magic: code 0).
constexpr float kRoundMagic = 12582912.0f;

__device__ __forceinline__ float round_magic_clamped(float t, float inv, float L) {
  const float u = __fmaf_rn(t, inv, kRoundMagic);
  return fminf(fmaxf(u, kRoundMagic), kRoundMagic + L);
}

}  // namespace rq
