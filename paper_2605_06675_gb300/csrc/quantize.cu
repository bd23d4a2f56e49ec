// Quantize + bit-pack one layer of the KV cache at per-head bit-widths (host
// entry points; the kernels are in quantize_kernel.cuh), the distortion sweep
// that calibrates D(b) per component, and decode-time append.
//
// RateQuant (arXiv 2605.06675): the quantizer kernel reads the per-head
// bit-width from the static allocation table (App. M "No runtime overhead",
// App. U "Runtime Analysis"); the sweep measures the MSE at every b for the
// fit of D(b) = alpha beta^-b (Alg. 1 stage 2, Sec. 3.4).
#include "quantize_kernel.cuh"

namespace rq {
namespace {

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
  float lm_lev[512];                    // Lloyd-Max levels of every width (at lm_offset(b))
  float lm_mid[512];                    // and the midpoints between them
};

// Lloyd-Max code at a width known only at run time (the sweep's loop)
__device__ __forceinline__ int lm_code_rt(float v, float sf, const float* mid, int b) {
  int c = 0;
  for (int k = b - 1; k >= 0; --k) {
    const int cand = c + (1 << k);
    c = v >= __fmul_rn(mid[cand - 1], sf) ? cand : c;
  }
  return sf != 0.0f ? c : 0;
}
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
  if (a.kq == RQ_LLOYDMAX || a.vq == RQ_LLOYDMAX) {
    for (int i = threadIdx.x; i < 510; i += kThreads) {
      sm.lm_lev[i] = __half2float(__ushort_as_half(a.lm.lv[i]));
    }
    __syncthreads();
    for (int b = 1; b <= 8; ++b)
      for (int i = threadIdx.x; i < (1 << b) - 1; i += kThreads)
        sm.lm_mid[lm_offset(b) + i] =
            __fmul_rn(__fadd_rn(sm.lm_lev[lm_offset(b) + i], sm.lm_lev[lm_offset(b) + i + 1]), 0.5f);
  }
  __syncthreads();
  const bool had = a.hadamard != 0;
  const T* xbase = static_cast<const T*>(a.x);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;

  int grouping = (static_cast<int>(tile / a.ntile) & 1) ? a.vg : a.kg;
  int form = (static_cast<int>(tile / a.ntile) & 1) ? a.vq : a.kq;
  bool row_mode = grouping == RQ_PER_TOKEN || had;
  uint4 ld[4];
  calib_load<T>(xbase + tile * kTile * kD, row_mode, ld);
  for (; tile < a.ntiles; tile += stride) {
    float v[kG];
    calib_group_values<T>(ld, row_mode, grouping, had, sm, x32, v);
    const long long next = tile + stride;
    const int form_now = form, grouping_now = grouping;
    const int span_now = (static_cast<int>(tile / a.ntile) & 1) ? a.vspan : a.kspan;
    if (next < a.ntiles) {
      form = (static_cast<int>(next / a.ntile) & 1) ? a.vq : a.kq;
      grouping = (static_cast<int>(next / a.ntile) & 1) ? a.vg : a.kg;
      row_mode = grouping == RQ_PER_TOKEN || had;
      calib_load<T>(xbase + next * kTile * kD, row_mode, ld);
    }
    float mn, mx;
    minmax32(v, mn, mx);
    if (grouping_now == RQ_PER_TOKEN) join_quarters(mn, mx, span_now);   // wide per-token groups
    const bool finite = isfinite(mn) && isfinite(mx);
    mn = __fadd_rn(mn, 0.0f);
    mx = __fadd_rn(mx, 0.0f);
    double acc[8];
    if (form_now == RQ_LLOYDMAX) {
      // the group's RMS scale (as the quantizer computes it), then every width
      const float s2s = __fadd_rn(sumsq16(v), sumsq16(v + 16));
      float sf = __half2float(__float2half_rn(__fsqrt_rn(__fmul_rn(s2s, 0.03125f))));
      if (!finite || !isfinite(sf)) {
        set_status(a.status, RQ_STATUS_NUMERIC);
        sf = 0.0f;
      }
      float vz[kG];
#pragma unroll
      for (int i = 0; i < kG; ++i) vz[i] = __fadd_rn(v[i], 0.0f);
#pragma unroll 1
      for (int b = 1; b <= 8; ++b) {
        const float* mid = sm.lm_mid + lm_offset(b);
        const float* lev = sm.lm_lev + lm_offset(b);
        float2 s2 = make_float2(0.0f, 0.0f);
#pragma unroll
        for (int i = 0; i < kG; i += 2) {
          const float x0 = __fmul_rn(lev[lm_code_rt(vz[i], sf, mid, b)], sf);
          const float x1 = __fmul_rn(lev[lm_code_rt(vz[i + 1], sf, mid, b)], sf);
          const float2 e = __fadd2_rn(make_float2(v[i], v[i + 1]), make_float2(-x0, -x1));
          s2 = __ffma2_rn(e, e, s2);
        }
        acc[b - 1] = static_cast<double>(s2.x) + static_cast<double>(s2.y);
      }
    } else {
#pragma unroll
    for (int b = 1; b <= 8; ++b) {
      const GroupParams g = group_params(mn, mx, finite, b, form_now == RQ_ABSMAX);
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

size_t calib_smem_bytes(bool hadamard, int kg, int vg) {
  const bool x32 = hadamard && (kg == RQ_PER_CHANNEL || vg == RQ_PER_CHANNEL);
  return sizeof(CalibSmem) + (x32 ? kTile * (kD + 1) * sizeof(float) : 0);
}

}  // namespace
}  // namespace rq

namespace rq {
namespace {
// K/V may be device memory or page-locked host memory (which the kernel then
// reads over the host link); plain pageable host memory is refused before any
// launch. cudaPointerGetAttributes reports memory it does not know as
// unregistered.
bool device_readable(const void* p) {
  cudaPointerAttributes at{};
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    cudaGetLastError();          // reset the error state the failed query left
    return false;
  }
  return at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged ||
         at.type == cudaMemoryTypeHost;
}
}  // namespace
}  // namespace rq

namespace rq {
namespace {
// the quantize instance for the dtype and rotation; the Lloyd-Max kernel when
// both kinds are Lloyd-Max
rq_status launch_quantize(const QuantArgs& a, int32_t dtype, cudaStream_t st) {
  const bool lm = a.kq == RQ_LLOYDMAX && a.vq == RQ_LLOYDMAX;
  if (dtype == RQ_F16) {
    if (lm) return a.hadamard ? launch_quantize_lm_f16_rot(a, st) : launch_quantize_lm_f16(a, st);
    return a.hadamard ? launch_quantize_f16_rot(a, st) : launch_quantize_f16(a, st);
  }
  if (lm) return a.hadamard ? launch_quantize_lm_bf16_rot(a, st) : launch_quantize_lm_bf16(a, st);
  return a.hadamard ? launch_quantize_bf16_rot(a, st) : launch_quantize_bf16(a, st);
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
    if (!grouping_ok(g)) return RQ_ERR_INVALID_ARG;
  if (!quantizers_ok(desc->k_quantizer, desc->k_grouping, desc->v_quantizer, desc->v_grouping))
    return RQ_ERR_INVALID_ARG;
  if (desc->d != kD || desc->group != kG || desc->S % kTile != 0) return RQ_ERR_SHAPE;
  if (!aligned16(k) || !aligned16(v) || !aligned16(packed)) return RQ_ERR_ALIGNMENT;
  if (!device_readable(k) || !device_readable(v)) return RQ_ERR_INVALID_ARG;
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
  a.kg = stored_grouping(desc->k_grouping);
  a.vg = stored_grouping(desc->v_grouping);
  a.kspan = token_span(desc->k_grouping);
  a.vspan = token_span(desc->v_grouping);
  a.kq = desc->k_quantizer;
  a.vq = desc->v_quantizer;
  if (a.kq == RQ_LLOYDMAX || a.vq == RQ_LLOYDMAX) fill_lm_book(a.lm);
  a.hadamard = desc->hadamard ? 1 : 0;
  a.j_dst0 = 0;
  a.row_pos = nullptr;
  a.cap = desc->S;
  a.ntiles = static_cast<long long>(desc->B) * desc->H_kv * 2 * a.nblk;
  if (a.ntiles == 0) return RQ_OK;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  return launch_quantize(a, desc->dtype, st);
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
    if (!grouping_ok(g)) return RQ_ERR_INVALID_ARG;
  if (!quantizers_ok(k_quantizer, k_grouping, v_quantizer, v_grouping)) return RQ_ERR_INVALID_ARG;
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
  a.kg = stored_grouping(k_grouping);
  a.vg = stored_grouping(v_grouping);
  a.kspan = token_span(k_grouping);
  a.vspan = token_span(v_grouping);
  a.kq = k_quantizer;
  a.vq = v_quantizer;
  if (a.kq == RQ_LLOYDMAX || a.vq == RQ_LLOYDMAX) fill_lm_book(a.lm);
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

// As append_token_kernel with a position per batch row: a negative position
// appends nothing for that row, one at or past the capacity is reported.
__global__ void append_token_rows_kernel(const uint4* k_new, const uint4* v_new,
                                         uint4* residual_layer, const int32_t* pos, int H,
                                         int cap, uint32_t* status) {
  const int bh = blockIdx.x, t = threadIdx.x, kind = t >> 4, ch = t & 15;
  const int p = pos[bh / H];
  if (p < 0) return;
  if (p >= cap) {
    if (t == 0 && bh % H == 0) set_status(status, RQ_STATUS_BAD_POSITION);
    return;
  }
  const uint4* src = (kind ? v_new : k_new) + bh * 16 + ch;
  residual_layer[(bh * 2 + kind) * 32 * 16 + (p % kTile) * 16 + ch] = *src;
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
    if (!grouping_ok(g)) return RQ_ERR_INVALID_ARG;
  if (!quantizers_ok(desc->k_quantizer, desc->k_grouping, desc->v_quantizer, desc->v_grouping))
    return RQ_ERR_INVALID_ARG;
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
  a.kg = stored_grouping(desc->k_grouping);
  a.vg = stored_grouping(desc->v_grouping);
  a.kspan = token_span(desc->k_grouping);
  a.vspan = token_span(desc->v_grouping);
  a.kq = desc->k_quantizer;
  a.vq = desc->v_quantizer;
  if (a.kq == RQ_LLOYDMAX || a.vq == RQ_LLOYDMAX) fill_lm_book(a.lm);
  a.hadamard = desc->hadamard ? 1 : 0;
  a.j_dst0 = pos / kTile;
  a.row_pos = nullptr;
  a.cap = desc->S;
  a.ntiles = static_cast<long long>(desc->B) * desc->H_kv * 2;
  return launch_quantize(a, desc->dtype, st);
}

// ---- decode-time append with a position per batch row ----------------------
extern "C" rq_status rq_append_rows(const rq_cache_desc* desc, int32_t layer,
                                    const int32_t* pos_dev, const void* k_new, const void* v_new,
                                    void* residual, const int8_t* signs_dev,
                                    const uint8_t* bits_dev, const uint64_t* offsets_dev,
                                    void* packed, uint32_t* status_dev, void* stream) {
  using namespace rq;
  if (!desc || !pos_dev || !k_new || !v_new || !residual || !bits_dev || !offsets_dev || !packed)
    return RQ_ERR_INVALID_ARG;
  if (desc->L <= 0 || desc->B < 0 || desc->H_kv <= 0 || desc->S < 0) return RQ_ERR_INVALID_ARG;
  if (layer < 0 || layer >= desc->L) return RQ_ERR_INVALID_ARG;
  if (desc->dtype != RQ_F16 && desc->dtype != RQ_BF16) return RQ_ERR_INVALID_ARG;
  for (int g : {desc->k_grouping, desc->v_grouping})
    if (!grouping_ok(g)) return RQ_ERR_INVALID_ARG;
  if (!quantizers_ok(desc->k_quantizer, desc->k_grouping, desc->v_quantizer, desc->v_grouping))
    return RQ_ERR_INVALID_ARG;
  if (desc->d != kD || desc->group != kG || desc->S % kTile != 0) return RQ_ERR_SHAPE;
  if (!aligned16(k_new) || !aligned16(v_new) || !aligned16(residual) || !aligned16(packed) ||
      (reinterpret_cast<uintptr_t>(pos_dev) & 3u))
    return RQ_ERR_ALIGNMENT;
  if (desc->B == 0) return RQ_OK;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const size_t layer_bytes = residual_layer_elems(desc) * 2;
  uint8_t* res_layer = static_cast<uint8_t*>(residual) + static_cast<size_t>(layer) * layer_bytes;
  append_token_rows_kernel<<<static_cast<unsigned>(desc->B * desc->H_kv), 32, 0, st>>>(
      static_cast<const uint4*>(k_new), static_cast<const uint4*>(v_new),
      reinterpret_cast<uint4*>(res_layer), pos_dev, desc->H_kv, desc->S, status_dev);
  if (launch_status() != RQ_OK) return RQ_ERR_CUDA;
  // every row whose window is now full (its position is 31 mod 32) packs it
  // as block position / 32; the kernel reads the positions and skips the rest
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
  a.kg = stored_grouping(desc->k_grouping);
  a.vg = stored_grouping(desc->v_grouping);
  a.kspan = token_span(desc->k_grouping);
  a.vspan = token_span(desc->v_grouping);
  a.kq = desc->k_quantizer;
  a.vq = desc->v_quantizer;
  if (a.kq == RQ_LLOYDMAX || a.vq == RQ_LLOYDMAX) fill_lm_book(a.lm);
  a.hadamard = desc->hadamard ? 1 : 0;
  a.j_dst0 = 0;
  a.row_pos = pos_dev;
  a.cap = desc->S;
  a.ntiles = static_cast<long long>(desc->B) * desc->H_kv * 2;
  return launch_quantize(a, desc->dtype, st);
}
