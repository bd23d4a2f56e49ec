// Quantize + bit-pack one layer of the KV cache at per-head bit-widths, and
// the distortion sweep that calibrates D(b) per component.
//
// RateQuant (arXiv 2605.06675): the quantizer kernel reads the per-head
// bit-width from the static allocation table (App. M "No runtime overhead",
// App. U "Runtime Analysis"); keys are quantized per channel and values per
// token (KIVI, Sec. 2 and App. W), optionally after a per-token Hadamard
// rotation (QuaRot, App. W "QuaRot kernel").
//
// One CTA of 128 threads owns one 32-token x 128-channel tile at a time
// (one packed block); its 128 groups map one-to-one onto threads. The next
// tile's 8 KB is loaded into registers while the current one is processed.
#include <algorithm>

#include "rq_internal.cuh"

namespace rq {
namespace {

constexpr int kThreads = 128;
constexpr int kXStride = kD + 1;        // fp32 tile row stride (bank spread)
constexpr int kCStride = kD + 4;        // code tile row stride in bytes

struct QuantArgs {
  const void* k;
  const void* v;
  const int8_t* signs;
  const uint8_t* bits;       // [L][H][2]
  const uint64_t* offsets;   // [L][B][H][2]
  uint8_t* packed;
  uint32_t* status;
  int layer, B, H, S, nblk, kg, vg, hadamard;
  long long ntiles;
};

struct QuantSmem {
  float x[kTile][kXStride];
  uint8_t c[kTile][kCStride];
  uint32_t out[128 * 9];    // codes image (128*b words) + meta image (128 words)
};

// (t, c) of slot e of fragment phi of lane L (the packed block format)
__device__ __forceinline__ void frag_elem(int kind, int L, int phi, int e, int& t, int& c) {
  const int gid = L >> 2, tig = L & 3;
  if (kind == 0) {                 // K: rows = tokens, k = channels
    const int ks = phi >> 1, mt = phi & 1;
    t = 16 * mt + gid + 8 * ((e >> 1) & 1);
    c = 16 * ks + 2 * tig + (e & 1) + 8 * (e >> 2);
  } else {                         // V: rows = channels, k = tokens
    const int ks = phi >> 3, mt = phi & 7;
    c = 16 * mt + gid + 8 * ((e >> 1) & 1);
    t = 16 * ks + 2 * tig + (e & 1) + 8 * (e >> 2);
  }
}

__device__ __forceinline__ void put_meta_half(uint32_t* meta, int word, int half, __half v) {
  reinterpret_cast<__half*>(meta)[2 * word + half] = v;
}

template <typename T>
__device__ __forceinline__ void tile_to_smem(QuantSmem& sm, const uint4 (&ld)[4],
                                             const int8_t* signs, bool hadamard) {
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int chunk = threadIdx.x + kThreads * i;  // 16 chunks of 8 elements per row
    const int row = chunk >> 4, col = (chunk & 15) * 8;
    float f[8];
    unpack8<T>(ld[i], f);
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      float x = f[e];
      if (hadamard && signs && signs[col + e] < 0) x = -x;
      sm.x[row][col + e] = x;
    }
  }
}

// In-place FWHT of every row: strides 1, 2, ..., 64 in that order, pair
// (i, i+h) with bit h of i clear -> (a + b, a - b); then * fp32(1/sqrt(128)).
__device__ void fwht_rows(QuantSmem& sm) {
  for (int lh = 0; lh < 7; ++lh) {
    const int h = 1 << lh;
#pragma unroll 4
    for (int p = threadIdx.x; p < kTile * (kD / 2); p += kThreads) {
      const int row = p >> 6, pi = p & 63;
      const int i = ((pi >> lh) << (lh + 1)) | (pi & (h - 1));
      const float a = sm.x[row][i], b = sm.x[row][i + h];
      sm.x[row][i] = __fadd_rn(a, b);
      sm.x[row][i + h] = __fsub_rn(a, b);
    }
    __syncthreads();
  }
  for (int p = threadIdx.x; p < kTile * kD; p += kThreads) {
    const int row = p >> 7, col = p & 127;
    sm.x[row][col] = __fmul_rn(sm.x[row][col], kInvSqrt128);
  }
  __syncthreads();
}

// Group of thread tau: per-channel -> channel tau, tokens 0..31;
// per-token -> token tau % 32, channels 32*(tau/32) .. +31.
__device__ __forceinline__ float group_elem(const QuantSmem& sm, int grouping, int i) {
  const int tau = threadIdx.x;
  return grouping == RQ_PER_CHANNEL ? sm.x[i][tau] : sm.x[tau & 31][32 * (tau >> 5) + i];
}

__device__ void quantize_groups(QuantSmem& sm, int kind, int grouping, int b, uint32_t* status) {
  const int tau = threadIdx.x;
  float mn = INFINITY, mx = -INFINITY;
  bool finite = true;
#pragma unroll 8
  for (int i = 0; i < kG; ++i) {
    const float v = __fadd_rn(group_elem(sm, grouping, i), 0.0f);  // -0 -> +0
    finite = finite && isfinite(v);
    mn = fminf(mn, v);
    mx = fmaxf(mx, v);
  }
  const GroupParams g = group_params(mn, mx, finite, b);
  if (g.bad) set_status(status, RQ_STATUS_NUMERIC);
  if (grouping == RQ_PER_CHANNEL) {
#pragma unroll 8
    for (int i = 0; i < kG; ++i) {
      const float v = __fadd_rn(sm.x[i][tau], 0.0f);
      sm.c[i][tau] = static_cast<uint8_t>(quant_code(v, g, b));
    }
  } else {
    const int t = tau & 31, c0 = 32 * (tau >> 5);
#pragma unroll
    for (int i = 0; i < kG; i += 4) {
      uint32_t packed4 = 0;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const float v = __fadd_rn(sm.x[t][c0 + i + j], 0.0f);
        packed4 |= static_cast<uint32_t>(quant_code(v, g, b)) << (8 * j);
      }
      *reinterpret_cast<uint32_t*>(&sm.c[t][c0 + i]) = packed4;
    }
  }
  // meta image
  uint32_t* meta = sm.out + 128 * b;
  if (kind == 0 && grouping == RQ_PER_CHANNEL) {
    const int c = tau;
    const int word = 16 * ((c & 7) >> 1) + 2 * (c >> 4) + ((c >> 3) & 1);
    put_meta_half(meta, word, c & 1, g.scale);
    put_meta_half(meta, 64 + word, c & 1, g.zero);
  } else if (kind == 1 && grouping == RQ_PER_TOKEN) {
    const int t = tau & 31, G = tau >> 5, p = t >> 1;
    const int word = 16 * (p & 3) + 4 * (p >> 2) + G;
    put_meta_half(meta, word, t & 1, g.scale);
    put_meta_half(meta, 64 + word, t & 1, g.zero);
  } else if (kind == 0) {          // K per-token: (scale, zero) word
    const int t = tau & 31, G = tau >> 5;
    const int word = 16 * (t & 7) + 4 * (t >> 3) + G;
    put_meta_half(meta, word, 0, g.scale);
    put_meta_half(meta, word, 1, g.zero);
  } else {                         // V per-channel: (scale, zero) word
    const int c = tau;
    const int word = 16 * (c & 7) + 2 * (c >> 4) + ((c >> 3) & 1);
    put_meta_half(meta, word, 0, g.scale);
    put_meta_half(meta, word, 1, g.zero);
  }
}

// Thread (lane L = tau % 32, quarter q = tau / 32) emits lane-stream words
// [b q, b q + b) from fragments 4q .. 4q+3, codes in slot-position order
// (a0 a2 a4 a6 a1 a3 a5 a7), b bits each, LSB first.
__device__ void pack_codes(QuantSmem& sm, int kind, int b) {
  const int L = threadIdx.x & 31, q = threadIdx.x >> 5;
  uint64_t acc = 0;
  int nacc = 0, w = b * q;
  for (int f = 0; f < 4; ++f) {
    const int phi = 4 * q + f;
#pragma unroll
    for (int pos = 0; pos < 8; ++pos) {
      const int e = pos < 4 ? 2 * pos : 2 * (pos - 4) + 1;
      int t, c;
      frag_elem(kind, L, phi, e, t, c);
      acc |= static_cast<uint64_t>(sm.c[t][c]) << nacc;
      nacc += b;
      if (nacc >= 32) {
        sm.out[128 * (w >> 2) + 4 * L + (w & 3)] = static_cast<uint32_t>(acc);
        acc >>= 32;
        nacc -= 32;
        ++w;
      }
    }
  }
}

template <typename T>
__global__ void __launch_bounds__(kThreads) quantize_pack_kernel(QuantArgs a) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  QuantSmem& sm = *reinterpret_cast<QuantSmem*>(smem_raw);
  const long long tile_stride = gridDim.x;
  long long tile = blockIdx.x;
  if (tile >= a.ntiles) return;

  auto tile_src = [&](long long tl) -> const uint4* {
    const int j = static_cast<int>(tl % a.nblk);
    const long long sk = tl / a.nblk;          // (b*H + h) * 2 + kind
    const int kind = static_cast<int>(sk & 1);
    const long long bh = sk >> 1;
    const T* base = static_cast<const T*>(kind ? a.v : a.k);
    return reinterpret_cast<const uint4*>(base + (bh * a.S + static_cast<long long>(kTile) * j) * kD);
  };

  uint4 ld[4];
  {
    const uint4* src = tile_src(tile);
#pragma unroll
    for (int i = 0; i < 4; ++i) ld[i] = ldg_stream(src + threadIdx.x + kThreads * i);
  }
  for (; tile < a.ntiles; tile += tile_stride) {
    const int j = static_cast<int>(tile % a.nblk);
    const long long sk = tile / a.nblk;
    const int kind = static_cast<int>(sk & 1);
    const long long bh = sk >> 1;
    const int h = static_cast<int>(bh % a.H);
    const int batch = static_cast<int>(bh / a.H);
    const int b = a.bits[(a.layer * a.H + h) * 2 + kind];

    tile_to_smem<T>(sm, ld, a.signs, a.hadamard != 0);
    __syncthreads();
    // prefetch the next tile while this one is processed
    const long long next = tile + tile_stride;
    if (next < a.ntiles) {
      const uint4* src = tile_src(next);
#pragma unroll
      for (int i = 0; i < 4; ++i) ld[i] = ldg_stream(src + threadIdx.x + kThreads * i);
    }
    if (b < 1 || b > 8) {
      if (threadIdx.x == 0) set_status(a.status, RQ_STATUS_BAD_BITS);
      __syncthreads();
      continue;
    }
    if (a.hadamard) fwht_rows(sm);
    const int grouping = kind ? a.vg : a.kg;
    quantize_groups(sm, kind, grouping, b, a.status);
    __syncthreads();
    pack_codes(sm, kind, b);
    __syncthreads();
    const uint64_t off = a.offsets[((static_cast<long long>(a.layer) * a.B + batch) * a.H + h) * 2 + kind];
    uint4* dst = reinterpret_cast<uint4*>(a.packed + off + static_cast<uint64_t>(j) * 512u * (b + 1));
    const uint4* srcs = reinterpret_cast<const uint4*>(sm.out);
    for (int i = threadIdx.x; i < 32 * (b + 1); i += kThreads) dst[i] = srcs[i];
    __syncthreads();
  }
}

template <typename T>
rq_status launch_quantize(const QuantArgs& a, cudaStream_t stream) {
  const size_t smem = sizeof(QuantSmem);
  auto kern = quantize_pack_kernel<T>;
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

// ------------------------------------------------------ distortion sweep ----
// Alg. 1 stage 2 / Sec. 3.4 "Distortion calibration": per component and
// b = 1..8, sum over the component's groups of (y - y_hat)^2 in fp64, where
// y_hat = fp32(fp32(c) * scale) + zero. One tile = 32 tokens of one component;
// per-tile partial sums are reduced in a fixed order (deterministic).

struct CalibArgs {
  const void* x;            // [n][T][128]
  const int8_t* signs;
  double* partial;          // [n][T/32][8]
  uint32_t* status;
  int n, T, ntile, kg, vg, hadamard;
  long long ntiles;
};

template <typename T>
__global__ void __launch_bounds__(kThreads) calib_sweep_kernel(CalibArgs a) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  QuantSmem& sm = *reinterpret_cast<QuantSmem*>(smem_raw);
  __shared__ double red[kThreads / 32][8];
  const long long tile_stride = gridDim.x;
  long long tile = blockIdx.x;
  if (tile >= a.ntiles) return;
  auto tile_src = [&](long long tl) -> const uint4* {
    const T* base = static_cast<const T*>(a.x);
    return reinterpret_cast<const uint4*>(base + tl * static_cast<long long>(kTile) * kD);
  };
  uint4 ld[4];
  {
    const uint4* src = tile_src(tile);
#pragma unroll
    for (int i = 0; i < 4; ++i) ld[i] = ldg_stream(src + threadIdx.x + kThreads * i);
  }
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (; tile < a.ntiles; tile += tile_stride) {
    const int comp = static_cast<int>(tile / a.ntile);
    const int grouping = (comp & 1) ? a.vg : a.kg;
    tile_to_smem<T>(sm, ld, a.signs, a.hadamard != 0);
    __syncthreads();
    const long long next = tile + tile_stride;
    if (next < a.ntiles) {
      const uint4* src = tile_src(next);
#pragma unroll
      for (int i = 0; i < 4; ++i) ld[i] = ldg_stream(src + threadIdx.x + kThreads * i);
    }
    if (a.hadamard) fwht_rows(sm);
    float v[kG];
    float mn = INFINITY, mx = -INFINITY;
    bool finite = true;
#pragma unroll
    for (int i = 0; i < kG; ++i) {
      v[i] = __fadd_rn(group_elem(sm, grouping, i), 0.0f);
      finite = finite && isfinite(v[i]);
      mn = fminf(mn, v[i]);
      mx = fmaxf(mx, v[i]);
    }
    double acc[8];
#pragma unroll
    for (int b = 1; b <= 8; ++b) {
      const GroupParams g = group_params(mn, mx, finite, b);
      if (b == 1 && g.bad) set_status(a.status, RQ_STATUS_NUMERIC);
      double s = 0.0;
#pragma unroll
      for (int i = 0; i < kG; ++i) {
        const int c = quant_code(v[i], g, b);
        const float xh = __fadd_rn(__fmul_rn(static_cast<float>(c), g.sf), g.zf);
        const double e = static_cast<double>(v[i]) - static_cast<double>(xh);
        s = __dadd_rn(s, __dmul_rn(e, e));
      }
      acc[b - 1] = s;
    }
    // fixed-order block reduction: warp butterfly, then warps 0..3 in order
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      double t = acc[k];
#pragma unroll
      for (int o = 16; o >= 1; o >>= 1) t = __dadd_rn(t, __shfl_xor_sync(0xffffffffu, t, o));
      if (lane == 0) red[warp][k] = t;
    }
    __syncthreads();
    if (threadIdx.x < 8) {
      double t = red[0][threadIdx.x];
#pragma unroll
      for (int w = 1; w < kThreads / 32; ++w) t = __dadd_rn(t, red[w][threadIdx.x]);
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

template <typename T>
rq_status launch_calib(const CalibArgs& a, double* mse, cudaStream_t stream) {
  const size_t smem = sizeof(QuantSmem);
  auto kern = calib_sweep_kernel<T>;
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
  if (launch_status() != RQ_OK) return RQ_ERR_CUDA;
  const int total = a.n * 8;
  calib_finalize_kernel<<<(total + 127) / 128, 128, 0, stream>>>(
      a.partial, mse, a.n, a.ntile, static_cast<double>(a.T) * kD);
  return launch_status();
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
  a.hadamard = desc->hadamard ? 1 : 0;
  a.ntiles = static_cast<long long>(desc->B) * desc->H_kv * 2 * a.nblk;
  if (a.ntiles == 0) return RQ_OK;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  return desc->dtype == RQ_F16 ? launch_quantize<__half>(a, st)
                               : launch_quantize<__nv_bfloat16>(a, st);
}

extern "C" size_t rq_calibrate_workspace_bytes(int32_t n, int32_t T) {
  if (n <= 0 || T <= 0) return 0;
  return static_cast<size_t>(n) * static_cast<size_t>((T + rq::kTile - 1) / rq::kTile) * 8 *
         sizeof(double);
}

extern "C" rq_status rq_calibrate_distortion(const void* x, int32_t dtype, int32_t n, int32_t T,
                                             int32_t k_grouping, int32_t v_grouping,
                                             int32_t hadamard, const int8_t* signs_dev,
                                             double* mse_dev, void* ws, size_t ws_bytes,
                                             uint32_t* status_dev, void* stream) {
  using namespace rq;
  if (!x || !mse_dev || !ws || n <= 0 || T <= 0) return RQ_ERR_INVALID_ARG;
  if (dtype != RQ_F16 && dtype != RQ_BF16) return RQ_ERR_INVALID_ARG;
  for (int g : {k_grouping, v_grouping})
    if (g != RQ_PER_TOKEN && g != RQ_PER_CHANNEL) return RQ_ERR_INVALID_ARG;
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
  a.hadamard = hadamard ? 1 : 0;
  a.ntiles = static_cast<long long>(n) * a.ntile;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  return dtype == RQ_F16 ? launch_calib<__half>(a, mse_dev, st)
                         : launch_calib<__nv_bfloat16>(a, mse_dev, st);
}
