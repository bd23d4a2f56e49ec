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
// One CTA of 128 threads owns one 32-token x 128-channel tile (one packed
// block) at a time; its 128 groups of 32 map one-to-one onto threads and a
// group's 32 values live in that thread's registers:
//   per-token group  (t, G): thread 4t + G loads its 64 bytes straight from
//                    global memory (the 4 groups of a token sit in 4
//                    neighbouring lanes, so the Hadamard butterflies across
//                    groups are two warp shuffles);
//   per-channel group c:    the tile is staged in shared memory as raw 16-bit
//                    values and thread c reads its column.
// The next tile's loads are in flight while the current one is processed.
#include <algorithm>

#include "rq_internal.cuh"

namespace rq {
namespace {

constexpr int kThreads = 128;
// CTAs per SM the quantizer's register budget is sized for
#ifndef RQ_QUANT_MIN_BLOCKS
#define RQ_QUANT_MIN_BLOCKS 8
#endif
constexpr int kX16Stride = kD + 8;      // u16 per staged row (272 B: spreads banks)
constexpr int kCStride = kD + 4;        // code tile [t][c], bytes per row
constexpr int kCTStride = kTile + 4;    // transposed code tile [c][t], bytes per row
constexpr int kCodeBytes = 4624;        // max(32 * 132, 128 * 36 + 4 * 4)
// row c of the transposed tile starts at ct_row(c): rows 32 apart are skewed
// by one bank so the four channel groups of a token store without conflicts
__host__ __device__ constexpr int ct_row(int c) { return c * kCTStride + 4 * (c >> 5); }
constexpr int kOutWords = 128 * 9;      // codes image (128 b words) + meta image (128 words)

struct TileSmem {
  uint16_t x16[kTile * kX16Stride];     // raw staged tile (column mode)
  uint8_t codes[kCodeBytes];            // code tile (K: [t][c], V: [c][t])
  uint32_t out[kOutWords];              // packed block image
  int8_t signs[kD];
};
// a rotated per-channel tile needs the rotated fp32 values in shared memory
constexpr int kX32Floats = kTile * (kD + 1);

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

struct CalibArgs {
  const void* x;             // [n][T][128]
  const int8_t* signs;
  double* partial;           // [n][T/32][8]
  uint32_t* status;
  int n, T, ntile, kg, vg, hadamard;
  long long ntiles;
};

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
// round to nearest even and saturate to [0, 255] in one conversion
__device__ __forceinline__ uint32_t cvt_rni_sat_u8(float x) {
  uint32_t r;
  asm("cvt.rni.sat.u8.f32 %0, %1;" : "=r"(r) : "f"(x));
  return r;
}

// ------------------------------------------------------------- loading ----

// Row mode (per-token groups, or any rotated tile): thread 4t + G holds the
// 64 bytes of token t, channels 32G..32G+31. Column mode: thread tau holds
// 16-byte chunks tau + 128 i of the tile (coalesced).
template <typename T>
__device__ __forceinline__ void load_tile(const T* tile_base, bool row_mode, uint4 (&ld)[4]) {
  const uint4* src = row_mode
      ? reinterpret_cast<const uint4*>(tile_base + (threadIdx.x >> 2) * kD + 32 * (threadIdx.x & 3))
      : reinterpret_cast<const uint4*>(tile_base) + threadIdx.x;
  const int stride = row_mode ? 1 : kThreads;
#pragma unroll
  for (int i = 0; i < 4; ++i) ld[i] = ldg_stream(src + i * stride);
}

// The 32 values of this thread's group, in the quantizer's domain, in
// registers (rotated when `hadamard`). Ends with every thread's group ready;
// contains __syncthreads (call uniformly).
template <typename T>
__device__ __forceinline__ void group_values(const uint4 (&ld)[4], bool row_mode, int grouping,
                                             bool hadamard, TileSmem& sm, float* x32,
                                             float (&v)[kG]) {
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
      const int G = tau & 3;
#pragma unroll
      for (int i = 0; i < kG; ++i)
        if (sm.signs[32 * G + i] < 0) v[i] = -v[i];
      // butterflies of stride 1..16 inside the group, in order
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
      // strides 32 and 64 pair this group with the lanes holding G^1, G^2;
      // the lower channel gets a + b, the upper a - b (a = lower's value)
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
      if (grouping == RQ_PER_CHANNEL) {       // regroup the rotated tile by column
        const int t = tau >> 2;
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

// min / max of the group; NaN propagates so a non-finite group is detected
__device__ __forceinline__ void group_minmax(const float (&v)[kG], float& mn, float& mx,
                                             bool& finite) {
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
  mn = __fadd_rn(lo[0], 0.0f);   // -0 -> +0
  mx = __fadd_rn(hi[0], 0.0f);
  finite = isfinite(mn) && isfinite(mx);
}

// codes c_i = clamp(rint((v_i - zero) * inv), 0, L); a group without codes
// (bad, or scale 0) has inv = 0 and yields 0 everywhere
__device__ __forceinline__ void group_codes(const float (&v)[kG], const GroupParams& g, int b,
                                            uint32_t (&c)[kG]) {
  const float2 nz = make_float2(-g.zf, -g.zf);
  const float2 iv = make_float2(g.inv, g.inv);
  const uint32_t L = (1u << b) - 1u;
#pragma unroll
  for (int i = 0; i < kG; i += 2) {
    const float2 t = __fmul2_rn(__fadd2_rn(make_float2(v[i], v[i + 1]), nz), iv);
    c[i] = min(cvt_rni_sat_u8(t.x), L);
    c[i + 1] = min(cvt_rni_sat_u8(t.y), L);
  }
}

// ------------------------------------------------------------- packing ----

// Fragment slot layout (the packed block format): fragment phi of lane L
// holds 8 codes in slots a0 a2 a4 a6 a1 a3 a5 a7, b bits each, LSB first.
// Pair k = (a_2k, a_2k+1) sits at adjacent bytes of the code tile (K: same
// token, channels c and c+1; V: same channel, tokens t and t+1, transposed tile).
template <int B>
__device__ __forceinline__ void put_bits(uint32_t (&w)[B], int pos, uint32_t x) {
  const int wi = pos >> 5, sh = pos & 31;
  w[wi] |= x << sh;
  if (sh + B > 32) w[wi + 1] |= x >> (32 - sh);
}

template <int B>
__device__ __forceinline__ void place_fragment(uint32_t (&w)[B], int f, const uint32_t (&p)[4]) {
  if constexpr (B == 2) {          // p << 2k puts lo at 2k and hi at 8 + 2k
    const uint32_t frag = p[0] | (p[1] << 2) | (p[2] << 4) | (p[3] << 6);
    w[f >> 1] |= frag << (16 * (f & 1));
  } else if constexpr (B == 4) {   // spread bytes to half-words, then << 4k
    uint32_t frag = 0;
#pragma unroll
    for (int k = 0; k < 4; ++k) frag |= __byte_perm(p[k], 0u, 0x4140) << (4 * k);
    w[f] = frag;
  } else if constexpr (B == 8) {   // lo bytes -> word 2f, hi bytes -> word 2f+1
    const uint32_t a = __byte_perm(p[0], p[1], 0x5140);
    const uint32_t b = __byte_perm(p[2], p[3], 0x5140);
    w[2 * f] = __byte_perm(a, b, 0x5410);
    w[2 * f + 1] = __byte_perm(a, b, 0x7632);
  } else {
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      put_bits<B>(w, 8 * B * f + B * k, p[k] & 0xFFu);
      put_bits<B>(w, 8 * B * f + 4 * B + B * k, p[k] >> 8);
    }
  }
}

// Thread (lane L = tau % 32, quarter q = tau / 32) writes lane-stream words
// [B q, B q + B) of lane L: fragments 4q .. 4q+3.
template <int KIND, int B>
__device__ __forceinline__ void pack_codes(const uint8_t* codes, uint32_t* out) {
  const int L = threadIdx.x & 31, q = threadIdx.x >> 5, gid = L >> 2, tig = L & 3;
  uint32_t w[B];
#pragma unroll
  for (int i = 0; i < B; ++i) w[i] = 0;
#pragma unroll
  for (int f = 0; f < 4; ++f) {
    uint32_t p[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      if (KIND == 0) {    // K: token 16 mt + gid + 8 (k&1), channel 16 ks + 2 tig + 8 (k>>1)
        const int t = 16 * (f & 1) + gid + 8 * (k & 1);
        const int c = 16 * (2 * q + (f >> 1)) + 2 * tig + 8 * (k >> 1);
        p[k] = *reinterpret_cast<const uint16_t*>(codes + t * kCStride + c);
      } else {            // V: channel 16 mt + gid + 8 (k&1), token 16 ks + 2 tig + 8 (k>>1)
        const int c = 16 * (4 * (q & 1) + f) + gid + 8 * (k & 1);
        const int t = 16 * (q >> 1) + 2 * tig + 8 * (k >> 1);
        p[k] = *reinterpret_cast<const uint16_t*>(codes + ct_row(c) + t);
      }
    }
    place_fragment<B>(w, f, p);
  }
#pragma unroll
  for (int i = 0; i < B; ++i) {
    const int ws = B * q + i;
    out[128 * (ws >> 2) + 4 * L + (ws & 3)] = w[i];
  }
}

template <int KIND>
__device__ __forceinline__ void pack_dispatch(int b, const uint8_t* codes, uint32_t* out) {
  switch (b) {
    case 1: pack_codes<KIND, 1>(codes, out); break;
    case 2: pack_codes<KIND, 2>(codes, out); break;
    case 3: pack_codes<KIND, 3>(codes, out); break;
    case 4: pack_codes<KIND, 4>(codes, out); break;
    case 5: pack_codes<KIND, 5>(codes, out); break;
    case 6: pack_codes<KIND, 6>(codes, out); break;
    case 7: pack_codes<KIND, 7>(codes, out); break;
    default: pack_codes<KIND, 8>(codes, out); break;
  }
}

__device__ __forceinline__ void put_meta_half(uint32_t* meta, int word, int half, __half x) {
  reinterpret_cast<__half*>(meta)[2 * word + half] = x;
}

// Quantize this thread's group and write its codes into the code tile and
// its (scale, zero) into the meta image, at the positions of the packed block
// format; codes are stored as they are produced (no code array stays live).
__device__ __forceinline__ void quantize_store_group(TileSmem& sm, int kind, int grouping, int b,
                                                     const float (&v)[kG], float mx,
                                                     const GroupParams& g) {
  const int tau = threadIdx.x;
  uint32_t* meta = sm.out + 128 * b;
  const float2 nz = make_float2(-g.zf, -g.zf);
  const float2 iv = make_float2(g.inv, g.inv);
  const uint32_t L = (1u << b) - 1u;
  // (v - zero) * inv is monotone in v, so the group max gives the largest
  // code; when no group of the warp exceeds L the upper clamp is skipped
  // (the saturating conversion already clamps at 0 and 255)
  const uint32_t cmax = cvt_rni_sat_u8(__fmul_rn(__fsub_rn(mx, g.zf), g.inv));
  const bool clamp = __any_sync(0xffffffffu, cmax > L);
  auto code2 = [&](int i, uint32_t& c0, uint32_t& c1) {
    const float2 t = __fmul2_rn(__fadd2_rn(make_float2(v[i], v[i + 1]), nz), iv);
    c0 = cvt_rni_sat_u8(t.x);
    c1 = cvt_rni_sat_u8(t.y);
    if (clamp) {
      c0 = min(c0, L);
      c1 = min(c1, L);
    }
  };
  if (grouping == RQ_PER_CHANNEL) {              // group = channel tau, tokens 0..31
    const int ch = tau;
    if (kind == 0) {
#pragma unroll
      for (int t = 0; t < kG; t += 2) {
        uint32_t c0, c1;
        code2(t, c0, c1);
        sm.codes[t * kCStride + ch] = static_cast<uint8_t>(c0);
        sm.codes[(t + 1) * kCStride + ch] = static_cast<uint8_t>(c1);
      }
      const int word = 16 * ((ch & 7) >> 1) + 2 * (ch >> 4) + ((ch >> 3) & 1);
      put_meta_half(meta, word, ch & 1, g.scale);
      put_meta_half(meta, 64 + word, ch & 1, g.zero);
    } else {
#pragma unroll
      for (int t = 0; t < kG; t += 4) {
        uint32_t c0, c1, c2, c3;
        code2(t, c0, c1);
        code2(t + 2, c2, c3);
        *reinterpret_cast<uint32_t*>(&sm.codes[ct_row(ch) + t]) =
            c0 | (c1 << 8) | (c2 << 16) | (c3 << 24);
      }
      const int word = 16 * (ch & 7) + 2 * (ch >> 4) + ((ch >> 3) & 1);
      put_meta_half(meta, word, 0, g.scale);
      put_meta_half(meta, word, 1, g.zero);
    }
  } else {                                        // group = (token t, channels 32G..)
    const int t = tau >> 2, G = tau & 3;
    if (kind == 0) {
#pragma unroll
      for (int i = 0; i < kG; i += 4) {
        uint32_t c0, c1, c2, c3;
        code2(i, c0, c1);
        code2(i + 2, c2, c3);
        *reinterpret_cast<uint32_t*>(&sm.codes[t * kCStride + 32 * G + i]) =
            c0 | (c1 << 8) | (c2 << 16) | (c3 << 24);
      }
      const int word = 16 * (t & 7) + 4 * (t >> 3) + G;
      put_meta_half(meta, word, 0, g.scale);
      put_meta_half(meta, word, 1, g.zero);
    } else {
#pragma unroll
      for (int i = 0; i < kG; i += 2) {
        uint32_t c0, c1;
        code2(i, c0, c1);
        sm.codes[ct_row(32 * G + i) + t] = static_cast<uint8_t>(c0);
        sm.codes[ct_row(32 * G + i + 1) + t] = static_cast<uint8_t>(c1);
      }
      const int p = t >> 1;
      const int word = 16 * (p & 3) + 4 * (p >> 2) + G;
      put_meta_half(meta, word, t & 1, g.scale);
      put_meta_half(meta, 64 + word, t & 1, g.zero);
    }
  }
}

// Tile position: block j of stream sk = (batch * H + h) * 2 + kind. A CTA
// walks tiles blockIdx.x, blockIdx.x + gridDim.x, ...; the position is
// advanced by carrying (no division in the loop).
struct TileRef {
  int j, sk;
};

__device__ __forceinline__ void advance(TileRef& r, int dj, int dsk, int nblk) {
  r.j += dj;
  r.sk += dsk;
  if (r.j >= nblk) {
    r.j -= nblk;
    r.sk += 1;
  }
}

template <typename T>
__device__ __forceinline__ const T* quant_tile_base(const QuantArgs& a, const TileRef& r) {
  const T* base = static_cast<const T*>((r.sk & 1) ? a.v : a.k);
  return base + (static_cast<long long>(r.sk >> 1) * a.S + static_cast<long long>(kTile) * r.j) * kD;
}

template <typename T>
__global__ void __launch_bounds__(kThreads, RQ_QUANT_MIN_BLOCKS) quantize_pack_kernel(QuantArgs a) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  TileSmem& sm = *reinterpret_cast<TileSmem*>(smem_raw);
  float* x32 = reinterpret_cast<float*>(smem_raw + sizeof(TileSmem));
  const long long stride = gridDim.x;
  long long tile = blockIdx.x;
  if (tile >= a.ntiles) return;
  if (threadIdx.x < kD) sm.signs[threadIdx.x] = a.signs ? a.signs[threadIdx.x] : int8_t(1);
  __syncthreads();
  const bool had = a.hadamard != 0;

  const int nblk = a.nblk;
  const int dsk = static_cast<int>(stride / nblk), dj = static_cast<int>(stride % nblk);
  TileRef r{static_cast<int>(tile % nblk), static_cast<int>(tile / nblk)};
  int grouping = (r.sk & 1) ? a.vg : a.kg;
  bool row_mode = grouping == RQ_PER_TOKEN || had;
  uint4 ld[4];
  load_tile<T>(quant_tile_base<T>(a, r), row_mode, ld);

  for (; tile < a.ntiles; tile += stride) {
    const TileRef cur = r;
    const int kind = cur.sk & 1;
    const int bh = cur.sk >> 1;
    const int h = bh % a.H;
    const int b = a.bits[(a.layer * a.H + h) * 2 + kind];
    float v[kG];
    group_values<T>(ld, row_mode, grouping, had, sm, x32, v);
    // the next tile's loads fly while this one is quantized and packed
    const int cur_grouping = grouping;
    if (tile + stride < a.ntiles) {
      advance(r, dj, dsk, nblk);
      grouping = (r.sk & 1) ? a.vg : a.kg;
      row_mode = grouping == RQ_PER_TOKEN || had;
      load_tile<T>(quant_tile_base<T>(a, r), row_mode, ld);
    }
    if (b < 1 || b > 8) {
      if (threadIdx.x == 0) set_status(a.status, RQ_STATUS_BAD_BITS);
      __syncthreads();
      continue;
    }
    float mn, mx;
    bool finite;
    group_minmax(v, mn, mx, finite);
    const GroupParams g = group_params(mn, mx, finite, b);
    if (g.bad) set_status(a.status, RQ_STATUS_NUMERIC);
    quantize_store_group(sm, kind, cur_grouping, b, v, mx, g);
    __syncthreads();
    if (kind == 0) pack_dispatch<0>(b, sm.codes, sm.out);
    else pack_dispatch<1>(b, sm.codes, sm.out);
    __syncthreads();
    // offsets[layer][batch][h][kind] = offsets[layer * B * H * 2 + sk]
    const uint64_t off = a.offsets[static_cast<long long>(a.layer) * a.B * a.H * 2 + cur.sk];
    uint4* dst = reinterpret_cast<uint4*>(a.packed + off + static_cast<uint64_t>(cur.j) * 512u * (b + 1));
    const uint4* src = reinterpret_cast<const uint4*>(sm.out);
    for (int i = threadIdx.x; i < 32 * (b + 1); i += kThreads) dst[i] = src[i];
    __syncthreads();
  }
}

// ------------------------------------------------------ distortion sweep ----
// Per component and b = 1..8: sum over the component's groups of
// (y - y_hat)^2 with y_hat = fp32(fp32(c * scale) + zero). A group's 32
// squared errors are summed in fp32 (two interleaved partial sums, fixed
// order) and the per-group sums in fp64; per-tile partials are reduced in a
// fixed order (deterministic).

template <typename T>
__global__ void __launch_bounds__(kThreads) calib_sweep_kernel(CalibArgs a) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  TileSmem& sm = *reinterpret_cast<TileSmem*>(smem_raw);
  float* x32 = reinterpret_cast<float*>(smem_raw + sizeof(TileSmem));
  __shared__ double red[kThreads / 32][8];
  const long long stride = gridDim.x;
  long long tile = blockIdx.x;
  if (tile >= a.ntiles) return;
  if (threadIdx.x < kD) sm.signs[threadIdx.x] = a.signs ? a.signs[threadIdx.x] : int8_t(1);
  __syncthreads();
  const bool had = a.hadamard != 0;
  const T* xbase = static_cast<const T*>(a.x);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;

  int grouping = (static_cast<int>(tile / a.ntile) & 1) ? a.vg : a.kg;
  bool row_mode = grouping == RQ_PER_TOKEN || had;
  uint4 ld[4];
  load_tile<T>(xbase + tile * kTile * kD, row_mode, ld);
  for (; tile < a.ntiles; tile += stride) {
    float v[kG];
    group_values<T>(ld, row_mode, grouping, had, sm, x32, v);
    const long long next = tile + stride;
    if (next < a.ntiles) {
      grouping = (static_cast<int>(next / a.ntile) & 1) ? a.vg : a.kg;
      row_mode = grouping == RQ_PER_TOKEN || had;
      load_tile<T>(xbase + next * kTile * kD, row_mode, ld);
    }
    float mn, mx;
    bool finite;
    group_minmax(v, mn, mx, finite);
    double acc[8];
#pragma unroll
    for (int b = 1; b <= 8; ++b) {
      const GroupParams g = group_params(mn, mx, finite, b);
      if (b == 1 && g.bad) set_status(a.status, RQ_STATUS_NUMERIC);
      uint32_t c[kG];
      group_codes(v, g, b, c);
      const float2 sf = make_float2(g.sf, g.sf), zf = make_float2(g.zf, g.zf);
      float2 s2 = make_float2(0.0f, 0.0f);
#pragma unroll
      for (int i = 0; i < kG; i += 2) {
        const float2 xh = __fadd2_rn(
            __fmul2_rn(make_float2(static_cast<float>(c[i]), static_cast<float>(c[i + 1])), sf), zf);
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

size_t tile_smem_bytes(bool hadamard, int kg, int vg) {
  const bool x32 = hadamard && (kg == RQ_PER_CHANNEL || vg == RQ_PER_CHANNEL);
  return sizeof(TileSmem) + (x32 ? kX32Floats * sizeof(float) : 0);
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
  const size_t smem = tile_smem_bytes(a.hadamard != 0, a.kg, a.vg);
  return desc->dtype == RQ_F16 ? launch_persistent(quantize_pack_kernel<__half>, a, smem, st)
                               : launch_persistent(quantize_pack_kernel<__nv_bfloat16>, a, smem, st);
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
  const size_t smem = tile_smem_bytes(a.hadamard != 0, a.kg, a.vg);
  const rq_status s = dtype == RQ_F16
                          ? launch_persistent(calib_sweep_kernel<__half>, a, smem, st)
                          : launch_persistent(calib_sweep_kernel<__nv_bfloat16>, a, smem, st);
  if (s != RQ_OK) return s;
  calib_finalize_kernel<<<(n * 8 + 127) / 128, 128, 0, st>>>(a.partial, mse_dev, n, a.ntile,
                                                              static_cast<double>(T) * kD);
  return launch_status();
}
