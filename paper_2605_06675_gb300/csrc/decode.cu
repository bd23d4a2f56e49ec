// Split-K GQA decode attention that reads the packed mixed-bit cache
// directly, plus the log-sum-exp combine of the split partials.
//
// RateQuant (arXiv 2605.06675): the allocation table is a static lookup
// indexed at run time (App. M, App. U) and the quantizers are fused with the
// consumer so the full-precision cache is never materialised (App. W "Kernel
// fusion"). Attention itself is standard decode attention (Sec. 1) with GQA
// (Sec. 4.1 "Models"); the QuaRot cache is used as Q(XR)R^T (App. W).
//
// Design (sm_103a): one CTA = (split of the sequence, kv head, batch), four
// warps, each warp walking its own 32-token blocks. Per block a warp runs
//   scores^T[32 tok x 8 heads] = K_hat[32 x 128] . q^T      (16 x mma m16n8k16)
//   online softmax in fp32 (log2 domain), P^T via movmatrix.trans
//   o^T[128 x 8 heads]       += V_hat^T[128 x 32] . P^T    (16 x mma m16n8k16)
// The GQA group (g <= 8 query heads) is the MMA n dimension, so it is never
// padded to 16. Codes are read in the MMA-fragment order the quantizer wrote,
// turned into exact fp16 integers with the 1024-exponent trick and dequantized
// with one fp16x2 FMA (scale, zero) in registers.
#include <algorithm>
#include <atomic>

#include "rq_internal.cuh"

namespace rq {

rq_status current_sm_count(int* sms) {
  static std::atomic<int> cache[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return RQ_ERR_CUDA;
  if (dev >= 0 && dev < 64) {
    const int c = cache[dev].load(std::memory_order_relaxed);
    if (c > 0) {
      *sms = c;
      return RQ_OK;
    }
  }
  int v = 0;
  if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || v <= 0)
    return RQ_ERR_CUDA;
  if (dev >= 0 && dev < 64) cache[dev].store(v, std::memory_order_relaxed);
  *sms = v;
  return RQ_OK;
}

namespace {

constexpr int kWarps = 4;
constexpr int kThreads = 32 * kWarps;
constexpr int kPart = kD + 2;   // partial record: o[128], m (log2 domain), l
constexpr int kMaxHeads = 8;    // MMA n

struct DecodeArgs {
  const void* q;
  const uint8_t* packed;
  const uint8_t* bits;
  const uint64_t* offsets;
  const int8_t* signs;
  float* partial;
  uint32_t* status;
  int layer, B, H, Hq, g, nblk, splits, bps, kg, vg, hadamard;
};

__device__ __forceinline__ uint32_t h2u(__half2 h) { return *reinterpret_cast<uint32_t*>(&h); }
__device__ __forceinline__ __half2 u2h(uint32_t u) { return *reinterpret_cast<__half2*>(&u); }
__device__ __forceinline__ uint32_t pack_f16x2(float lo, float hi) {
  return h2u(__floats2half2_rn(lo, hi));
}

__device__ __forceinline__ void mma16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                         uint32_t b1) {
  asm("mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};\n"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint32_t movmatrix_trans(uint32_t x) {
  uint32_t y;
  asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;\n" : "=r"(y) : "r"(x));
  return y;
}

// lane's 4*BW code words of one block: 16-byte piece i of lane L at 16*(32 i + L)
template <int BW>
__device__ __forceinline__ void load_lane_codes(const uint8_t* blk, int lane, uint32_t (&w)[4 * BW]) {
#pragma unroll
  for (int i = 0; i < BW; ++i) {
    const uint4 u = ldg_stream(blk + 16 * (32 * i + lane));
    w[4 * i + 0] = u.x;
    w[4 * i + 1] = u.y;
    w[4 * i + 2] = u.z;
    w[4 * i + 3] = u.w;
  }
}

// BW-bit code at lane-stream bit p (p is a compile-time constant after unrolling)
template <int BW>
__device__ __forceinline__ uint32_t lane_code(const uint32_t (&w)[4 * BW], int p) {
  const int wi = p >> 5, sh = p & 31;
  uint32_t v = w[wi] >> sh;
  if (sh + BW > 32) v |= w[wi + 1] << (32 - sh);
  return v & ((1u << BW) - 1u);
}

// Register k of the A fragment of fragment phi: codes (a_2k, a_2k+1) at slot
// positions k and 4+k, as exact fp16 integers: the code is OR-ed into the
// mantissa of fp16 1024.0 and 1024.0 is subtracted.
template <int BW>
__device__ __forceinline__ __half2 code_pair(const uint32_t (&w)[4 * BW], int phi, int k) {
  const int base = 8 * BW * phi;
  const uint32_t lo = lane_code<BW>(w, base + BW * k);
  const uint32_t hi = lane_code<BW>(w, base + BW * (4 + k));
  constexpr uint32_t kMagic = 0x64006400u;
  return __hsub2(u2h(lo | (hi << 16) | kMagic), u2h(kMagic));
}

// 16 meta words of this lane starting at uint4 index q4
__device__ __forceinline__ void load_meta16(const uint4* meta, int q4, uint32_t (&m)[16]) {
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const uint4 u = ldg_stream(meta + q4 + i);
    m[4 * i + 0] = u.x;
    m[4 * i + 1] = u.y;
    m[4 * i + 2] = u.z;
    m[4 * i + 3] = u.w;
  }
}

// scores^T[mt] (tokens 16 mt + gid (+8), heads 2 tig (+1)) for one K block
template <int BW, int KG>
__device__ __forceinline__ void qk_block(const uint8_t* blk, int lane, const uint32_t (&qb)[8][2],
                                         float (&s)[2][4]) {
  const int gid = lane >> 2, tig = lane & 3;
  uint32_t w[4 * BW];
  load_lane_codes<BW>(blk, lane, w);
  const uint4* meta = reinterpret_cast<const uint4*>(blk + 512 * BW);
  uint32_t ms[16], mz[16];
  if (KG == RQ_PER_CHANNEL) {   // scale pairs at words 16 tig.., zero pairs at 64 + 16 tig..
    load_meta16(meta, 4 * tig, ms);
    load_meta16(meta, 16 + 4 * tig, mz);
  } else {                      // (scale, zero) words at 16 gid..
    load_meta16(meta, 4 * gid, ms);
  }
#pragma unroll
  for (int mt = 0; mt < 2; ++mt)
#pragma unroll
    for (int r = 0; r < 4; ++r) s[mt][r] = 0.0f;
#pragma unroll
  for (int ks = 0; ks < 8; ++ks) {
#pragma unroll
    for (int mt = 0; mt < 2; ++mt) {
      const int phi = 2 * ks + mt;
      uint32_t a[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const __half2 c = code_pair<BW>(w, phi, k);
        __half2 sc, zr;
        if (KG == RQ_PER_CHANNEL) {        // channels 16 ks + 8 (k>>1) + 2 tig, +1
          const int wd = 2 * ks + (k >> 1);
          sc = u2h(ms[wd]);
          zr = u2h(mz[wd]);
        } else {                           // token 16 mt + gid + 8 (k&1), group ks/2
          const __half2 sz = u2h(ms[4 * (2 * mt + (k & 1)) + (ks >> 1)]);
          sc = __low2half2(sz);
          zr = __high2half2(sz);
        }
        a[k] = h2u(__hfma2(c, sc, zr));
      }
      mma16816(s[mt], a, qb[ks][0], qb[ks][1]);
    }
  }
}

// o^T[mt] (channels 16 mt + gid (+8), heads 2 tig (+1)) += V_hat^T . P^T for one V block
template <int BW, int VG>
__device__ __forceinline__ void pv_block(const uint8_t* blk, int lane, const uint32_t (&pb)[2][2],
                                         float (&o)[8][4]) {
  const int gid = lane >> 2, tig = lane & 3;
  uint32_t w[4 * BW];
  load_lane_codes<BW>(blk, lane, w);
  const uint4* meta = reinterpret_cast<const uint4*>(blk + 512 * BW);
  uint32_t ms[16], mz[16];
  if (VG == RQ_PER_TOKEN) {
    load_meta16(meta, 4 * tig, ms);
    load_meta16(meta, 16 + 4 * tig, mz);
  } else {
    load_meta16(meta, 4 * gid, ms);
  }
#pragma unroll
  for (int ks = 0; ks < 2; ++ks) {
#pragma unroll
    for (int mt = 0; mt < 8; ++mt) {
      const int phi = 8 * ks + mt;
      uint32_t a[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const __half2 c = code_pair<BW>(w, phi, k);
        __half2 sc, zr;
        if (VG == RQ_PER_TOKEN) {          // tokens 16 ks + 8 (k>>1) + 2 tig, +1; group mt/2
          const int wd = 4 * (2 * ks + (k >> 1)) + (mt >> 1);
          sc = u2h(ms[wd]);
          zr = u2h(mz[wd]);
        } else {                           // channel 16 mt + gid + 8 (k&1)
          const __half2 sz = u2h(ms[2 * mt + (k & 1)]);
          sc = __low2half2(sz);
          zr = __high2half2(sz);
        }
        a[k] = h2u(__hfma2(c, sc, zr));
      }
      mma16816(o[mt], a, pb[ks][0], pb[ks][1]);
    }
  }
}

template <int BW>
__device__ __forceinline__ void qk_dispatch_g(int kg, const uint8_t* blk, int lane,
                                              const uint32_t (&qb)[8][2], float (&s)[2][4]) {
  if (kg == RQ_PER_CHANNEL) qk_block<BW, RQ_PER_CHANNEL>(blk, lane, qb, s);
  else qk_block<BW, RQ_PER_TOKEN>(blk, lane, qb, s);
}

template <int BW>
__device__ __forceinline__ void pv_dispatch_g(int vg, const uint8_t* blk, int lane,
                                              const uint32_t (&pb)[2][2], float (&o)[8][4]) {
  if (vg == RQ_PER_TOKEN) pv_block<BW, RQ_PER_TOKEN>(blk, lane, pb, o);
  else pv_block<BW, RQ_PER_CHANNEL>(blk, lane, pb, o);
}

__device__ __forceinline__ void qk_dispatch(int bw, int kg, const uint8_t* blk, int lane,
                                            const uint32_t (&qb)[8][2], float (&s)[2][4]) {
  switch (bw) {
    case 1: qk_dispatch_g<1>(kg, blk, lane, qb, s); break;
    case 2: qk_dispatch_g<2>(kg, blk, lane, qb, s); break;
    case 3: qk_dispatch_g<3>(kg, blk, lane, qb, s); break;
    case 4: qk_dispatch_g<4>(kg, blk, lane, qb, s); break;
    case 5: qk_dispatch_g<5>(kg, blk, lane, qb, s); break;
    case 6: qk_dispatch_g<6>(kg, blk, lane, qb, s); break;
    case 7: qk_dispatch_g<7>(kg, blk, lane, qb, s); break;
    default: qk_dispatch_g<8>(kg, blk, lane, qb, s); break;
  }
}

__device__ __forceinline__ void pv_dispatch(int bw, int vg, const uint8_t* blk, int lane,
                                            const uint32_t (&pb)[2][2], float (&o)[8][4]) {
  switch (bw) {
    case 1: pv_dispatch_g<1>(vg, blk, lane, pb, o); break;
    case 2: pv_dispatch_g<2>(vg, blk, lane, pb, o); break;
    case 3: pv_dispatch_g<3>(vg, blk, lane, pb, o); break;
    case 4: pv_dispatch_g<4>(vg, blk, lane, pb, o); break;
    case 5: pv_dispatch_g<5>(vg, blk, lane, pb, o); break;
    case 6: pv_dispatch_g<6>(vg, blk, lane, pb, o); break;
    case 7: pv_dispatch_g<7>(vg, blk, lane, pb, o); break;
    default: pv_dispatch_g<8>(vg, blk, lane, pb, o); break;
  }
}

// 128-point FWHT of each of `rows` rows of x (row stride 128), strides 1..64
__device__ void fwht_smem(float* x, int rows) {
  for (int lh = 0; lh < 7; ++lh) {
    const int h = 1 << lh;
    for (int p = threadIdx.x; p < rows * 64; p += blockDim.x) {
      const int row = p >> 6, pi = p & 63;
      const int i = ((pi >> lh) << (lh + 1)) | (pi & (h - 1));
      float* r = x + row * kD;
      const float a = r[i], b = r[i + h];
      r[i] = a + b;
      r[i + h] = a - b;
    }
    __syncthreads();
  }
}

template <typename T>
__global__ void __launch_bounds__(kThreads) decode_split_kernel(DecodeArgs a) {
  __shared__ float qs[kMaxHeads][kD];
  __shared__ float red_o[kWarps][kMaxHeads][kD];
  __shared__ float red_m[kWarps][kMaxHeads];
  __shared__ float red_l[kWarps][kMaxHeads];
  const int split = blockIdx.x, h = blockIdx.y, batch = blockIdx.z;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int gid = lane >> 2, tig = lane & 3;

  // q of the g query heads of this kv head (rows >= g are zero), rotated
  // into the cache's domain when the cache is Hadamard-rotated
  const T* qp = static_cast<const T*>(a.q) + (static_cast<long long>(batch) * a.Hq +
                                              static_cast<long long>(h) * a.g) * kD;
  for (int idx = threadIdx.x; idx < kMaxHeads * kD; idx += kThreads) {
    const int n = idx >> 7, d = idx & 127;
    float x = 0.0f;
    if (n < a.g) {
      x = to_f32<T>(qp[n * kD + d]);
      if (a.hadamard && a.signs && a.signs[d] < 0) x = -x;
    }
    qs[n][d] = x;
  }
  __syncthreads();
  if (a.hadamard) fwht_smem(&qs[0][0], kMaxHeads);
  // softmax scale 1/sqrt(128) and log2(e) folded into q (scores in log2 units)
  const float qscale = kLog2e * kInvSqrt128 * (a.hadamard ? kInvSqrt128 : 1.0f);
  uint32_t qb[8][2];
#pragma unroll
  for (int ks = 0; ks < 8; ++ks) {
    const int c0 = 16 * ks + 2 * tig;
    qb[ks][0] = pack_f16x2(qs[gid][c0] * qscale, qs[gid][c0 + 1] * qscale);
    qb[ks][1] = pack_f16x2(qs[gid][c0 + 8] * qscale, qs[gid][c0 + 9] * qscale);
  }

  const int bK = a.bits[(a.layer * a.H + h) * 2 + 0];
  const int bV = a.bits[(a.layer * a.H + h) * 2 + 1];
  const bool valid = bK >= 1 && bK <= 8 && bV >= 1 && bV <= 8;
  if (!valid && threadIdx.x == 0) set_status(a.status, RQ_STATUS_BAD_BITS);
  const uint64_t* offp =
      a.offsets + ((static_cast<long long>(a.layer) * a.B + batch) * a.H + h) * 2;
  const uint8_t* kbase = a.packed + offp[0];
  const uint8_t* vbase = a.packed + offp[1];
  const int blk0 = split * a.bps;
  const int blk1 = min(a.nblk, blk0 + a.bps);

  float o[8][4];
#pragma unroll
  for (int mt = 0; mt < 8; ++mt)
#pragma unroll
    for (int r = 0; r < 4; ++r) o[mt][r] = 0.0f;
  float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.0f, l1 = 0.0f;

  if (valid) {
    for (int blk = blk0 + warp; blk < blk1; blk += kWarps) {
      float s[2][4];
      qk_dispatch(bK, a.kg, kbase + static_cast<size_t>(blk) * 512u * (bK + 1), lane, qb, s);
      // online softmax over this block's 32 tokens, per head column
      float bm0 = fmaxf(fmaxf(s[0][0], s[0][2]), fmaxf(s[1][0], s[1][2]));
      float bm1 = fmaxf(fmaxf(s[0][1], s[0][3]), fmaxf(s[1][1], s[1][3]));
#pragma unroll
      for (int off = 4; off <= 16; off <<= 1) {
        bm0 = fmaxf(bm0, __shfl_xor_sync(0xffffffffu, bm0, off));
        bm1 = fmaxf(bm1, __shfl_xor_sync(0xffffffffu, bm1, off));
      }
      const float nm0 = fmaxf(m0, bm0), nm1 = fmaxf(m1, bm1);
      const float al0 = exp2f(m0 - nm0), al1 = exp2f(m1 - nm1);
      m0 = nm0;
      m1 = nm1;
      float p[2][4];
#pragma unroll
      for (int mt = 0; mt < 2; ++mt) {
        p[mt][0] = exp2f(s[mt][0] - m0);
        p[mt][1] = exp2f(s[mt][1] - m1);
        p[mt][2] = exp2f(s[mt][2] - m0);
        p[mt][3] = exp2f(s[mt][3] - m1);
      }
      l0 = l0 * al0 + ((p[0][0] + p[0][2]) + (p[1][0] + p[1][2]));
      l1 = l1 * al1 + ((p[0][1] + p[0][3]) + (p[1][1] + p[1][3]));
#pragma unroll
      for (int mt = 0; mt < 8; ++mt) {
        o[mt][0] *= al0;
        o[mt][1] *= al1;
        o[mt][2] *= al0;
        o[mt][3] *= al1;
      }
      uint32_t pb[2][2];
#pragma unroll
      for (int ks = 0; ks < 2; ++ks) {
        pb[ks][0] = movmatrix_trans(pack_f16x2(p[ks][0], p[ks][1]));
        pb[ks][1] = movmatrix_trans(pack_f16x2(p[ks][2], p[ks][3]));
      }
      pv_dispatch(bV, a.vg, vbase + static_cast<size_t>(blk) * 512u * (bV + 1), lane, pb, o);
    }
  }
#pragma unroll
  for (int off = 4; off <= 16; off <<= 1) {
    l0 += __shfl_xor_sync(0xffffffffu, l0, off);
    l1 += __shfl_xor_sync(0xffffffffu, l1, off);
  }
  // merge the four warps (log-sum-exp), one partial record per query head
#pragma unroll
  for (int mt = 0; mt < 8; ++mt) {
    red_o[warp][2 * tig][16 * mt + gid] = o[mt][0];
    red_o[warp][2 * tig + 1][16 * mt + gid] = o[mt][1];
    red_o[warp][2 * tig][16 * mt + gid + 8] = o[mt][2];
    red_o[warp][2 * tig + 1][16 * mt + gid + 8] = o[mt][3];
  }
  if (gid == 0) {
    red_m[warp][2 * tig] = m0;
    red_m[warp][2 * tig + 1] = m1;
    red_l[warp][2 * tig] = l0;
    red_l[warp][2 * tig + 1] = l1;
  }
  __syncthreads();
  const int d = threadIdx.x;
  for (int n = 0; n < a.g; ++n) {
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) M = fmaxf(M, red_m[w][n]);
    float osum = 0.0f, lsum = 0.0f;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) {
      const float mw = red_m[w][n];
      const float sc = (mw == -INFINITY) ? 0.0f : exp2f(mw - M);
      osum += sc * red_o[w][n][d];
      lsum += sc * red_l[w][n];
    }
    float* dst = a.partial + ((static_cast<long long>(batch) * a.Hq + h * a.g + n) * a.splits + split) * kPart;
    dst[d] = osum;
    if (d == 0) {
      dst[kD] = M;
      dst[kD + 1] = lsum;
    }
  }
}

// out[row] = sum_s 2^(m_s - M) o_s / sum_s 2^(m_s - M) l_s, rotated back
// (o R^T = FWHT(o) / sqrt(128) * signs) for a Hadamard cache.
__global__ void __launch_bounds__(kD) decode_combine_kernel(const float* partial, float* out,
                                                           const int8_t* signs, uint32_t* status,
                                                           int splits, int hadamard) {
  __shared__ float y[kD];
  const long long row = blockIdx.x;
  const int d = threadIdx.x;
  const float* p = partial + row * splits * kPart;
  float M = -INFINITY;
  for (int s = 0; s < splits; ++s) M = fmaxf(M, p[s * kPart + kD]);
  float L = 0.0f, acc = 0.0f;
  if (M != -INFINITY) {
    for (int s = 0; s < splits; ++s) {
      const float ms = p[s * kPart + kD];
      const float sc = (ms == -INFINITY) ? 0.0f : exp2f(ms - M);
      L += sc * p[s * kPart + kD + 1];
      acc += sc * p[s * kPart + d];
    }
  }
  float r = L > 0.0f ? acc / L : 0.0f;
  if (!(L > 0.0f) || !isfinite(r)) {
    if (d == 0) set_status(status, RQ_STATUS_NUMERIC);
    if (!isfinite(r)) r = 0.0f;
  }
  if (hadamard) {
    y[d] = r;
    __syncthreads();
    fwht_smem(y, 1);
    r = y[d] * kInvSqrt128;
    if (signs && signs[d] < 0) r = -r;
  }
  out[row * kD + d] = r;
}

void decode_plan(const rq_cache_desc* desc, int sms, int* splits, int* bps) {
  const int nblk = desc->S / kTile;
  const long long units = static_cast<long long>(desc->B) * desc->H_kv;
  const long long target = static_cast<long long>(sms) * 8;
  long long sp = units > 0 ? (target + units - 1) / units : 1;
  sp = std::max<long long>(1, std::min<long long>(sp, nblk));
  const int b = static_cast<int>((nblk + sp - 1) / sp);
  *bps = std::max(b, 1);
  *splits = std::max(1, (nblk + *bps - 1) / *bps);
}

rq_status check_desc(const rq_cache_desc* desc) {
  if (!desc) return RQ_ERR_INVALID_ARG;
  if (desc->L <= 0 || desc->B < 0 || desc->H_kv <= 0 || desc->H_q <= 0 || desc->S < 0)
    return RQ_ERR_INVALID_ARG;
  if (desc->dtype != RQ_F16 && desc->dtype != RQ_BF16) return RQ_ERR_INVALID_ARG;
  for (int g : {desc->k_grouping, desc->v_grouping})
    if (g != RQ_PER_TOKEN && g != RQ_PER_CHANNEL) return RQ_ERR_INVALID_ARG;
  if (desc->d != kD || desc->group != kG || desc->S % kTile != 0 || desc->S == 0)
    return RQ_ERR_SHAPE;
  if (desc->H_q % desc->H_kv != 0 || desc->H_q / desc->H_kv > kMaxHeads) return RQ_ERR_SHAPE;
  return RQ_OK;
}

}  // namespace
}  // namespace rq

extern "C" rq_status rq_decode_workspace_bytes(const rq_cache_desc* desc, size_t* bytes) {
  using namespace rq;
  if (!bytes) return RQ_ERR_INVALID_ARG;
  const rq_status st = check_desc(desc);
  if (st != RQ_OK) return st;
  int sms = 0;
  if (current_sm_count(&sms) != RQ_OK) return RQ_ERR_CUDA;
  int splits = 1, bps = 1;
  decode_plan(desc, sms, &splits, &bps);
  *bytes = static_cast<size_t>(desc->B) * desc->H_q * splits * kPart * sizeof(float);
  return RQ_OK;
}

extern "C" rq_status rq_decode_attention(const rq_cache_desc* desc, int32_t layer, const void* q,
                                         const void* packed, const uint8_t* bits_dev,
                                         const uint64_t* offsets_dev, const int8_t* signs_dev,
                                         float* out, void* ws, size_t ws_bytes,
                                         uint32_t* status_dev, void* stream) {
  using namespace rq;
  const rq_status st = check_desc(desc);
  if (st != RQ_OK) return st;
  if (!q || !packed || !bits_dev || !offsets_dev || !out || !ws) return RQ_ERR_INVALID_ARG;
  if (layer < 0 || layer >= desc->L) return RQ_ERR_INVALID_ARG;
  if (!aligned16(packed) || !aligned16(ws) || (reinterpret_cast<uintptr_t>(q) & 1u) ||
      (reinterpret_cast<uintptr_t>(out) & 3u))
    return RQ_ERR_ALIGNMENT;
  if (desc->B == 0) return RQ_OK;
  int sms = 0;
  if (current_sm_count(&sms) != RQ_OK) return RQ_ERR_CUDA;
  int splits = 1, bps = 1;
  decode_plan(desc, sms, &splits, &bps);
  const size_t need = static_cast<size_t>(desc->B) * desc->H_q * splits * kPart * sizeof(float);
  if (ws_bytes < need) return RQ_ERR_WORKSPACE;
  DecodeArgs a;
  a.q = q;
  a.packed = static_cast<const uint8_t*>(packed);
  a.bits = bits_dev;
  a.offsets = offsets_dev;
  a.signs = signs_dev;
  a.partial = static_cast<float*>(ws);
  a.status = status_dev;
  a.layer = layer;
  a.B = desc->B;
  a.H = desc->H_kv;
  a.Hq = desc->H_q;
  a.g = desc->H_q / desc->H_kv;
  a.nblk = desc->S / kTile;
  a.splits = splits;
  a.bps = bps;
  a.kg = desc->k_grouping;
  a.vg = desc->v_grouping;
  a.hadamard = desc->hadamard ? 1 : 0;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const dim3 grid(static_cast<unsigned>(splits), static_cast<unsigned>(desc->H_kv),
                  static_cast<unsigned>(desc->B));
  if (desc->dtype == RQ_F16) decode_split_kernel<__half><<<grid, kThreads, 0, s>>>(a);
  else decode_split_kernel<__nv_bfloat16><<<grid, kThreads, 0, s>>>(a);
  if (launch_status() != RQ_OK) return RQ_ERR_CUDA;
  decode_combine_kernel<<<static_cast<unsigned>(desc->B * desc->H_q), kD, 0, s>>>(
      a.partial, out, signs_dev, status_dev, splits, a.hadamard);
  return launch_status();
}

// ---------------------------------------------------------------------------
// Allocation-free decode: the split-K partials live in a fixed device array
// of this library instead of a caller-supplied workspace, for callers that
// cannot allocate (graph replays, foreign allocators, plugins handed only
// their inputs and outputs). The array is shared by every call on a device.
namespace rq {
namespace {

constexpr size_t kStaticScratchFloats = RQ_STATIC_SCRATCH_BYTES / sizeof(float);
static __device__ __align__(256) float g_decode_scratch[kStaticScratchFloats];

// device address of g_decode_scratch for the current device, looked up once
// per device (host code only sees a host-side stand-in for the symbol)
rq_status static_scratch_ptr(float** ptr) {
  static std::atomic<uintptr_t> cache[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return RQ_ERR_CUDA;
  if (dev >= 0 && dev < 64) {
    const uintptr_t c = cache[dev].load(std::memory_order_acquire);
    if (c != 0) {
      *ptr = reinterpret_cast<float*>(c);
      return RQ_OK;
    }
  }
  void* p = nullptr;
  if (cudaGetSymbolAddress(&p, g_decode_scratch) != cudaSuccess || p == nullptr) return RQ_ERR_CUDA;
  if (dev >= 0 && dev < 64) cache[dev].store(reinterpret_cast<uintptr_t>(p), std::memory_order_release);
  *ptr = static_cast<float*>(p);
  return RQ_OK;
}

}  // namespace
}  // namespace rq

extern "C" rq_status rq_decode_attention_static(const rq_cache_desc* desc, int32_t layer,
                                                const void* q, const void* packed,
                                                const uint8_t* bits_dev,
                                                const uint64_t* offsets_dev,
                                                const int8_t* signs_dev, float* out,
                                                uint32_t* status_dev, void* stream) {
  using namespace rq;
  const rq_status st = check_desc(desc);
  if (st != RQ_OK) return st;
  if (!q || !packed || !bits_dev || !offsets_dev || !out) return RQ_ERR_INVALID_ARG;
  if (layer < 0 || layer >= desc->L) return RQ_ERR_INVALID_ARG;
  if (!aligned16(packed) || (reinterpret_cast<uintptr_t>(q) & 1u) ||
      (reinterpret_cast<uintptr_t>(out) & 3u))
    return RQ_ERR_ALIGNMENT;
  if (desc->B == 0) return RQ_OK;
  int sms = 0;
  if (current_sm_count(&sms) != RQ_OK) return RQ_ERR_CUDA;
  int splits = 1, bps = 1;
  decode_plan(desc, sms, &splits, &bps);
  const size_t need = static_cast<size_t>(desc->B) * desc->H_q * splits * kPart * sizeof(float);
  if (need > RQ_STATIC_SCRATCH_BYTES) return RQ_ERR_WORKSPACE;
  float* scratch = nullptr;
  if (static_scratch_ptr(&scratch) != RQ_OK) return RQ_ERR_CUDA;
  DecodeArgs a;
  a.q = q;
  a.packed = static_cast<const uint8_t*>(packed);
  a.bits = bits_dev;
  a.offsets = offsets_dev;
  a.signs = signs_dev;
  a.partial = scratch;
  a.status = status_dev;
  a.layer = layer;
  a.B = desc->B;
  a.H = desc->H_kv;
  a.Hq = desc->H_q;
  a.g = desc->H_q / desc->H_kv;
  a.nblk = desc->S / kTile;
  a.splits = splits;
  a.bps = bps;
  a.kg = desc->k_grouping;
  a.vg = desc->v_grouping;
  a.hadamard = desc->hadamard ? 1 : 0;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const dim3 grid(static_cast<unsigned>(splits), static_cast<unsigned>(desc->H_kv),
                  static_cast<unsigned>(desc->B));
  if (desc->dtype == RQ_F16) decode_split_kernel<__half><<<grid, kThreads, 0, s>>>(a);
  else decode_split_kernel<__nv_bfloat16><<<grid, kThreads, 0, s>>>(a);
  if (launch_status() != RQ_OK) return RQ_ERR_CUDA;
  decode_combine_kernel<<<static_cast<unsigned>(desc->B * desc->H_q), kD, 0, s>>>(
      a.partial, out, signs_dev, status_dev, splits, a.hadamard);
  return launch_status();
}
